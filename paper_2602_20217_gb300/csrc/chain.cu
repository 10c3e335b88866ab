// Chained projections for bf16 models: one persistent launch runs a sequence
// of decoder projections ("phases": QKV, O + residual, gate/up + SwiGLU,
// down + residual, LM head + argmax) of the Sec. 2 sublayers that a pass
// executes back to back, i.e. everything between two attention cores.
//
// Why: at R <= 16 rows each projection is a pure stream over its weights.
// Launched one by one, every projection pays a ramp (first tiles in flight),
// a tail (the last items on a few SMs) and a launch gap, which cost small
// matrices (W_o: 33.6 MB, 5 us at HBM speed) two thirds of their time.  Here
// the weight stream never stops at a phase boundary: weights do not depend on
// the activations, so each CTA's producer keeps loading the next phase's
// weight tiles while the previous phase is still finishing anywhere on the
// GPU.  Only the small activation tiles wait for the previous phase.
//
// Per CTA (two per SM for up to 8 rows, else one; 7 warps):
//  * warp 4 (weights): claims work items phase by phase from per-phase
//    atomic queues (16 output features over the full K) and issues their
//    2-D TMA weight boxes into a ring of shared-memory stages;
//  * warp 5 (activations): follows the same stage sequence; before a stage
//    it waits until the block of the previous phase's output that the stage
//    reads is complete, then issues the stage's activation boxes;
//  * warps 0-3 (consumers): mma.sync m16n8k16 with weights as A and the R
//    activation rows as B (columns independent: batch invariant), each warp
//    a quarter of every stage's columns,
//    then hand each item's per-warp sums to
//  * warp 6 (epilogue): adds them in warp order (fixed), computes the rows'
//    1/rms at its first item of a normed phase (normalised inputs), runs the
//    fused epilogue, and after the CTA's last item of a phase adds its item count
//    to the phase's done-counter (one release per CTA and phase).  LM head:
//    each CTA keeps its best (logit, id) per row and merges it into a 64-bit
//    key with atomicMax (value first, then the lower id: any merge order gives
//    the same argmax); the CTA whose count completes the phase reads it.
//    Partials are double buffered, so consumers never wait for an epilogue.
// A stage is full when both loaders have arrived and all bytes have landed.
// A CTA's first unit of each phase is fixed by its index; further units are
// claimed from per-phase atomic queues.  Deadlock-free: every CTA of the grid
// becomes resident once the kernels before it finish (the grid is sized to
// fit), a CTA works its units in phase order, and the lowest unfinished phase
// always has all its inputs.  Every wait is bounded (2 s): on expiry the
// status word is set and the CTA leaves.
#include "common.cuh"
#include "internal.h"
#include "tma.cuh"

#include <algorithm>
#include <climits>

namespace ks {

namespace {

constexpr int kThreads = 224;
constexpr int kWarpW = 4;      // weight loader
constexpr int kWarpA = 5;      // activation loader
constexpr int kWarpE = 6;      // epilogue
constexpr int kMaxStages = 8;
constexpr int kBoxElems = 256 * 16;                  // 256 columns x 16 rows of a stage
constexpr int kChunkBytes = 64 * 16 * 2;             // weight chunk: 64 columns x 16 rows, 128-byte swizzled
constexpr uint32_t kWBytes = 4u * kBoxElems * 2u;    // weight bytes per stage (4 boxes)
// Ring per CTA: up to 8 rows run two CTAs per SM (two independent pipelines
// per SM measured 21 % faster than one with twice the ring); more rows need
// the room of one CTA per SM.
constexpr size_t kRingBudget1 = 196u * 1024u;        // one CTA per SM
constexpr size_t kRingBudget2 = 104u * 1024u;        // two CTAs per SM
constexpr int kMaxRows = 16;

// Status word codes (the first one recorded stays): a bounded wait ran out,
// or a self-check found a stage or item record out of range (the access it
// guards is skipped).
constexpr int kErrWait = 1;
constexpr int kErrCheckW = 2, kErrCheckA = 3, kErrCheckC = 4, kErrCheckE = 5;
KS_DEV void set_err(int* e, int code) { atomicCAS(e, 0, code); }

struct Phase {
    int kind, layer, N, K, n_items, tpi;
    int n_sl, sl_len, n_units;   // K-slices per item (residual phases with few items), stages per slice
};

// The residual projections W_o and W_down have only d / 16 row groups (256 for
// d = 4096): fewer items than CTAs.  Long items (8 stages or more: W_down, and
// W_o at hq * hd >= 8192) are split into two K-slices (fixed by the shape,
// never by R, so every row has the same arithmetic); the slice that finishes
// second adds both partial sums in slice order.  Short items stay whole: a
// slice's partial-sum round trip would cost more than it balances.
constexpr int kSliceMaxItems = kChainSliceMaxItems;

KS_DEV Phase decode(const ChainArgs& a, int k) {
    const int code = a.code[k];
    Phase p;
    if (code >= 4 * a.n_layers) {
        p.kind = CH_LM; p.layer = 0; p.N = a.vocab; p.K = a.d;
    } else {
        p.kind = code & 3;
        p.layer = code >> 2;
        switch (p.kind) {
            case CH_QKV: p.N = a.nqkv; p.K = a.d; break;
            case CH_O: p.N = a.d; p.K = a.hqd; break;
            case CH_GU: p.N = a.F; p.K = a.d; break;
            default: p.N = a.d; p.K = a.F; break;
        }
    }
    p.n_items = (p.N + 15) >> 4;
    const int cols = p.kind == CH_GU ? 512 : 1024;   // k columns per stage
    p.tpi = (p.K + cols - 1) / cols;
    p.n_sl = ((p.kind == CH_O || p.kind == CH_DOWN) && p.n_items <= kSliceMaxItems && p.tpi >= 8) ? 2 : 1;
    p.sl_len = (p.tpi + p.n_sl - 1) / p.n_sl;
    p.n_units = p.n_items * p.n_sl;
    return p;
}
KS_DEV bool normed_input(int kind) { return kind == CH_QKV || kind == CH_GU || kind == CH_LM; }
KS_DEV int stage_cols(int kind) { return kind == CH_GU ? 512 : 1024; }

// Wavefront between phases: a stage of phase k reads columns kt * cols ..
// of phase k - 1's output, so it waits only for the row groups that produce
// them (block kt of phase k - 1), not for the whole phase.  Each finished row
// group of phase k - 1 adds 1 to its block's counter.
constexpr int kMaxBlocks = 64;
KS_DEV int block_rowgroups(int n_out, int cols, int b) {   // row groups of block b
    const int first = b * (cols / 16);
    const int last = min((n_out + 15) / 16, (b + 1) * (cols / 16));
    return last - first;
}
KS_DEV const CUtensorMap* amap_of(const ChainArgs& a, int kind) {
    return &a.amap[kind == CH_GU ? 1 : kind == CH_O ? 2 : kind == CH_DOWN ? 3 : 0];
}
// K % 256 == 0: the activation map is 3-D and a stage is one copy
KS_DEV bool stage_maps(const Phase& P) { return (P.K & 255) == 0; }
// K % 64 == 0: the weight map is 3-D and a stage's weights are one copy
KS_DEV bool weight_3d(const Phase& P) { return (P.K & 63) == 0; }

// Independent accumulator chains per consumer warp: the MMAs of a stage go
// round-robin to kChains accumulators, so consecutive MMAs do not wait on each
// other's results (one dependent chain made the loop latency-bound).  The
// chains are added in chain order at the end of an item: a fixed order that
// depends on neither R nor the CTA.
constexpr int kChains = 2;

// One stage of one consumer warp: its quarter of the stage's columns.
template <int NT, bool PAIR>
KS_DEV void mma_stage(const __nv_bfloat16* st, int R, int warp, int lane, float (&acc)[kChains][NT][4],
                      float (&accu)[kChains][NT][4]) {
    constexpr int kNB = PAIR ? 2 : 4;              // 256-column activation boxes per stage
    constexpr int kWarpCols = 256 * kNB / 4;
    const int g = lane >> 2, t4 = lane & 3;
    const int wb = (warp * kWarpCols) / 256, wc = (warp * kWarpCols) % 256;
    // weights: chunk c (64 columns) of 16 rows at c * 2 KB, row r at r * 128 B,
    // 16-byte unit u at (u ^ (r & 7)) * 16; rows g and g + 8 share the XOR
    const unsigned char* wbase = reinterpret_cast<const unsigned char*>(st) + g * 128;
    const __nv_bfloat16* ap = st + 4 * kBoxElems + wb * (256 * R) + g * 256 + wc + 8 * t4;
    const uint4 z = make_uint4(0, 0, 0, 0);
#pragma unroll
    for (int ks = 0; ks < kWarpCols / 32; ++ks) {
        const int j0 = warp * kWarpCols + 32 * ks;               // first column of the step
        const int off = (j0 >> 6) * kChunkBytes + (((((j0 & 63) >> 3) + t4) ^ g) << 4);
        const uint4 w0 = lds128(wbase + off);
        const uint4 w1 = lds128(wbase + off + 8 * 128);
        uint4 u0 = z, u1 = z;
        if (PAIR) {   // up rows: the second half of the stage (8 chunks on)
            u0 = lds128(wbase + 8 * kChunkBytes + off);
            u1 = lds128(wbase + 8 * kChunkBytes + off + 8 * 128);
        }
        const int c0 = (2 * ks) % kChains, c1 = (2 * ks + 1) % kChains;   // constants once unrolled
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
            const uint4 bv = (nt * 8 + g < R) ? lds128(ap + nt * 8 * 256 + 32 * ks) : z;
            mma_bf16(acc[c0][nt], w0.x, w1.x, w0.y, w1.y, bv.x, bv.y);
            mma_bf16(acc[c1][nt], w0.z, w1.z, w0.w, w1.w, bv.z, bv.w);
            if (PAIR) {
                mma_bf16(accu[c0][nt], u0.x, u1.x, u0.y, u1.y, bv.x, bv.y);
                mma_bf16(accu[c1][nt], u0.z, u1.z, u0.w, u1.w, bv.z, bv.w);
            }
        }
    }
}

// Item epilogue on warp 0 (after the warp-order sum).  Fragment (nt, i) of
// lane (g, t) is feature it * 16 + g + 8 (i >> 1), row nt * 8 + 2 t + (i & 1).
// Argmax key of (logit v, token i): larger v first, then the lower id; an
// unsigned 64-bit max over keys is the argmax in any order of merging.
KS_DEV unsigned long long argmax_key(float v, int i) {
    const uint32_t b = __float_as_uint(v);
    const uint32_t ord = (b & 0x80000000u) ? ~b : (b | 0x80000000u);
    return ((unsigned long long)ord << 32) | (0xFFFFFFFFu - (uint32_t)i);
}

template <int NT>
KS_DEV void epilogue(const ChainArgs& a, const Phase& P, int k, int it, float (&acc)[NT][4],
                     float (&accu)[NT][4], const float* scale, float (&run_v)[NT][2], int (&run_i)[NT][2]) {
    const int lane = threadIdx.x & 31;
    const int g = lane >> 2, t4 = lane & 3;
    float ssq[NT][2], bv[NT][2];
    int bi[NT][2];
#pragma unroll
    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int c = 0; c < 2; ++c) {
            ssq[nt][c] = 0.f;
            bv[nt][c] = -INFINITY;
            bi[nt][c] = INT_MAX;
        }
    const bool resid = P.kind == CH_O || P.kind == CH_DOWN;
    float* cap = nullptr;
    if (resid && a.capture) cap = a.capture + (size_t)(2 * P.layer + 1 + (P.kind == CH_DOWN)) * a.capture_plane;
    const __nv_bfloat16* gain = a.gain[k];
#pragma unroll
    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int n = it * 16 + g + 8 * (i >> 1);
            const int r = nt * 8 + 2 * t4 + (i & 1);
            if (n >= P.N || r >= a.R) continue;
            const float v = acc[nt][i] * scale[r];
            switch (P.kind) {
                case CH_QKV:
                    a.qkv[(size_t)r * a.nqkv + n] = v;
                    break;
                case CH_GU:
                    a.act[(size_t)r * a.F + n] = __float2bfloat16_rn(silu(v) * (accu[nt][i] * scale[r]));
                    break;
                case CH_LM:
                    a.logits[(size_t)r * a.vocab + n] = v;
                    if (better(v, n, bv[nt][i & 1], bi[nt][i & 1])) {
                        bv[nt][i & 1] = v;
                        bi[nt][i & 1] = n;
                    }
                    break;
                default: {  // residual add; the new residual feeds the next RMSNorm
                    float* x = a.x + (size_t)r * a.d + n;
                    const float nx = __ldcg(x) + v;
                    *x = nx;
                    if (cap) cap[(size_t)r * a.d + n] = nx;
                    a.xg[(size_t)r * a.d + n] = __float2bfloat16_rn(nx * __bfloat162float(gain[n]));
                    ssq[nt][i & 1] = fmaf(nx, nx, ssq[nt][i & 1]);
                }
            }
        }
    if (resid || P.kind == CH_LM) {
        // over the 8 lanes with the same t (features g and g + 8 of the item)
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
#pragma unroll
            for (int c = 0; c < 2; ++c) {
                const int r = nt * 8 + 2 * t4 + c;
#pragma unroll
                for (int o = 4; o < 32; o <<= 1) {
                    if (resid) {
                        ssq[nt][c] += __shfl_xor_sync(0xffffffffu, ssq[nt][c], o);
                    } else {
                        const float ov = __shfl_xor_sync(0xffffffffu, bv[nt][c], o);
                        const int oi = __shfl_xor_sync(0xffffffffu, bi[nt][c], o);
                        if (better(ov, oi, bv[nt][c], bi[nt][c])) {
                            bv[nt][c] = ov;
                            bi[nt][c] = oi;
                        }
                    }
                }
                if (resid) {
                    if (g == 0 && r < a.R) a.ss[it * kMaxRows + r] = ssq[nt][c];
                } else if (better(bv[nt][c], bi[nt][c], run_v[nt][c], run_i[nt][c])) {
                    run_v[nt][c] = bv[nt][c];   // this CTA's best of the phase so far
                    run_i[nt][c] = bi[nt][c];
                }
            }
    }
}

// 1 / rms of each of the R rows from the 16-feature partial sums of squares
// of the residual (ss[group][row]): lane l adds groups l, l + 32, ... in that
// order, then a butterfly, and lane 0's total is used; the same order for
// every R.  A group's row sums are contiguous, so all rows load together.
template <int NT>
KS_DEV void row_scales(const ChainArgs& a, int lane, float* out) {
    constexpr int kRows = NT * 8;
    const int R = a.R;   // <= kRows
    const int groups = (a.d + 15) >> 4;
    float s[kRows];
#pragma unroll
    for (int r = 0; r < kRows; ++r) s[r] = 0.f;
#pragma unroll 2
    for (int q = lane; q < groups; q += 32) {
        const float4* src = reinterpret_cast<const float4*>(a.ss + (size_t)q * kMaxRows);
#pragma unroll
        for (int v = 0; v < kRows / 4; ++v) {
            if (4 * v < R) {
                const float4 f = __ldcg(src + v);
                s[4 * v] += f.x;
                s[4 * v + 1] += f.y;
                s[4 * v + 2] += f.z;
                s[4 * v + 3] += f.w;
            }
        }
    }
#pragma unroll
    for (int r = 0; r < kRows; ++r) {
        if (r < R) {
            const float t = warp_sum(s[r]);
            if (lane == 0) out[r] = rsqrtf(t / (float)a.d + a.eps);
        }
    }
    __syncwarp();
}

// One thread per CTA, as the CTA leaves: the last CTA of the launch to leave
// resets the queues and counters of its counter set for a later launch.
KS_DEV void count_out(int n_phases, int* queue, int* done, int* exits, int* blocks) {
    __threadfence();
    if (atomicAdd(exits, 1) == (int)gridDim.x - 1) {
        __threadfence();
        for (int k = 0; k < n_phases; ++k) {
            queue[k] = 0;
            done[k] = 0;
            for (int b = 0; b < kMaxBlocks; ++b) blocks[k * kMaxBlocks + b] = 0;
        }
        *exits = 0;
        __threadfence();
    }
}

template <int NT, int CTAS_PER_SM>
__global__ void __launch_bounds__(kThreads, CTAS_PER_SM) chain_kernel(const __grid_constant__ ChainArgs a) {
    // A draft pass after the dynamic exit: nothing to do.  The flag only
    // changes between passes, so every CTA of the launch sees the same value.
    if (a.stop && *a.stop) return;
    extern __shared__ unsigned char smem_raw[];
    // 1024-byte aligned: the 128-byte swizzle pattern repeats every 1024 bytes
    __nv_bfloat16* ring = reinterpret_cast<__nv_bfloat16*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    __shared__ __align__(8) uint64_t full[kMaxStages];
    __shared__ __align__(8) uint64_t empty[kMaxStages];
    __shared__ __align__(8) uint64_t pub[kMaxStages];
    __shared__ int slot_k[kMaxStages], slot_it[kMaxStages], slot_kt[kMaxStages];
    __shared__ int slot_last[kMaxStages];   // the stage ends this CTA's last item of its phase
    __shared__ int slot_sl[kMaxStages];     // the item's K-slice
    __shared__ float ones[kMaxRows];        // the input scale of phases without a norm
    __shared__ float scale[kMaxRows];       // 1 / rms of the rows (epilogue warp only)
    __shared__ float red[2][4][2][NT * 4][32];   // [buffer][consumer warp][gate, up][fragment][lane]
    __shared__ int red_k[2], red_it[2], red_last[2], red_sl[2];
    __shared__ __align__(8) uint64_t red_full[2];   // 4 consumer warps arrive
    __shared__ __align__(8) uint64_t red_free[2];   // the epilogue warp arrives
    __shared__ int void_job;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int R = a.R, S = a.stages;
    const int stage_elems = 4 * kBoxElems + 4 * 256 * R;
    int* queue = a.counters;
    int* done = a.counters + kChainMaxPhases;
    int* exits = a.counters + 2 * kChainMaxPhases;
    int* blocks = a.counters + 2 * kChainMaxPhases + 1;   // [phase][kMaxBlocks]

    if (tid == 0) {
        // A job whose status word already holds an error is void (the word
        // stays set until the model is created again): the CTA skips its
        // work, so each later launch of the job ends at once instead of
        // running into bounded waits of its own.  One thread reads the word
        // (it can change during the launch) and the barrier below hands the
        // decision to the whole CTA.
        void_job = __ldcg(a.err) != 0;
        for (int i = 0; i < S; ++i) {
            mbar_init(&full[i], 2);
            mbar_init(&empty[i], 4);
            mbar_init(&pub[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&red_full[i], 4);
            mbar_init(&red_free[i], 1);
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (tid < kMaxRows) ones[tid] = 1.f;
    __syncthreads();
    if (void_job) {   // still counted out, so the launch's counters are reset
        if (tid == 0) count_out(a.n_phases, queue, done, exits, blocks);
        return;
    }

    if (warp == kWarpW) {
        // -------------------------------------------------- weight loader
        if (lane == 0) {
            bool ok = true;
            int t = 0;
            auto issue = [&](int k, const Phase& P, int it, int kt, int sl, bool last_item) -> bool {
                const int slot = t % S;
                // self-check: every box coordinate below follows from these ranges
                if (k < 0 || k >= a.n_phases || it < 0 || it >= P.n_items || kt < 0 || kt >= P.tpi || sl < 0 ||
                    sl >= P.n_sl) {
                    set_err(a.err, kErrCheckW);
                    return false;
                }
                if (t >= S && !mbar_wait(&empty[slot], (uint32_t)(((t / S) - 1) & 1), kWaitLimitNs)) return false;
                slot_k[slot] = k;
                slot_it[slot] = it;
                slot_kt[slot] = kt;
                slot_last[slot] = last_item;
                slot_sl[slot] = sl;
                mbar_expect_tx(&full[slot], kWBytes);
                __nv_bfloat16* st = ring + (size_t)slot * stage_elems;
                const CUtensorMap* wm = &a.wmap[k];
                unsigned char* sb = reinterpret_cast<unsigned char*>(st);
                if (weight_3d(P)) {
                    if (P.kind == CH_GU) {   // 8 gate chunks, then 8 up chunks
                        tma_3d(sb, wm, 0, it * 16, 8 * kt, &full[slot]);
                        tma_3d(sb + 8 * kChunkBytes, wm, 0, P.N + it * 16, 8 * kt, &full[slot]);
                    } else {
                        tma_3d(sb, wm, 0, it * 16, 16 * kt, &full[slot]);
                    }
                } else if (P.kind == CH_GU) {
                    for (int c = 0; c < 8; ++c) {
                        tma_2d(sb + c * kChunkBytes, wm, kt * 512 + 64 * c, it * 16, &full[slot]);
                        tma_2d(sb + (8 + c) * kChunkBytes, wm, kt * 512 + 64 * c, P.N + it * 16, &full[slot]);
                    }
                } else {
                    for (int c = 0; c < 16; ++c)
                        tma_2d(sb + c * kChunkBytes, wm, kt * 1024 + 64 * c, it * 16, &full[slot]);
                }
                mbar_arrive(&pub[slot]);
                ++t;
                return true;
            };
            // Work assignment per phase: the CTA's first unit is fixed by its
            // index (unit blockIdx.x, if the phase has that many), so phases
            // with about one unit per CTA (W_o, W_down, QKV) spread over every
            // CTA; further units come from the phase's atomic queue, offset by
            // the grid size.  This launch's queues were zeroed by the launch
            // before the previous one (counter sets alternate), which has
            // completed.  Weight boxes need no input, so the first S stages
            // go out while the previous kernel runs.  No deadlock: every CTA
            // of the grid is co-resident once the kernels before it finish,
            // and a CTA finishes its units of a phase before it waits for the
            // next phase's inputs.
            const int grid = (int)gridDim.x;
            int k = 0;
            Phase P = decode(a, 0);
            int it = (int)blockIdx.x;
            while (ok) {   // `it` counts units: K-slice it / n_items, item it % n_items
                if (it >= P.n_units) {
                    if (++k >= a.n_phases) break;
                    P = decode(a, k);
                    it = (int)blockIdx.x;
                    continue;
                }
                // claimed ahead: its latency hides behind the stream (the
                // ticket is first needed at the unit's last stage, so its
                // round trip overlaps the unit's other stages)
                const int next = P.n_units > grid ? grid + atomicAdd(&queue[k], 1) : INT_MAX;
                // slice-major: every item's first K-slice comes before any
                // second one, so the units taken first (one per CTA) read the
                // previous phase's first blocks, which complete first
                const int sl = it / P.n_items, item = it - sl * P.n_items;
                const int kt0 = sl * P.sl_len, kt1 = min(P.tpi, kt0 + P.sl_len);
                for (int kt = kt0; kt < kt1 && ok; ++kt)
                    ok = issue(k, P, item, kt, sl, kt == kt1 - 1 && next >= P.n_units);
                it = next;
            }
            if (ok) {  // sentinel stage: no more work
                const int slot = t % S;
                if (t >= S && !mbar_wait(&empty[slot], (uint32_t)(((t / S) - 1) & 1), kWaitLimitNs)) {
                    ok = false;
                } else {
                    slot_k[slot] = -1;
                    mbar_arrive(&full[slot]);
                    mbar_arrive(&pub[slot]);
                }
            }
            if (!ok) set_err(a.err, kErrWait);
            // (a dependent launch starts only after this grid's predecessor
            // completed, so the alternating counter sets never overlap)
            grid_dependency_wait();
            grid_launch_dependents();
        }
    } else if (warp == kWarpA) {
        // ---------------------------------------------- activation loader
        grid_dependency_wait();   // the first phase's input comes from the previous kernel
        int cur = -1, ready = 0;
        bool ok = true;
        for (int t = 0;; ++t) {
            const int slot = t % S;
            // lane 0 waits; the shuffle broadcasts the outcome and orders the
            // other lanes' reads of the slot after it
            bool got = true;
            if (lane == 0) got = mbar_wait(&pub[slot], (uint32_t)((t / S) & 1), kWaitLimitNs);
            if (!__shfl_sync(0xffffffffu, (int)got, 0)) {
                ok = false;
                break;
            }
            const int k = slot_k[slot];
            if (k < 0) {
                if (lane == 0) mbar_arrive(&full[slot]);
                break;
            }
            const int kt = slot_kt[slot];
            if (k >= a.n_phases || kt < 0) {   // self-check of the stage record
                if (lane == 0) set_err(a.err, kErrCheckA);
                ok = false;
                break;
            }
            const Phase P = decode(a, k);
            if (kt >= P.tpi) {
                if (lane == 0) set_err(a.err, kErrCheckA);
                ok = false;
                break;
            }
            if (k != cur) {
                cur = k;
                ready = 0;      // blocks of phase k - 1 known to be complete
            }
            if (k > 0 && kt >= ready) {
                // wait for the block of phase k - 1 that this stage reads
                const int n_prev = decode(a, k - 1).N;
                bool dep = true;
                if (lane == 0)
                    dep = wait_at_least(&blocks[(k - 1) * kMaxBlocks + kt],
                                        block_rowgroups(n_prev, stage_cols(P.kind), kt), kWaitLimitNs);
                if (!__shfl_sync(0xffffffffu, (int)dep, 0)) {
                    ok = false;
                    break;
                }
                fence_proxy_async_global();
                if (kt == ready) ++ready;   // stages of an item come in order
            }
            if (lane == 0) {
                const int nb = (P.kind == CH_GU) ? 2 : 4;
                const int cols = 256 * nb;
                mbar_expect_tx(&full[slot], (uint32_t)(nb * 256 * R * 2));
                __nv_bfloat16* dst = ring + (size_t)slot * stage_elems + 4 * kBoxElems;
                const CUtensorMap* am = amap_of(a, P.kind);
                if (stage_maps(P)) tma_3d(dst, am, 0, 0, nb * kt, &full[slot]);
                else for (int b = 0; b < nb; ++b) tma_2d(dst + b * 256 * R, am, kt * cols + 256 * b, 0, &full[slot]);
            }
            __syncwarp();
        }
        if (!ok && lane == 0) set_err(a.err, kErrWait);
    } else if (warp < 4) {
        // ------------------------------------------------------ consumers
        float acc[kChains][NT][4], accu[kChains][NT][4];
        bool failed = false;
        // A wait of one consumer warp that gives up is acted on by all four
        // together at the next stage's barrier (they must leave the loop
        // together: a warp left behind at the named barrier would wait forever).
        bool gave_up = false;
        int n_items = 0;   // items finished by this CTA (selects the partials buffer)
        for (int t = 0;; ++t) {
            const int slot = t % S;
            const bool ok = !gave_up && mbar_wait(&full[slot], (uint32_t)((t / S) & 1), kWaitLimitNs);
            if (consumers_or(!ok)) {
                failed = true;
                break;
            }
            const int k = slot_k[slot];
            const int it = slot_it[slot], kt = slot_kt[slot], sl = slot_sl[slot];
            const bool last_item = slot_last[slot] != 0;
            const int b = n_items & 1;
            if (k < 0) {
                // no more stages: tell the epilogue warp to stop
                if (n_items >= 2 && !mbar_wait(&red_free[b], (uint32_t)(((n_items >> 1) - 1) & 1), kWaitLimitNs))
                    failed = true;
                if (warp == 0 && lane == 0) red_k[b] = -1;
                __syncwarp();
                if (lane == 0) mbar_arrive(&red_full[b]);
                break;
            }
            if (k >= a.n_phases || kt < 0 || it < 0) {   // self-check (the same record in every warp)
                if (lane == 0) set_err(a.err, kErrCheckC);
                failed = true;
                break;
            }
            const Phase P = decode(a, k);
            if (kt >= P.tpi || it >= P.n_items || sl < 0 || sl >= P.n_sl) {
                if (lane == 0) set_err(a.err, kErrCheckC);
                failed = true;
                break;
            }
            const int kt0 = sl * P.sl_len, kt1 = min(P.tpi, kt0 + P.sl_len);
            if (kt == kt0) {
#pragma unroll
                for (int c = 0; c < kChains; ++c)
#pragma unroll
                    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
                        for (int i = 0; i < 4; ++i) acc[c][nt][i] = accu[c][nt][i] = 0.f;
            }
            const __nv_bfloat16* st = ring + (size_t)slot * stage_elems;
            if (P.kind == CH_GU) mma_stage<NT, true>(st, R, warp, lane, acc, accu);
            else mma_stage<NT, false>(st, R, warp, lane, acc, accu);
            __syncwarp();
            if (lane == 0) mbar_arrive(&empty[slot]);   // this warp is done with the stage
            if (kt != kt1 - 1) continue;

            // item done: add the chains in chain order and hand this warp's
            // sums to the epilogue warp through partials buffer b (double
            // buffered: the consumers move straight on to the next item)
#pragma unroll
            for (int c = 1; c < kChains; ++c)
#pragma unroll
                for (int nt = 0; nt < NT; ++nt)
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        acc[0][nt][i] += acc[c][nt][i];
                        accu[0][nt][i] += accu[c][nt][i];
                    }
            if (n_items >= 2 && !mbar_wait(&red_free[b], (uint32_t)(((n_items >> 1) - 1) & 1), kWaitLimitNs)) {
                gave_up = true;   // leave at the next barrier, with the other warps
                continue;
            }
#pragma unroll
            for (int nt = 0; nt < NT; ++nt)
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    red[b][warp][0][nt * 4 + i][lane] = acc[0][nt][i];
                    if (P.kind == CH_GU) red[b][warp][1][nt * 4 + i][lane] = accu[0][nt][i];
                }
            if (warp == 0 && lane == 0) {
                red_k[b] = k;
                red_it[b] = it;
                red_last[b] = last_item;
                red_sl[b] = sl;
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&red_full[b]);
            ++n_items;
        }
        if (failed && lane == 0) set_err(a.err, kErrWait);
    } else if (warp == kWarpE) {
        // --------------------------------------------------- epilogue warp
        grid_dependency_wait();   // epilogues write buffers the previous kernel uses
        float acc[NT][4], accu[NT][4];
        float run_v[NT][2];       // LM head: this CTA's best (logit, id) per row
        int run_i[NT][2];
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
#pragma unroll
            for (int c = 0; c < 2; ++c) {
                run_v[nt][c] = -INFINITY;
                run_i[nt][c] = INT_MAX;
            }
        int items_in_phase = 0;   // items of the current phase finished by this CTA
        int scale_k = -1;         // the phase whose row scales `scale` holds
        bool ok = true;
        for (int n = 0;; ++n) {
            const int b = n & 1;
            if (!mbar_wait(&red_full[b], (uint32_t)((n >> 1) & 1), kWaitLimitNs)) {
                ok = false;
                break;
            }
            const int k = red_k[b];
            if (k < 0) break;
            const int it = red_it[b];
            const bool last_item = red_last[b] != 0;
            if (k >= a.n_phases || it < 0 || it >= decode(a, k).n_items) {   // self-check
                set_err(a.err, kErrCheckE);
                ok = false;
                break;
            }
            const Phase P = decode(a, k);
            // the four warps' K quarters, added in warp order
#pragma unroll
            for (int nt = 0; nt < NT; ++nt)
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    acc[nt][i] = red[b][0][0][nt * 4 + i][lane];
                    accu[nt][i] = (P.kind == CH_GU) ? red[b][0][1][nt * 4 + i][lane] : 0.f;
                }
#pragma unroll
            for (int w = 1; w < 4; ++w)
#pragma unroll
                for (int nt = 0; nt < NT; ++nt)
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        acc[nt][i] += red[b][w][0][nt * 4 + i][lane];
                        if (P.kind == CH_GU) accu[nt][i] += red[b][w][1][nt * 4 + i][lane];
                    }
            const int sl = red_sl[b];
            __syncwarp();
            if (lane == 0) mbar_arrive(&red_free[b]);   // partials read: the buffer is free
            bool complete = true;
            if (P.n_sl > 1) {
                // a K-slice: leave its sums in global memory; the slice that
                // completes the item adds all of them in slice order
                const int g = lane >> 2, t4 = lane & 3;
                float* part = a.slice_part + ((size_t)(k & 1) * kSliceMaxItems + it) * (2 * 256);
#pragma unroll
                for (int nt = 0; nt < NT; ++nt)
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                        part[sl * 256 + (g + 8 * (i >> 1)) * 16 + nt * 8 + 2 * t4 + (i & 1)] = acc[nt][i];
                __syncwarp();
                int last = 0;
                if (lane == 0) {
                    __threadfence();
                    int* tk = a.slice_ticket + (k & 1) * kSliceMaxItems + it;
                    last = atomicAdd(tk, 1) == P.n_sl - 1;
                    if (last) *tk = 0;   // every slice has arrived: ready for the next use
                }
                complete = __shfl_sync(0xffffffffu, last, 0) != 0;
                if (complete) {
                    __threadfence();
#pragma unroll
                    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
                        for (int i = 0; i < 4; ++i) {
                            const int o = (g + 8 * (i >> 1)) * 16 + nt * 8 + 2 * t4 + (i & 1);
                            float v = __ldcg(&part[o]);
                            for (int q = 1; q < P.n_sl; ++q) v += __ldcg(&part[q * 256 + o]);
                            acc[nt][i] = v;
                        }
                }
            }
            if (complete && normed_input(P.kind) && k != scale_k) {
                // This CTA's first item of a normed phase: its last stage
                // waited for every block of phase k - 1 (an item's stages
                // cover them all), so every row group's partial sums of
                // squares are written.
                scale_k = k;
                row_scales<NT>(a, lane, scale);
            }
            if (complete) {
                epilogue<NT>(a, P, k, it, acc, accu, normed_input(P.kind) ? scale : ones, run_v, run_i);
                ++items_in_phase;
            }
            if (complete && k + 1 < a.n_phases) {
                // publish this row group to the next phase's stages that read it
                fence_proxy_async_global();
                __syncwarp();
                if (lane == 0) {
                    __threadfence();
                    atomicAdd(&blocks[k * kMaxBlocks + (it * 16) / stage_cols(decode(a, k + 1).kind)], 1);
                }
            }
            if (last_item) {
                // this CTA has no more items in the phase: publish them all
                // with one release (the next phase reads them by TMA)
                if (P.kind == CH_LM) {
                    // merge this CTA's per-row best into the global keys
                    const int g = lane >> 2, t4 = lane & 3;
#pragma unroll
                    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
                        for (int c = 0; c < 2; ++c) {
                            const int r = nt * 8 + 2 * t4 + c;
                            if (g == 0 && r < R && run_i[nt][c] != INT_MAX)
                                atomicMax(&a.best[r], argmax_key(run_v[nt][c], run_i[nt][c]));
                        }
                }
                fence_proxy_async_global();
                __syncwarp();
                int fin = 0;
                if (lane == 0) {
                    __threadfence();
                    const int prev = atomicAdd(&done[k], items_in_phase);
                    fin = (P.kind == CH_LM && prev + items_in_phase == P.n_items);
                }
                items_in_phase = 0;
                if (__shfl_sync(0xffffffffu, fin, 0)) {
                    // every CTA has merged: read the keys (and leave them zero)
                    __threadfence();
                    if (lane < R) {
                        const unsigned long long key = atomicExch(&a.best[lane], 0ull);
                        a.tokens[lane] = key == 0ull ? 0 : (int)(0xFFFFFFFFu - (uint32_t)(key & 0xFFFFFFFFull));
                    }
                }
            }
        }
        if (!ok && lane == 0) set_err(a.err, kErrWait);
    }

    // the last CTA to leave resets the queues and counters for the next launch
    __syncthreads();
    if (tid == 0) count_out(a.n_phases, queue, done, exits, blocks);
}

}  // namespace

size_t chain_counter_ints() { return 2 * (size_t)kChainMaxPhases + 1 + (size_t)kChainMaxPhases * kMaxBlocks; }

cudaError_t launch_chain(const ChainArgs& args, cudaStream_t s) {
    if (args.R < 1 || args.R > kMaxRows || args.n_phases < 1 || args.n_phases > kChainMaxPhases ||
        args.err == nullptr || args.counters == nullptr)
        return cudaErrorInvalidValue;
    ChainArgs a = args;
    const int per_sm = a.R <= 8 ? 2 : 1;
    const size_t stage_bytes = kWBytes + 4u * 256u * 2u * (size_t)a.R;
    a.stages = (int)((per_sm == 2 ? kRingBudget2 : kRingBudget1) / stage_bytes);
    if (a.stages > kMaxStages) a.stages = kMaxStages;
    const size_t smem = (size_t)a.stages * stage_bytes + 1024;  // + alignment slack
    auto run = [&](auto kern) -> cudaError_t {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        cudaLaunchConfig_t cfg = {};
        // two CTAs per SM when they fit (they normally do); fewer only slows
        // the launch down, since no CTA waits for one that is not running
        int fit = per_sm;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&fit, kern, kThreads, smem) != cudaSuccess || fit < 1)
            fit = 1;
        cfg.gridDim = dim3(std::min(fit, per_sm) * sm_count());
        cfg.blockDim = dim3(kThreads);
        cfg.dynamicSmemBytes = smem;
        cfg.stream = s;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        return cudaLaunchKernelEx(&cfg, kern, a);
    };
    return per_sm == 2 ? run(chain_kernel<1, 2>) : run(chain_kernel<2, 1>);
}

}  // namespace ks
