// Skinny GEMM kernels for the decode / verify passes (R <= 16 activation rows).
//
// Y[r][n] = sum_k W[n][k] A[r][k]: the per-token projections of the Attn and
// MLP sublayers and the LM head (Sec. 2 decoder; every pass of a1 / a2).  At
// R <= 16 rows the work is a stream over the weights (at most 16 flop per
// weight byte pair), so the bf16 kernel is built to keep HBM busy:
//  * persistent and warp-specialised: one CTA per SM; a producer warp claims
//    work items (16 output features over the full K) and streams their
//    weight and activation tiles with 2-D TMA into a multi-stage shared
//    memory ring (about 150-190 KB in flight per SM, no registers held);
//    four consumer warps split each stage's columns and multiply;
//  * the tiles are fed as the A operand of mma.sync.m16n8k16 (16 weight rows x
//    16 k) and the activation rows as B (16 k x 8 rows); the k-slots of A and
//    B are permuted identically so each lane reads 8 contiguous weights and 8
//    contiguous activations; column j of the result depends only on
//    activation row j, so a row computed alone (greedy decode) and the same
//    row inside a gamma+1-row verify pass are bit-identical;
//  * the consumer warps' K quarters are added in warp order (bf16), K slices
//    of the fp32 kernel in slice order by the last CTA of a group (an atomic
//    ticket, no waiting): results depend only on (N, K), never on R or on
//    which CTA did what;
//  * prologue: optional RMSNorm of the fp32 residual, with the row's sum of
//    squares assembled from per-64-feature partials that the residual's
//    producer wrote (embed or a residual epilogue), summed in group order;
//    epilogues: plain store (QKV), residual add with optional history capture
//    and the new partial sums of squares (W_o, W_down), SwiGLU (gate and up
//    rows paired in one warp), LM head logits with a per-row argmax (ties to
//    the lowest id).
// fp32 models (the tiny parity workload) use a simpler CUDA-core kernel with
// the same tile ownership, epilogues and split rule.
#include "common.cuh"
#include "internal.h"

#include <cudaTypedefs.h>

#include <climits>

namespace ks {

constexpr int kGemvWarps = 4;
constexpr int kRowsPerCta = 16 * kGemvWarps;  // output features per group (CTA or work item)
constexpr int kMaxRows = 16;
constexpr int kKT = 128;                      // k columns per streamed weight tile
constexpr int kKP = kKT + 32;                 // tile row pitch (elements): conflict-free LDS.128
constexpr int kMaxKc = 1024;                  // largest K slice of a bf16 work item
// counters: [0] next work item, [1] finished CTAs, [2 + g] ticket of group g

__host__ __device__ __forceinline__ int div_up(int a, int b) { return (a + b - 1) / b; }

int gemv_grid_x(int N) { return div_up(N, kRowsPerCta); }
int gemv_groups(int N, int dtype) { return dtype == 1 ? div_up(N, 16) : div_up(N, kRowsPerCta); }

static int sm_count() {
    static int n = 0;
    if (n == 0) {
        int dev = 0;
        cudaGetDevice(&dev);
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 152;
    }
    return n;
}


void gemv_plan(GemvArgs& a, int epi) {
    // Depends on (N, K, dtype) only, never on R: the split decides the
    // summation order, which must be the same for 1 row and gamma + 1 rows.
    const int gx = gemv_grid_x(a.N);
    if (a.dtype == 1) {
        // bf16 streaming kernel: 16-row work items over the full K (the four
        // consumer warps of a CTA split K inside each stage), no global split
        a.kc = a.K;
        a.ksplit = 1;
        return;
    }
    int s = 1;
    if (epi != EPI_LMHEAD) {
        s = div_up(5 * 152, gx);
        if (s > 16) s = 16;
        if (s < 1) s = 1;
    }
    int kc = div_up(div_up(a.K, s), 64) * 64;
    if (kc < 64) kc = 64;
    a.kc = kc;
    a.ksplit = div_up(a.K, kc);
}

size_t gemv_partial_floats(int N, int K, int R, int epi, int dtype) {
    GemvArgs a{};
    a.N = N;
    a.K = K;
    a.dtype = dtype;
    gemv_plan(a, epi);
    if (a.ksplit <= 1) return 0;
    return (size_t)a.ksplit * R * N * (epi == EPI_SWIGLU ? 2 : 1);
}

// --------------------------------------------------------------- prologue
// Stage A[r][kbeg .. kbeg + kc) for r < R into shared memory (pitch elements
// per row), applying RMSNorm when norm_gain is set.  Elements past K are 0.
template <typename WT>
KS_DEV void stage_activations(const GemvArgs& a, WT* act, int pitch, int kbeg, float* red) {
    const int tid = threadIdx.x;
    const int R = a.R;
    const int kc = a.kc;
    __syncthreads();  // the previous user of act / red is done
    if (a.norm_gain != nullptr) {
        // inv_rms[r] from the producer's per-64-feature partial sums of
        // squares, added in group order (the same for every CTA and every R)
        const float* x = reinterpret_cast<const float*>(a.in);
        const WT* gain = reinterpret_cast<const WT*>(a.norm_gain);
        if (tid < R) {
            float s = 0.f;
            for (int g = 0; g < a.ss_groups; ++g) s += a.ss_in[g * kMaxRows + tid];
            red[tid] = rsqrtf(s / (float)a.K + a.eps);
        }
        __syncthreads();
        for (int idx = tid; idx < R * kc; idx += blockDim.x) {
            const int r = idx / kc, k = idx - r * kc;
            const int kg = kbeg + k;
            float v = 0.f;
            if (kg < a.K) v = (x[(size_t)r * a.in_ld + kg] * red[r]) * to_float(gain[kg]);
            act[r * pitch + k] = from_float<WT>(v);
        }
    } else {
        const WT* in = reinterpret_cast<const WT*>(a.in);
        for (int idx = tid; idx < R * kc; idx += blockDim.x) {
            const int r = idx / kc, k = idx - r * kc;
            const int kg = kbeg + k;
            act[r * pitch + k] = kg < a.K ? in[(size_t)r * a.in_ld + kg] : from_float<WT>(0.f);
        }
    }
    __syncthreads();
}

// -------------------------------------------------------------- fp32 rows
// fp32: the warp computes its 16 rows one at a time (lanes stride over k in
// float4 steps, butterfly sum), then redistributes the results into the same
// fragment layout the bf16 path produces.
template <int NT, bool PAIR>
KS_DEV void fma_rows(const float* W, int K, int N, int n_base, int kbeg, const float* act,
                     int pitch, int R, int kc, int kvalid, float* tile /* [2][16][16] per warp */,
                     float (&acc)[NT][4], float (&accu)[NT][4]) {
    const int lane = threadIdx.x & 31, g = lane >> 2, t = lane & 3;
    for (int half = 0; half < (PAIR ? 2 : 1); ++half) {
        for (int j = 0; j < 16; ++j) {
            const int n = n_base + j;
            float s[kMaxRows];
#pragma unroll
            for (int r = 0; r < kMaxRows; ++r) s[r] = 0.f;
            if (n < N) {
                const float* wr = W + (size_t)(n + half * N) * K + kbeg;
                for (int k = 4 * lane; k < kvalid; k += 128) {
                    const float4 w = *reinterpret_cast<const float4*>(wr + k);
#pragma unroll
                    for (int r = 0; r < kMaxRows; ++r) {
                        if (r < R) {
                            const float4 x = *reinterpret_cast<const float4*>(act + r * pitch + k);
                            s[r] = fmaf(w.x, x.x, s[r]);
                            s[r] = fmaf(w.y, x.y, s[r]);
                            s[r] = fmaf(w.z, x.z, s[r]);
                            s[r] = fmaf(w.w, x.w, s[r]);
                        }
                    }
                }
            }
#pragma unroll
            for (int r = 0; r < kMaxRows; ++r) {
                const float v = warp_sum(s[r]);
                if (lane == 0) tile[(half * 16 + j) * 16 + r] = v;
            }
        }
    }
    __syncwarp();
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
        const int c = nt * 8 + 2 * t;
        acc[nt][0] = tile[g * 16 + c];
        acc[nt][1] = tile[g * 16 + c + 1];
        acc[nt][2] = tile[(g + 8) * 16 + c];
        acc[nt][3] = tile[(g + 8) * 16 + c + 1];
        if (PAIR) {
            accu[nt][0] = tile[(16 + g) * 16 + c];
            accu[nt][1] = tile[(16 + g) * 16 + c + 1];
            accu[nt][2] = tile[(16 + g + 8) * 16 + c];
            accu[nt][3] = tile[(16 + g + 8) * 16 + c + 1];
        }
    }
}

// --------------------------------------------------------------- epilogue
template <typename WT, int EPI>
KS_DEV void apply_epilogue(const GemvArgs& a, int n, int r, float v, float vu) {
    if (EPI == EPI_STORE) {
        a.out[(size_t)r * a.out_ld + n] = v;
    } else if (EPI == EPI_RESID) {
        float* x = a.resid + (size_t)r * a.resid_ld + n;
        const float nx = *x + v;
        *x = nx;
        if (a.capture) a.capture[(size_t)r * a.capture_ld + n] = nx;
        if (a.xg_out)
            a.xg_out[(size_t)r * a.resid_ld + n] =
                __float2bfloat16_rn(nx * to_float(reinterpret_cast<const __nv_bfloat16*>(a.next_gain)[n]));
    } else if (EPI == EPI_SWIGLU) {
        WT* act = reinterpret_cast<WT*>(a.act);
        act[(size_t)r * a.act_ld + n] = from_float<WT>(silu(v) * vu);
    }
}

// After a residual update of features [64 b, 64 b + 64): per row, the sum of
// squares of the new residual over those features, for the next RMSNorm.
// Lane l adds features l and l + 32, then a butterfly: a fixed order.
// Barrier of the 128 threads that own the output fragments: the whole CTA in
// the fp32 kernel, the four consumer warps (named barrier 1) in the streaming
// kernel, whose producer warp never joins.
template <bool CONSUMERS>
KS_DEV void out_sync() {
    if (CONSUMERS) asm volatile("bar.sync 1, 128;" ::: "memory");
    else __syncthreads();
}

template <bool CONSUMERS = false>
KS_DEV void residual_sumsq(const GemvArgs& a, int group) {
    out_sync<CONSUMERS>();
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int n0 = group * kRowsPerCta;
    // 16-feature partials: lanes 0-15 and 16-31 each reduce one half-warp
    for (int r = warp; r < a.R; r += kGemvWarps) {
        const float* x = a.resid + (size_t)r * a.resid_ld;
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int n = n0 + 32 * h + lane;
            float s = (n < a.N) ? x[n] * x[n] : 0.f;
#pragma unroll
            for (int o = 8; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
            if ((lane & 15) == 0) {
                const int q = (n0 + 32 * h + lane) / kSsGroup;
                if (q * kSsGroup < a.N) a.ss_out[q * kMaxRows + r] = s;
            }
        }
    }
}

// LM head: after the logits of features [64 g, 64 g + 64) are in global memory,
// each row's best (value, index) of the group -> amax[g][r].
template <bool CONSUMERS = false>
KS_DEV void group_argmax(const GemvArgs& a, int group) {
    out_sync<CONSUMERS>();
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int n0 = group * kRowsPerCta;
    for (int r = warp; r < a.R; r += kGemvWarps) {
        const float* lg = a.logits + (size_t)r * a.logits_ld;
        float bv = -INFINITY;
        int bi = INT_MAX;
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int n = n0 + lane + 32 * h;
            if (n < a.N) {
                const float v = lg[n];
                if (better(v, n, bv, bi)) { bv = v; bi = n; }
            }
        }
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const float ov = __shfl_xor_sync(0xffffffffu, bv, o);
            const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
            if (better(ov, oi, bv, bi)) { bv = ov; bi = oi; }
        }
        if (lane == 0) {
            a.amax_val[group * kMaxRows + r] = bv;
            a.amax_idx[group * kMaxRows + r] = bi;
        }
    }
}

// LM head, last CTA of the launch: per row, the best candidate over groups.
KS_DEV void final_argmax(const GemvArgs& a, int groups) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int r = warp; r < a.R; r += kGemvWarps) {
        float bv = -INFINITY;
        int bi = INT_MAX;
        for (int c = lane; c < groups; c += 32) {
            const float v = __ldcg(&a.amax_val[c * kMaxRows + r]);
            const int i = __ldcg(&a.amax_idx[c * kMaxRows + r]);
            if (better(v, i, bv, bi)) { bv = v; bi = i; }
        }
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const float ov = __shfl_xor_sync(0xffffffffu, bv, o);
            const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
            if (better(ov, oi, bv, bi)) { bv = ov; bi = oi; }
        }
        if (lane == 0) a.tokens[r] = (bi == INT_MAX) ? 0 : bi;
    }
}

// ---------------------------------------------------- fp32 register kernel
// One CTA per (64-feature group, K slice); used for fp32 models only.
template <int NT, int EPI>
__global__ void __launch_bounds__(128) gemv_f32_kernel(const GemvArgs a) {
    constexpr bool PAIR = (EPI == EPI_SWIGLU);
    extern __shared__ __align__(16) unsigned char smem[];
    __shared__ float red[kGemvWarps * kMaxRows + kMaxRows];
    __shared__ int is_last;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int g = lane >> 2, t = lane & 3;
    const int kbeg = blockIdx.y * a.kc;
    const int kvalid = min(a.kc, a.K - kbeg);
    const int pitch = a.kc + 4;
    float* act = reinterpret_cast<float*>(smem);
    stage_activations<float>(a, act, pitch, kbeg, red);

    const int n_base = blockIdx.x * kRowsPerCta + warp * 16;
    float acc[NT][4], accu[NT][4];
#pragma unroll
    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int i = 0; i < 4; ++i) acc[nt][i] = accu[nt][i] = 0.f;
    float* tile = reinterpret_cast<float*>(smem + sizeof(float) * (size_t)a.R * pitch) + warp * 2 * 16 * 16;
    fma_rows<NT, PAIR>(reinterpret_cast<const float*>(a.W), a.K, a.N, n_base, kbeg, act, pitch, a.R, a.kc,
                       kvalid, tile, acc, accu);

    const int group = blockIdx.x;
    if (a.ksplit == 1) {
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int n = n_base + g + 8 * (i >> 1);
                const int r = nt * 8 + 2 * t + (i & 1);
                if (n < a.N && r < a.R) {
                    if (EPI == EPI_LMHEAD) a.logits[(size_t)r * a.logits_ld + n] = acc[nt][i];
                    else apply_epilogue<float, EPI>(a, n, r, acc[nt][i], accu[nt][i]);
                }
            }
    } else {
        const int NP = PAIR ? 2 * a.N : a.N;
        float* mine = a.partial + (size_t)blockIdx.y * a.R * NP;
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int n = n_base + g + 8 * (i >> 1);
                const int r = nt * 8 + 2 * t + (i & 1);
                if (n < a.N && r < a.R) {
                    mine[(size_t)r * NP + n] = acc[nt][i];
                    if (PAIR) mine[(size_t)r * NP + a.N + n] = accu[nt][i];
                }
            }
        __threadfence();
        __syncthreads();
        if (tid == 0) is_last = (atomicAdd(&a.counters[2 + group], 1) == a.ksplit - 1);
        __syncthreads();
        if (!is_last) return;
        __threadfence();
        const int row0 = group * kRowsPerCta;
        for (int idx = tid; idx < kRowsPerCta * a.R; idx += blockDim.x) {
            const int r = idx / kRowsPerCta;
            const int n = row0 + (idx - r * kRowsPerCta);
            if (n >= a.N) continue;
            float v = 0.f, vu = 0.f;
            for (int sl = 0; sl < a.ksplit; ++sl) {
                const float* pp = a.partial + ((size_t)sl * a.R + r) * NP;
                v += __ldcg(pp + n);
                if (PAIR) vu += __ldcg(pp + a.N + n);
            }
            if (EPI == EPI_LMHEAD) a.logits[(size_t)r * a.logits_ld + n] = v;
            else apply_epilogue<float, EPI>(a, n, r, v, vu);
        }
        if (tid == 0) a.counters[2 + group] = 0;
    }
    if (EPI == EPI_RESID) residual_sumsq(a, group);
    if (EPI == EPI_LMHEAD) {
        group_argmax(a, group);
        __threadfence();
        __syncthreads();
        if (tid == 0) is_last = (atomicAdd(&a.counters[1], 1) == (int)(gridDim.x * gridDim.y) - 1);
        __syncthreads();
        if (!is_last) return;
        __threadfence();
        final_argmax(a, gridDim.x);
        if (tid == 0) a.counters[1] = 0;
    }
}

// ------------------------------------------------- bf16 streaming kernel
// Work item = 16 output features (16 weight rows, or 16 gate + 16 up rows)
// over the full K.  A ring stage holds NB x 256 columns of the item's weight
// rows (one 256 x 16 TMA box per 256 columns and row block) and of its R
// activation rows (256 x R boxes), rows 512 bytes apart.  The four
// consumer warps split each stage's columns evenly; at the end of an item
// their partial fragments are added in warp order in shared memory.
//
// Warp specialisation: warp 4 (the producer) claims items and fills stages
// with 2-D TMA loads that complete on the stage's `full` mbarrier; warps 0-3
// wait on `full`, multiply, and arrive on the stage's `empty` mbarrier, which
// the producer waits on before refilling.  Item epilogues run on the
// consumers only, so the weight stream never pauses for them.
//
// Launched with programmatic stream serialisation: the barrier set-up and
// the weight boxes of the first item (its index is the CTA index) are issued
// before griddepcontrol.wait; everything that reads or writes data another
// kernel touches comes after it.
template <int NT, bool PAIR>
struct StreamCfg {
    static constexpr int kNB = PAIR ? 2 : 4;              // 256-column boxes per stage
    static constexpr int kCols = 256 * kNB;               // k columns per stage
    static constexpr int kWarpCols = kCols / 4;           // columns per consumer warp
    static constexpr int kBoxW = 256 * 16;                // elements of a weight box
    static constexpr int kARows = 8 * NT;
    static constexpr int kBoxA = 256 * kARows;            // elements of an activation box
    static constexpr int kWBlocks = PAIR ? 2 : 1;
    static constexpr int kStage = kWBlocks * kNB * kBoxW + kNB * kBoxA;  // elements per stage
    static constexpr uint32_t kBytes = 2u * kStage;
    static constexpr int kStages = (int)((200u * 1024u) / kBytes) > 8 ? 8 : (int)((200u * 1024u) / kBytes);
};

template <int NT, bool PAIR>
static size_t stream_smem() {
    using C = StreamCfg<NT, PAIR>;
    return sizeof(__nv_bfloat16) * (size_t)C::kStages * C::kStage + 128;  // + alignment slack
}

KS_DEV uint32_t smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

KS_DEV void mbar_init(uint64_t* bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
KS_DEV void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
                 : "memory");
}
KS_DEV void mbar_arrive(uint64_t* bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
KS_DEV void tma_2d(void* dst, const CUtensorMap* map, int x, int y, uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], "
        "[%4];" ::"r"(smem_u32(dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_u32(bar))
        : "memory");
}
KS_DEV void grid_dependency_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
KS_DEV uint64_t global_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t));
    return t;
}
// Wait for the mbarrier phase with the given parity; gives up after limit_ns.
KS_DEV bool mbar_wait(uint64_t* bar, uint32_t parity, uint64_t limit_ns) {
    const uint32_t b = smem_u32(bar);
    uint64_t t0 = 0;
    for (uint32_t i = 0;; ++i) {
        uint32_t ok;
        asm volatile(
            "{ .reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2; selp.u32 %0, 1, 0, p; }"
            : "=r"(ok)
            : "r"(b), "r"(parity)
            : "memory");
        if (ok) return true;
        if (i == 0) t0 = global_ns();
        else if ((i & 63) == 0 && global_ns() - t0 > limit_ns) return false;
    }
}
// Barrier of the four consumer warps that also ORs a flag across them.
KS_DEV bool consumers_or(bool v) {
    uint32_t r;
    asm volatile(
        "{ .reg .pred p, q; setp.ne.u32 p, %1, 0; bar.red.or.pred q, 1, 128, p; selp.u32 %0, 1, 0, q; }"
        : "=r"(r)
        : "r"((uint32_t)v)
        : "memory");
    return r != 0;
}

constexpr uint64_t kWaitLimitNs = 2000000000ull;  // 2 s: only a broken copy waits this long

// Persistent: grid = SM count, one CTA (5 warps) per SM.  CTA b starts with
// item b, then takes gridDim.x + (ticket from counters[0]); its tiles go
// through ring slot t % S in order.
template <int NT, int EPI>
__global__ void __launch_bounds__(160, 1) gemv_stream_kernel(const __grid_constant__ GemvArgs a) {
    constexpr bool PAIR = (EPI == EPI_SWIGLU);
    using Cfg = StreamCfg<NT, PAIR>;
    constexpr int S = Cfg::kStages;
    extern __shared__ unsigned char smem_raw[];
    __nv_bfloat16* stages = reinterpret_cast<__nv_bfloat16*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 127) & ~static_cast<uintptr_t>(127));
    __shared__ __align__(8) uint64_t full[S];
    __shared__ __align__(8) uint64_t empty[S];
    __shared__ int slot_item[S];
    __shared__ int slot_kt[S];
    __shared__ float scale[kMaxRows];
    __shared__ float red[3][2][NT * 4][32];   // partial fragments of warps 1-3
    __shared__ int is_last;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int g = lane >> 2, t4 = lane & 3;
    const int n_items = div_up(a.N, 16);
    const int TPI = div_up(a.K, Cfg::kCols);

    if (tid == 0) {
        for (int i = 0; i < S; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], kGemvWarps);
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();

    if (warp == kGemvWarps) {
        // ------------------------------------------------------ producer
        if (lane != 0) return;
        auto load_w = [&](int slot, int it, int kt) {
            __nv_bfloat16* st = stages + (size_t)slot * Cfg::kStage;
            const int k0 = kt * Cfg::kCols;
#pragma unroll
            for (int b = 0; b < Cfg::kNB; ++b) {
                tma_2d(st + b * Cfg::kBoxW, &a.wmap, k0 + 256 * b, it * 16, &full[slot]);
                if (PAIR) tma_2d(st + (Cfg::kNB + b) * Cfg::kBoxW, &a.wmap, k0 + 256 * b, a.N + it * 16, &full[slot]);
            }
        };
        auto load_x = [&](int slot, int kt) {
            __nv_bfloat16* st = stages + (size_t)slot * Cfg::kStage + Cfg::kWBlocks * Cfg::kNB * Cfg::kBoxW;
            const int k0 = kt * Cfg::kCols;
#pragma unroll
            for (int b = 0; b < Cfg::kNB; ++b) tma_2d(st + b * Cfg::kBoxA, &a.xmap, k0 + 256 * b, 0, &full[slot]);
        };
        // bytes landing per stage: the weight boxes plus activation boxes of R rows
        const uint32_t bytes = 2u * (Cfg::kWBlocks * Cfg::kNB * Cfg::kBoxW + Cfg::kNB * 256 * a.R);
        // first item (static): weights before the grid dependency resolves
        int it = blockIdx.x;
        int t = 0;
        const int pre = (it < n_items) ? min(S, TPI) : 0;
        for (int kt = 0; kt < pre; ++kt) {
            slot_item[kt] = it;
            slot_kt[kt] = kt;
            mbar_expect_tx(&full[kt], bytes);
            load_w(kt, it, kt);
        }
        grid_dependency_wait();
        for (int kt = 0; kt < pre; ++kt) load_x(kt, kt);
        bool ok = true;
        int kt0 = pre;
        t = pre;
        for (;;) {
            if (it < n_items) {
                for (int kt = kt0; kt < TPI; ++kt, ++t) {
                    const int slot = t % S;
                    if (t >= S && !mbar_wait(&empty[slot], (uint32_t)(((t / S) - 1) & 1), kWaitLimitNs)) {
                        ok = false;
                        break;
                    }
                    slot_item[slot] = it;
                    slot_kt[slot] = kt;
                    mbar_expect_tx(&full[slot], bytes);
                    load_w(slot, it, kt);
                    load_x(slot, kt);
                }
                if (!ok) break;
                it = gridDim.x + atomicAdd(&a.counters[0], 1);
                kt0 = 0;
                continue;
            }
            // no more work: a sentinel stage tells the consumers
            const int slot = t % S;
            if (t >= S && !mbar_wait(&empty[slot], (uint32_t)(((t / S) - 1) & 1), kWaitLimitNs)) {
                ok = false;
                break;
            }
            slot_item[slot] = -1;
            mbar_arrive(&full[slot]);
            break;
        }
        if (!ok) atomicExch(a.err, 1);
        // nothing more to stream: the next kernel may start on SMs as they free up
        asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
        return;
    }

    // ---------------------------------------------------------- consumers
    grid_dependency_wait();
    if (tid < kMaxRows) {
        // per-row output scale: 1 / rms(x) from the producer's sums of squares
        float sc = 1.f;
        if (a.ss_in != nullptr && tid < a.R) {
            float ssum = 0.f;
            for (int q = 0; q < a.ss_groups; ++q) ssum += a.ss_in[q * kMaxRows + tid];
            sc = rsqrtf(ssum / (float)a.K + a.eps);
        }
        scale[tid] = sc;
    }
    out_sync<true>();

    const uint4 z = make_uint4(0, 0, 0, 0);
    // this warp's columns inside a stage: box wb, columns [wc, wc + kWarpCols)
    const int wb = (warp * Cfg::kWarpCols) / 256, wc = (warp * Cfg::kWarpCols) % 256;
    float acc[NT][4], accu[NT][4];
    bool failed = false;
    for (int t = 0;; ++t) {
        const int slot = t % S;
        const bool ok = mbar_wait(&full[slot], (uint32_t)((t / S) & 1), kWaitLimitNs);
        if (consumers_or(!ok)) {
            failed = true;
            break;
        }
        const int it = slot_item[slot];
        if (it < 0) break;
        const int kt = slot_kt[slot];
        if (kt == 0) {
#pragma unroll
            for (int nt = 0; nt < NT; ++nt)
#pragma unroll
                for (int i = 0; i < 4; ++i) acc[nt][i] = accu[nt][i] = 0.f;
        }
        const __nv_bfloat16* st = stages + (size_t)slot * Cfg::kStage;
        const __nv_bfloat16* w0p = st + wb * Cfg::kBoxW + g * 256 + wc + 8 * t4;
        const __nv_bfloat16* ap = st + Cfg::kWBlocks * Cfg::kNB * Cfg::kBoxW + wb * Cfg::kBoxA + g * 256 + wc + 8 * t4;
#pragma unroll
        for (int ks = 0; ks < Cfg::kWarpCols / 32; ++ks) {
            const uint4 w0 = lds128(w0p + 32 * ks);
            const uint4 w1 = lds128(w0p + 8 * 256 + 32 * ks);
            uint4 u0 = z, u1 = z;
            if (PAIR) {
                u0 = lds128(w0p + Cfg::kNB * Cfg::kBoxW + 32 * ks);
                u1 = lds128(w0p + Cfg::kNB * Cfg::kBoxW + 8 * 256 + 32 * ks);
            }
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) {
                const uint4 bv = (nt * 8 + g < a.R) ? lds128(ap + nt * 8 * 256 + 32 * ks) : z;
                mma_bf16(acc[nt], w0.x, w1.x, w0.y, w1.y, bv.x, bv.y);
                mma_bf16(acc[nt], w0.z, w1.z, w0.w, w1.w, bv.z, bv.w);
                if (PAIR) {
                    mma_bf16(accu[nt], u0.x, u1.x, u0.y, u1.y, bv.x, bv.y);
                    mma_bf16(accu[nt], u0.z, u1.z, u0.w, u1.w, bv.z, bv.w);
                }
            }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&empty[slot]);  // this warp is done with the stage
        if (kt != TPI - 1) continue;

        // ------------------------------------------------ item epilogue
        // warps 1-3 hand their K-quarter partials to warp 0, which adds them
        // in warp order; the fragment of lane (g, t) covers features
        // 16 it + g (+ 8) and rows nt * 8 + 2 t (+ 1).
        if (warp > 0) {
#pragma unroll
            for (int nt = 0; nt < NT; ++nt)
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    red[warp - 1][0][nt * 4 + i][lane] = acc[nt][i];
                    if (PAIR) red[warp - 1][1][nt * 4 + i][lane] = accu[nt][i];
                }
        }
        out_sync<true>();
        if (warp == 0) {
#pragma unroll
            for (int w = 0; w < 3; ++w)
#pragma unroll
                for (int nt = 0; nt < NT; ++nt)
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        acc[nt][i] += red[w][0][nt * 4 + i][lane];
                        if (PAIR) accu[nt][i] += red[w][1][nt * 4 + i][lane];
                    }
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
#pragma unroll
            for (int nt = 0; nt < NT; ++nt)
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int n = it * 16 + g + 8 * (i >> 1);
                    const int r = nt * 8 + 2 * t4 + (i & 1);
                    if (n < a.N && r < a.R) {
                        const float sc = scale[r];
                        const float v = acc[nt][i] * sc;
                        if (EPI == EPI_LMHEAD) {
                            a.logits[(size_t)r * a.logits_ld + n] = v;
                            if (better(v, n, bv[nt][i & 1], bi[nt][i & 1])) {
                                bv[nt][i & 1] = v;
                                bi[nt][i & 1] = n;
                            }
                        } else if (EPI == EPI_RESID) {
                            float* x = a.resid + (size_t)r * a.resid_ld + n;
                            const float nx = *x + v;
                            *x = nx;
                            if (a.capture) a.capture[(size_t)r * a.capture_ld + n] = nx;
                            a.xg_out[(size_t)r * a.resid_ld + n] = __float2bfloat16_rn(
                                nx * to_float(reinterpret_cast<const __nv_bfloat16*>(a.next_gain)[n]));
                            ssq[nt][i & 1] = fmaf(nx, nx, ssq[nt][i & 1]);
                        } else {
                            apply_epilogue<__nv_bfloat16, EPI>(a, n, r, v, accu[nt][i] * sc);
                        }
                    }
                }
            if (EPI == EPI_RESID || EPI == EPI_LMHEAD) {
                // reduce over the 8 lanes with the same t (features g, g + 8)
#pragma unroll
                for (int nt = 0; nt < NT; ++nt)
#pragma unroll
                    for (int c = 0; c < 2; ++c) {
                        const int r = nt * 8 + 2 * t4 + c;
#pragma unroll
                        for (int o = 4; o < 32; o <<= 1) {
                            if (EPI == EPI_RESID) {
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
                        if (g == 0 && r < a.R) {
                            if (EPI == EPI_RESID) {
                                a.ss_out[it * kMaxRows + r] = ssq[nt][c];
                            } else {
                                a.amax_val[it * kMaxRows + r] = bv[nt][c];
                                a.amax_idx[it * kMaxRows + r] = bi[nt][c];
                            }
                        }
                    }
            }
        }
        out_sync<true>();  // red[] may be reused
    }
    if (failed) {
        if (tid == 0) atomicExch(a.err, 1);
        return;  // leave the queue alone; the host sees the status word
    }
    // the last CTA to finish resets the queue (every producer has stopped claiming)
    out_sync<true>();
    if (tid == 0) {
        __threadfence();
        is_last = (atomicAdd(&a.counters[1], 1) == (int)gridDim.x - 1);
    }
    out_sync<true>();
    if (!is_last) return;
    __threadfence();
    if (EPI == EPI_LMHEAD) final_argmax(a, n_items);
    if (tid == 0) {
        a.counters[0] = 0;
        a.counters[1] = 0;
    }
}

// ---------------------------------------------------------------- launcher
bool make_tma_map(CUtensorMap* map, const void* base, uint64_t rows, uint64_t K, uint32_t box_rows) {
    static PFN_cuTensorMapEncodeTiled_v12000 encode = nullptr;
    if (encode == nullptr) {
        void* fn = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) !=
                cudaSuccess ||
            q != cudaDriverEntryPointSuccess || fn == nullptr)
            return false;
        encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    }
    if (K % 8 != 0 || (reinterpret_cast<uintptr_t>(base) & 15) != 0) return false;
    const cuuint64_t dims[2] = {K, rows};
    const cuuint64_t strides[1] = {K * 2};
    const cuuint32_t box[2] = {256, box_rows};
    const cuuint32_t estr[2] = {1, 1};
    return encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}


template <int EPI>
static cudaError_t launch_stream(const GemvArgs& a, cudaStream_t s) {
    if (a.err == nullptr || a.R > kMaxRows || a.K % 8 != 0) return cudaErrorInvalidValue;
    auto run = [&](auto kern, size_t smem) -> cudaError_t {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(sm_count());
        cfg.blockDim = dim3(160);
        cfg.dynamicSmemBytes = smem;
        cfg.stream = s;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        return cudaLaunchKernelEx(&cfg, kern, a);
    };
    constexpr bool PAIR = EPI == EPI_SWIGLU;
    if (a.R <= 8) return run(gemv_stream_kernel<1, EPI>, stream_smem<1, PAIR>());
    return run(gemv_stream_kernel<2, EPI>, stream_smem<2, PAIR>());
}

template <int EPI>
static cudaError_t launch_f32(const GemvArgs& a, cudaStream_t s) {
    const int pitch = a.kc + 4;
    const size_t smem = sizeof(float) * ((size_t)a.R * pitch + kGemvWarps * 2 * 16 * 16);
    dim3 grid(gemv_grid_x(a.N), a.ksplit);
    auto run = [&](auto kern) -> cudaError_t {
        if (smem > 48 * 1024) {
            cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
            if (e != cudaSuccess) return e;
        }
        kern<<<grid, 128, smem, s>>>(a);
        return cudaGetLastError();
    };
    if (a.R <= 8) return run(gemv_f32_kernel<1, EPI>);
    return run(gemv_f32_kernel<2, EPI>);
}

cudaError_t launch_gemv(int dtype, int epi, const GemvArgs& a, cudaStream_t s) {
    if (a.R < 1 || a.R > kMaxRows || a.dtype != dtype) return cudaErrorInvalidValue;
    if (dtype == 1) {
        switch (epi) {
            case EPI_STORE: return launch_stream<EPI_STORE>(a, s);
            case EPI_RESID: return launch_stream<EPI_RESID>(a, s);
            case EPI_SWIGLU: return launch_stream<EPI_SWIGLU>(a, s);
            default: return launch_stream<EPI_LMHEAD>(a, s);
        }
    }
    switch (epi) {
        case EPI_STORE: return launch_f32<EPI_STORE>(a, s);
        case EPI_RESID: return launch_f32<EPI_RESID>(a, s);
        case EPI_SWIGLU: return launch_f32<EPI_SWIGLU>(a, s);
        default: return launch_f32<EPI_LMHEAD>(a, s);
    }
}

}  // namespace ks
