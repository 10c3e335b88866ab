// Causal GQA attention over the KV cache for R <= 16 query rows (the Attn
// sublayer of Sec. 2 inside a draft step or the gamma+1-row verify pass).
//
// Split-KV ("flash-decode") over a fixed partition of the key axis into
// chunks whose boundaries are absolute positions (attn_chunk_start): 128 keys
// below 8192, 512 keys below 32768, 2048 keys beyond.  One CTA per (KV head,
// chunk, round of query rows); the largest chunks are scheduled first.  Keys
// past a row's own position are masked to -inf (their exp2 is exactly 0) and
// chunks past it are skipped by the merge, so the arithmetic applied to one
// query row does not depend on how many rows share the pass: greedy decoding
// and the verify pass produce bit-identical attention outputs.
//
// bf16 models, three launches per Attn sublayer:
//  * attn_prep_kernel, once per pass: QK-RMSNorm and RoPE of the new rows'
//    queries (pre-scaled by log2(e)/sqrt(hd), bf16) and keys, and the K/V
//    cache write of the new rows;
//  * attn_bf16_kernel: keys sit on the M side of mma.sync.m16n8k16 and each
//    of the four warps streams its own 16-key K and V tiles (every fourth
//    tile of the chunk) through a private ring filled by TMA, with an fp32
//    online softmax in the log2 domain per query column and no block barrier
//    in the key loop; P reaches the P V product through registers
//    (movmatrix).  The warps' (m, l, o) are combined in warp order at the end
//    of the chunk;
//  * attn_merge_kernel: the chunk partials (m, l, o) per (row, query head)
//    merged in a fixed order.
// All three use programmatic dependent launch: the attention kernel loads its
// first tiles of old keys before waiting for the query prep, and the merge
// lets the next projections launch (and start streaming their weights) early.
// fp32 models: CUDA-core dot products, the new rows' K/V written by the CTA
// whose chunk holds them.
#include "common.cuh"
#include "internal.h"
#include "tma.cuh"

namespace ks {

constexpr int kAttnWarps = 4;
constexpr int kPartPad = 4;  // partial row: m, l, 2 pad, o[hd] (16-byte aligned o)

// bf16 K/V tiles in shared memory: rows of HD elements, no padding; the
// 16-byte chunk c of row r is stored at chunk c ^ (r & 7), so the eight rows
// an ldmatrix reads hit eight different bank groups.
template <int HD>
KS_DEV int kv_off(int row, int col) {
    return row * HD + ((((col >> 3) ^ (row & 7)) << 3) | (col & 7));
}
constexpr float kLog2e = 1.4426950408889634f;

// ------------------------------------------------------------ chunk schedule
__host__ __device__ int attn_chunk_start(int c) {
    if (c < 64) return 128 * c;
    if (c < 112) return 8192 + 512 * (c - 64);
    return 32768 + 2048 * (c - 112);
}
__host__ __device__ int attn_chunk_of(int pos) {
    if (pos < 8192) return pos / 128;
    if (pos < 32768) return 64 + (pos - 8192) / 512;
    return 112 + (pos - 32768) / 2048;
}
int attn_num_chunks(int n_keys) { return n_keys <= 0 ? 0 : attn_chunk_of(n_keys - 1) + 1; }

// ------------------------------------------------------------ small helpers
KS_DEV void cp_async16(void* smem, const void* gmem, bool valid) {
    const uint32_t s = (uint32_t)__cvta_generic_to_shared(smem);
    const int n = valid ? 16 : 0;
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(s), "l"(gmem), "r"(n));
}
KS_DEV void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::); }
template <int N>
KS_DEV void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N)); }

KS_DEV void ldmatrix_x4(uint32_t (&r)[4], const void* p) {
    const uint32_t s = (uint32_t)__cvta_generic_to_shared(p);
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(s));
}
KS_DEV void ldmatrix_x4_trans(uint32_t (&r)[4], const void* p) {
    const uint32_t s = (uint32_t)__cvta_generic_to_shared(p);
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];\n"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(s));
}

// Load one head vector (hd = 32 * NPL elements) of a row from the fp32
// projections, apply optional RMSNorm with gain, then rotate-half RoPE at
// position pos.  Lane l holds elements l + 32 i.
template <typename WT, int NPL>
KS_DEV void head_vector(const float* src, const WT* gain, float eps, const float* rope, int pos,
                        float (&v)[NPL]) {
    const int lane = threadIdx.x & 31;
    constexpr int hd = 32 * NPL;
#pragma unroll
    for (int i = 0; i < NPL; ++i) v[i] = src[lane + 32 * i];
    if (gain != nullptr) {
        float ss = 0.f;
#pragma unroll
        for (int i = 0; i < NPL; ++i) ss = fmaf(v[i], v[i], ss);
        ss = warp_sum(ss);
        const float inv = rsqrtf(ss / (float)hd + eps);
#pragma unroll
        for (int i = 0; i < NPL; ++i) v[i] = (v[i] * inv) * to_float(gain[lane + 32 * i]);
    }
    const float* rp = rope + (size_t)pos * hd;  // [hd/2][2]
#pragma unroll
    for (int i = 0; i < NPL / 2; ++i) {
        const int j = lane + 32 * i;
        const float c = rp[2 * j], s = rp[2 * j + 1];
        const float a = v[i], b = v[i + NPL / 2];
        v[i] = a * c - b * s;
        v[i + NPL / 2] = b * c + a * s;
    }
}

// Batched form of head_vector: a warp loads B vectors (and their RoPE rows) in
// one round of independent loads, then normalises and rotates them.  valid[j]
// = false skips vector j (its output is undefined).
template <typename WT, int NPL, int B>
KS_DEV void head_vectors(const float* const (&src)[B], const bool (&valid)[B], const int (&pos)[B],
                         const WT* gain, float eps, const float* rope, float (&v)[B][NPL]) {
    const int lane = threadIdx.x & 31;
    constexpr int hd = 32 * NPL;
    float cs[B][NPL / 2], sn[B][NPL / 2];
#pragma unroll
    for (int j = 0; j < B; ++j) {
        if (!valid[j]) continue;
#pragma unroll
        for (int i = 0; i < NPL; ++i) v[j][i] = src[j][lane + 32 * i];
        const float* rp = rope + (size_t)pos[j] * hd;
#pragma unroll
        for (int i = 0; i < NPL / 2; ++i) {
            cs[j][i] = rp[2 * (lane + 32 * i)];
            sn[j][i] = rp[2 * (lane + 32 * i) + 1];
        }
    }
#pragma unroll
    for (int j = 0; j < B; ++j) {
        float ss = 0.f;
        if (valid[j] && gain != nullptr) {
#pragma unroll
            for (int i = 0; i < NPL; ++i) ss = fmaf(v[j][i], v[j][i], ss);
        }
        if (gain != nullptr) ss = warp_sum(ss);  // every lane takes part (valid is warp-uniform)
        if (!valid[j]) continue;
        if (gain != nullptr) {
            const float inv = rsqrtf(ss / (float)hd + eps);
#pragma unroll
            for (int i = 0; i < NPL; ++i) v[j][i] = (v[j][i] * inv) * to_float(gain[lane + 32 * i]);
        }
#pragma unroll
        for (int i = 0; i < NPL / 2; ++i) {
            const float a = v[j][i], b = v[j][i + NPL / 2];
            v[j][i] = a * cs[j][i] - b * sn[j][i];
            v[j][i + NPL / 2] = b * cs[j][i] + a * sn[j][i];
        }
    }
}

// Write this chunk's new K/V rows (positions p0 .. p0+R-1 inside [cs, ce)).
template <typename WT, int NPL>
KS_DEV void write_new_kv(const AttnArgs& a, int h, int cs, int ce) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    constexpr int hd = 32 * NPL;
    constexpr int B = 4;
    WT* kc = reinterpret_cast<WT*>(a.kcache) + (size_t)h * a.max_seq * hd;
    WT* vc = reinterpret_cast<WT*>(a.vcache) + (size_t)h * a.max_seq * hd;
    const WT* kn = reinterpret_cast<const WT*>(a.k_norm);
    for (int r0 = warp * B; r0 < a.R; r0 += kAttnWarps * B) {
        const float* src[B];
        bool valid[B];
        int pos[B];
#pragma unroll
        for (int j = 0; j < B; ++j) {
            const int r = r0 + j;
            pos[j] = a.p0 + r;
            valid[j] = r < a.R && pos[j] >= cs && pos[j] < ce;
            src[j] = a.qkv + (size_t)(valid[j] ? r : 0) * a.qkv_ld + (a.hq + h) * hd;
            if (!valid[j]) pos[j] = 0;
        }
        float k[B][NPL];
        head_vectors<WT, NPL, B>(src, valid, pos, kn, a.eps, a.rope, k);
#pragma unroll
        for (int j = 0; j < B; ++j) {
            if (!valid[j]) continue;
            const float* vsrc = a.qkv + (size_t)(r0 + j) * a.qkv_ld + (a.hq + a.hk + h) * hd;
#pragma unroll
            for (int i = 0; i < NPL; ++i) {
                kc[(size_t)pos[j] * hd + lane + 32 * i] = from_float<WT>(k[j][i]);
                vc[(size_t)pos[j] * hd + lane + 32 * i] = from_float<WT>(vsrc[lane + 32 * i]);
            }
        }
    }
}

// chunk handled by this CTA: the largest (latest) chunks get the lowest blockIdx.y
KS_DEV int my_chunk(const AttnArgs& a) {
    const int nch = attn_chunk_of(a.p0 + a.R - 1) + 1;
    return nch - 1 - (int)blockIdx.y;
}

// ------------------------------------------------------- bf16 query prep
// One warp per head vector of one row, once per pass: a query head gets its
// QK-RMSNorm, RoPE at the row's position and the log2(e)/sqrt(hd) scale, and
// goes to q[kv head][m = r G + gq] in bf16; a key head gets its RMSNorm and
// RoPE and goes to the K cache at the row's position; a value head is copied
// to the V cache.  The attention CTAs then only stream the cache.
template <int HD>
__global__ void __launch_bounds__(128) attn_prep_kernel(const __grid_constant__ AttnArgs a) {
    if (a.stop && *a.stop) return;   // a draft pass after the dynamic exit
    // The attention kernel may launch now: before its own dependency wait it
    // only loads keys written by earlier passes.
    grid_launch_dependents();
    grid_dependency_wait();          // the projections of this pass
    constexpr int NPL = HD / 32;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int r = blockIdx.x, v = blockIdx.y * 4 + warp;
    const int G = a.hq / a.hk, M = G * a.R, pos = a.p0 + r;
    const float* row = a.qkv + (size_t)r * a.qkv_ld;
    float x[NPL];
    if (v < a.hq) {
        head_vector<__nv_bfloat16, NPL>(row + v * HD, reinterpret_cast<const __nv_bfloat16*>(a.q_norm), a.eps,
                                        a.rope, pos, x);
        const float qscale = kLog2e * rsqrtf((float)HD);
        const int h = v / G, m = r * G + (v - h * G);
        __nv_bfloat16* dst = a.q + ((size_t)h * M + m) * HD;
#pragma unroll
        for (int i = 0; i < NPL; ++i) dst[lane + 32 * i] = __float2bfloat16_rn(x[i] * qscale);
    } else if (v < a.hq + a.hk) {
        const int h = v - a.hq;
        head_vector<__nv_bfloat16, NPL>(row + (a.hq + h) * HD, reinterpret_cast<const __nv_bfloat16*>(a.k_norm),
                                        a.eps, a.rope, pos, x);
        __nv_bfloat16* kc = reinterpret_cast<__nv_bfloat16*>(a.kcache) + ((size_t)h * a.max_seq + pos) * HD;
        __nv_bfloat16* vc = reinterpret_cast<__nv_bfloat16*>(a.vcache) + ((size_t)h * a.max_seq + pos) * HD;
        const float* vs = row + (a.hq + a.hk + h) * HD;
#pragma unroll
        for (int i = 0; i < NPL; ++i) {
            kc[lane + 32 * i] = __float2bfloat16_rn(x[i]);
            vc[lane + 32 * i] = __float2bfloat16_rn(vs[lane + 32 * i]);
        }
    }
}

// ----------------------------------------------------------- bf16 kernel
// Keys on the M side of the MMA.  Warp w owns keys 16 w .. 16 w + 15 of every
// 64 keys of the chunk and runs its own online softmax over them, so the key
// loop needs no block barrier:
//   S^T (16 keys x 8 NQ query rows)  = K_w Q^T     A = K rows (ldmatrix),
//                                                   B = Q rows (ldmatrix)
//   O^T (HD dims x 8 NQ query rows) += V_w^T P^T   A = V (ldmatrix.trans),
//                                                   B = the S^T accumulator as
//                                                   bf16, transposed in
//                                                   registers (movmatrix)
// A warp's 16-key K and V tiles arrive by TMA (one 3-D box each: 16 rows of
// hd / 64 swizzled 64-column chunks) in its own ring of kWarpStages stages,
// each completing on the warp's mbarrier; lane 0 issues them.  At the end of
// the chunk the four warps' (m, l, O) meet in their ring space and are
// combined in warp order.  Query rows m = r G + gq come in rounds of 8 NQ
// rows; each round is its own CTA, and the rounds of one (KV head, chunk)
// are adjacent in the grid so that all but the first read the chunk from L2.
// Every step of a query row's arithmetic is fixed by the chunk and the key
// index alone, never by R or by the other rows of the pass.
constexpr int kWarpKeys = 16;
// Two stages per warp (one tile in flight while the other is computed) keep
// a CTA at about 71 KB of shared memory, so that with at most 168 registers
// per thread three CTAs (twelve warps) share an SM: the key loop is bound by
// the latency of its dependent steps, and more resident warps hide it.
constexpr int kWarpStages = 2;
constexpr int kAttnCtasPerSm = 3;

// 8x8 b16 matrix transpose across the warp: the fragment of X becomes the
// fragment of X^T
KS_DEV uint32_t movmatrix_trans(uint32_t x) {
    uint32_t y;
    asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;\n" : "=r"(y) : "r"(x));
    return y;
}

// Byte offset of (row, col) in a K or V tile as TMA stores it with the
// 128-byte swizzle: 64-column chunks of 16 rows x 128 bytes, 16-byte unit u
// of row r at unit u ^ (r & 7).  col is a multiple of 8.
KS_DEV uint32_t tile_off(int row, int col) {
    return ((uint32_t)(col >> 6) << 11) + ((uint32_t)row << 7) + ((uint32_t)(((col >> 3) & 7) ^ (row & 7)) << 4);
}
KS_DEV void fence_proxy_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }
// 2^x by the hardware approximation (ex2.approx.ftz: 2^-inf = +0); the same
// instruction for every query row, so results stay independent of R.
KS_DEV float fast_exp2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}


// One CTA's work: query rows q0 .. q0 + 8 NQ - 1 of KV head h over one chunk.
// `a` is the kernel's parameter (its tensor map is read in place by TMA).
template <int HD, int NQ>
__device__ __forceinline__ void attn_bf16_body(const AttnArgs& a, int h, int q0, unsigned char* smem_raw,
                                               uint64_t (*full)[kWarpStages]) {
    constexpr int P = HD + 8;          // Qs row pitch (bf16)
    constexpr int KD = HD / 16;        // k-steps of K Q^T = dim tiles of V^T P^T
    constexpr int QR = 8 * NQ;         // query rows per round
    constexpr int TB = kWarpKeys * HD * 2;           // bytes of one K (or V) tile
    constexpr int STAGE = 2 * TB;                    // K tile, then V tile
    constexpr int RING = kWarpStages * STAGE;        // one warp's ring
    constexpr int OP = HD + 4;         // pitch of a query row in the combine area (fp32)
    static_assert(QR * (OP + 2) * 4 <= RING, "combine area exceeds the warp's ring");
    // 1024-byte aligned: the swizzle pattern repeats every 1024 bytes
    unsigned char* rings = reinterpret_cast<unsigned char*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    __nv_bfloat16* Qs = reinterpret_cast<__nv_bfloat16*>(rings + kAttnWarps * RING);   // [QR][P]

    const int G = a.hq / a.hk;
    const int M = G * a.R;
    const int c = my_chunk(a);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int g = lane >> 2, t = lane & 3;
    const int cs = attn_chunk_start(c);
    const int ce = min(attn_chunk_start(c + 1), a.p0 + a.R);  // valid keys [cs, ce)
    const int nwt = (ce - cs + kWarpKeys - 1) / kWarpKeys;    // 16-key tiles of the chunk
    const int my_n = nwt > warp ? (nwt - warp + kAttnWarps - 1) / kAttnWarps : 0;  // tiles warp, warp + 4, ..
    unsigned char* ring = rings + warp * RING;
    uint64_t* bar = full[warp];

    if (lane == 0) {
        for (int i = 0; i < kWarpStages; ++i) mbar_init(&bar[i], 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncwarp();
    // this warp's i-th tile -> stage i % kWarpStages (lane 0 issues)
    auto issue = [&](int i) {
        const int st = i % kWarpStages;
        unsigned char* dst = ring + st * STAGE;
        const int row = h * a.max_seq + cs + (warp + kAttnWarps * i) * kWarpKeys;
        fence_proxy_async_smem();   // the warp's reads of the stage come before the copy's writes
        mbar_expect_tx(&bar[st], STAGE);
        tma_3d(dst, &a.kvmap, 0, a.kv_row_k + row, 0, &bar[st]);
        tma_3d(dst + TB, &a.kvmap, 0, a.kv_row_v + row, 0, &bar[st]);
    };
    auto tile_old = [&](int i) { return cs + (warp + kAttnWarps * i + 1) * kWarpKeys <= a.p0; };
    // Keys before p0 were written by earlier passes, so this warp's first
    // tiles of old keys go out before waiting for the query prep.
    const int pre = min(kWarpStages - 1, my_n);
    int issued = 0;
    if (lane == 0)
        while (issued < pre && tile_old(issued)) issue(issued++);
    grid_dependency_wait();          // queries and new K/V rows of this pass
    grid_launch_dependents();        // the merge may launch; it waits for this grid
    if (lane == 0)
        while (issued < pre) issue(issued++);

    // queries of this round, rows m = q0 + row (rows past M are zero)
    constexpr int CPR = HD / 8;      // 16-byte pieces per row
    for (int j = tid; j < QR * CPR; j += blockDim.x) {
        const int row = j / CPR, col = (j - row * CPR) * 8;
        const bool ok = q0 + row < M;
        cp_async16(Qs + row * P + col, a.q + ((size_t)h * M + (ok ? q0 + row : 0)) * HD + col, ok);
    }
    cp_async_commit();
    cp_async_wait<0>();
    __syncthreads();                 // Qs complete
    // Q^T fragments (B operand): query tile j = rows 8 j .., k-step ks;
    // held in registers for up to two query tiles, else read from Qs
    constexpr bool kQReg = NQ <= 2;
    uint32_t qf[kQReg ? NQ : 1][KD][2];
#pragma unroll
    for (int j = 0; j < (kQReg ? NQ : 0); ++j)
#pragma unroll
        for (int ks = 0; ks < KD; ks += 2) {
            uint32_t r4[4];
            ldmatrix_x4(r4, Qs + (8 * j + (lane & 7)) * P + ks * 16 + (lane >> 3) * 8);
            qf[j][ks][0] = r4[0];
            qf[j][ks][1] = r4[1];
            qf[j][ks + 1][0] = r4[2];
            qf[j][ks + 1][1] = r4[3];
        }
    // this thread's query columns: 8 j + 2 t + e; padding rows see no key
    int qpos[NQ][2];
#pragma unroll
    for (int j = 0; j < NQ; ++j)
#pragma unroll
        for (int e = 0; e < 2; ++e) {
            const int m = q0 + 8 * j + 2 * t + e;
            qpos[j][e] = m < M ? a.p0 + m / G : -1;
        }
    float o[KD][NQ][4];          // O^T: dims 16 d + g (+ 8), query columns 8 j + 2 t (+ 1)
    float mcol[NQ][2], lsum[NQ][2];
#pragma unroll
    for (int j = 0; j < NQ; ++j) {
#pragma unroll
        for (int d = 0; d < KD; ++d) o[d][j][0] = o[d][j][1] = o[d][j][2] = o[d][j][3] = 0.f;
        mcol[j][0] = mcol[j][1] = -INFINITY;
        lsum[j][0] = lsum[j][1] = 0.f;   // this thread's keys g, g + 8 only
    }

    bool ok = true;
    int waited = 0;                   // tiles whose copies this warp has seen complete
    for (int i = 0; i < my_n; ++i) {
        // tile i + kWarpStages - 1 goes into the stage tile i - 1 used
        if (lane == 0 && i + kWarpStages - 1 < my_n) issue(i + kWarpStages - 1);
        const int st = i % kWarpStages;
        const bool got = mbar_wait(&bar[st], (uint32_t)((i / kWarpStages) & 1), kWaitLimitNs);
        if (!__all_sync(0xffffffffu, got)) {   // warp-uniform: the loop below shuffles
            ok = false;
            break;
        }
        waited = i + 1;
        const unsigned char* Ks = ring + st * STAGE;
        const unsigned char* Vs = Ks + TB;
        const int k0 = cs + (warp + kAttnWarps * i) * kWarpKeys;
        // (a) S^T = K Q^T for this warp's 16 keys
        float s[NQ][4];
#pragma unroll
        for (int j = 0; j < NQ; ++j) s[j][0] = s[j][1] = s[j][2] = s[j][3] = 0.f;
#pragma unroll
        for (int ks = 0; ks < KD; ks += 2) {
            uint32_t ka[2][4];
#pragma unroll
            for (int u = 0; u < 2; ++u)
                ldmatrix_x4(ka[u], Ks + tile_off((lane & 7) + ((lane >> 3) & 1) * 8, (ks + u) * 16 + (lane >> 4) * 8));
#pragma unroll
            for (int j = 0; j < NQ; ++j) {
                uint32_t b[4];
                if constexpr (kQReg) {
                    b[0] = qf[j][ks][0];
                    b[1] = qf[j][ks][1];
                    b[2] = qf[j][ks + 1][0];
                    b[3] = qf[j][ks + 1][1];
                } else {
                    ldmatrix_x4(b, Qs + (8 * j + (lane & 7)) * P + ks * 16 + (lane >> 3) * 8);
                }
                mma_bf16(s[j], ka[0][0], ka[0][1], ka[0][2], ka[0][3], b[0], b[1]);
                mma_bf16(s[j], ka[1][0], ka[1][1], ka[1][2], ka[1][3], b[2], b[3]);
            }
        }
        // (b) mask, online softmax per query column over this warp's keys.
        // Only a tile reaching position p0 has keys that some row may not see
        // (every row sits at p0 or later; keys at or past ce are past every row).
        const bool masked = k0 + kWarpKeys > a.p0;
        const int key0 = k0 + g, key1 = k0 + g + 8;
        uint32_t pb[NQ][2];
        float alpha[NQ][2];
        bool grew = false;   // some column's running maximum changed
#pragma unroll
        for (int j = 0; j < NQ; ++j) {
#pragma unroll
            for (int e = 0; e < 2; ++e) {
                float& va = s[j][e];
                float& vb = s[j][2 + e];
                if (masked) {
                    if (key0 > qpos[j][e] || key0 >= ce) va = -INFINITY;
                    if (key1 > qpos[j][e] || key1 >= ce) vb = -INFINITY;
                }
                float tmax = fmaxf(va, vb);
                tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, 4));
                tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, 8));
                tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, 16));
                const float mnew = fmaxf(mcol[j][e], tmax);
                float al = 1.f;
                if (mnew == -INFINITY) {   // no key of this column seen yet
                    va = vb = 0.f;
                } else {
                    al = fast_exp2(mcol[j][e] - mnew);
                    va = fast_exp2(va - mnew);
                    vb = fast_exp2(vb - mnew);
                }
                grew |= mnew != mcol[j][e];
                mcol[j][e] = mnew;
                lsum[j][e] = lsum[j][e] * al + (va + vb);
                alpha[j][e] = al;
            }
            // P^T (keys x queries) as the B operand: transposed S^T fragments
            pb[j][0] = movmatrix_trans(pack_bf16(s[j][0], s[j][1]));
            pb[j][1] = movmatrix_trans(pack_bf16(s[j][2], s[j][3]));
        }
        // rescale O only when a maximum moved: otherwise every alpha is
        // exactly 1 and the products would not change a bit
        if (__any_sync(0xffffffffu, grew)) {
#pragma unroll
            for (int j = 0; j < NQ; ++j)
#pragma unroll
                for (int e = 0; e < 2; ++e)
#pragma unroll
                    for (int d = 0; d < KD; ++d) {
                        o[d][j][e] *= alpha[j][e];
                        o[d][j][2 + e] *= alpha[j][e];
                    }
        }
        // (c) O^T += V^T P^T over this warp's 16 keys
#pragma unroll
        for (int d = 0; d < KD; ++d) {
            uint32_t va[4];
            const int mi = lane >> 3;
            ldmatrix_x4_trans(va, Vs + tile_off((lane & 7) + (mi >> 1) * 8, d * 16 + (mi & 1) * 8));
#pragma unroll
            for (int j = 0; j < NQ; ++j) mma_bf16(o[d][j], va[0], va[1], va[2], va[3], pb[j][0], pb[j][1]);
        }
        __syncwarp();   // every lane is done with the stage before it is refilled
    }
    if (!ok) {
        // a copy did not arrive in time: record it, and account for the
        // copies still in flight (bounded) before the ring space is reused
        if (lane == 0) atomicCAS(a.err, 0, 1);
        const int last = min(my_n, waited + kWarpStages);
        for (int i = waited; i < last; ++i)
            mbar_wait(&bar[i % kWarpStages], (uint32_t)((i / kWarpStages) & 1), kWaitLimitNs);
    }
    // (d) this warp's column sums, then (m, l, O^T) into its ring space
#pragma unroll
    for (int j = 0; j < NQ; ++j)
#pragma unroll
        for (int e = 0; e < 2; ++e) {
            float l = lsum[j][e];
            l += __shfl_xor_sync(0xffffffffu, l, 4);
            l += __shfl_xor_sync(0xffffffffu, l, 8);
            l += __shfl_xor_sync(0xffffffffu, l, 16);
            lsum[j][e] = l;
        }
    __syncthreads();                  // every warp is done with Qs and its ring
    float* cm = reinterpret_cast<float*>(ring);   // [QR] m, [QR] l, [QR][OP] o
    float* cl = cm + QR;
    float* co = cl + QR;
#pragma unroll
    for (int j = 0; j < NQ; ++j)
#pragma unroll
        for (int e = 0; e < 2; ++e) {
            const int q = 8 * j + 2 * t + e;
            if (g == 0) {
                cm[q] = mcol[j][e];
                cl[q] = lsum[j][e];
            }
#pragma unroll
            for (int d = 0; d < KD; ++d) {
                co[q * OP + 16 * d + g] = o[d][j][e];
                co[q * OP + 16 * d + g + 8] = o[d][j][2 + e];
            }
        }
    __syncthreads();
    // (e) the four warps combined in warp order -> this chunk's partials:
    //     per query row the chunk maximum, each warp's scale factor and the
    //     sum l (one thread per row), then O element by element
    const int nq = min(QR, M - q0);
    constexpr int WF = RING / 4;                                  // floats per warp's ring
    const float* wsum = reinterpret_cast<const float*>(rings);    // warp w at w * WF floats
    float* fac = reinterpret_cast<float*>(Qs);                    // [kAttnWarps][QR]
    if (tid < nq) {
        const int q = tid;
        float gm = -INFINITY;
#pragma unroll
        for (int w = 0; w < kAttnWarps; ++w) gm = fmaxf(gm, wsum[w * WF + q]);
        float L = 0.f;
#pragma unroll
        for (int w = 0; w < kAttnWarps; ++w) {
            const float f = gm == -INFINITY ? 0.f : exp2f(wsum[w * WF + q] - gm);   // 0: a warp that saw no key
            fac[w * QR + q] = f;
            L += wsum[w * WF + QR + q] * f;
        }
        const int m = q0 + q, r = m / G, gq = m - r * G;
        float* dst = a.part + (((size_t)r * a.hq + h * G + gq) * a.n_chunks_max + c) * (HD + kPartPad);
        dst[0] = gm;
        dst[1] = L;
    }
    __syncthreads();
    constexpr int HV = HD / 4;   // float4 pieces of a row
    for (int idx = tid; idx < nq * HV; idx += blockDim.x) {
        const int q = idx / HV, d4 = (idx - q * HV) * 4;
        float4 O = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int w = 0; w < kAttnWarps; ++w) {
            const float4 v = *reinterpret_cast<const float4*>(wsum + w * WF + 2 * QR + q * OP + d4);
            const float f = fac[w * QR + q];
            O.x += v.x * f;
            O.y += v.y * f;
            O.z += v.z * f;
            O.w += v.w * f;
        }
        const int m = q0 + q, r = m / G, gq = m - r * G;
        *reinterpret_cast<float4*>(a.part + (((size_t)r * a.hq + h * G + gq) * a.n_chunks_max + c) * (HD + kPartPad) +
                                   kPartPad + d4) = O;
    }
}

// Query rows m = r G + gq in rounds of 8 NQ rows, one round per CTA (the
// rounds of a KV head adjacent in x).  A last round with at most 8 (NQ - 1)
// rows (the second round of 40 rows at eight query heads per KV head) runs
// with one query tile less; a row's arithmetic is the same in either.
template <int HD, int NQ>
__global__ void __launch_bounds__(128, kAttnCtasPerSm) attn_bf16_kernel(const __grid_constant__ AttnArgs a) {
    if (a.stop && *a.stop) return;   // a draft pass after the dynamic exit
    extern __shared__ unsigned char smem_raw[];
    __shared__ __align__(8) uint64_t full[kAttnWarps][kWarpStages];
    constexpr int QR = 8 * NQ;
    const int M = (a.hq / a.hk) * a.R;
    const int rounds = (M + QR - 1) / QR;
    const int h = (int)blockIdx.x / rounds, q0 = ((int)blockIdx.x - h * rounds) * QR;
    if constexpr (NQ > 1) {
        if (M - q0 <= 8 * (NQ - 1)) {
            attn_bf16_body<HD, NQ - 1>(a, h, q0, smem_raw, full);
            return;
        }
    }
    attn_bf16_body<HD, NQ>(a, h, q0, smem_raw, full);
}

// ----------------------------------------------------------- fp32 kernel
// One warp per query row at a time; K/V read from the cache (L2).  Used for
// fp32 models.
template <int HD>
__global__ void __launch_bounds__(128) attn_f32_kernel(const AttnArgs a) {
    if (a.stop && *a.stop) return;   // a draft pass after the dynamic exit
    constexpr int NPL = HD / 32;
    constexpr int C = 2048;  // largest chunk of the schedule
    extern __shared__ float fsm[];
    float* qsh = fsm;                    // [4][HD]
    float* psh = fsm + kAttnWarps * HD;  // [4][C]
    const int h = blockIdx.x, c = my_chunk(a);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int G = a.hq / a.hk;
    const int M = G * a.R;
    const int cs = attn_chunk_start(c);
    const int ce = min(attn_chunk_start(c + 1), a.p0 + a.R);

    write_new_kv<float, NPL>(a, h, cs, ce);
    __syncthreads();

    const float* kc = reinterpret_cast<const float*>(a.kcache) + (size_t)h * a.max_seq * HD;
    const float* vc = reinterpret_cast<const float*>(a.vcache) + (size_t)h * a.max_seq * HD;
    const float qscale = kLog2e * rsqrtf((float)HD);
    const float* qn = reinterpret_cast<const float*>(a.q_norm);
    float* q_w = qsh + warp * HD;
    float* p_w = psh + warp * C;
    for (int m = warp; m < M; m += kAttnWarps) {
        const int r = m / G, gq = m - r * G;
        const int pos = a.p0 + r;
        float q[NPL];
        head_vector<float, NPL>(a.qkv + (size_t)r * a.qkv_ld + (h * G + gq) * HD, qn, a.eps, a.rope, pos, q);
#pragma unroll
        for (int i = 0; i < NPL; ++i) q_w[lane + 32 * i] = q[i] * qscale;
        __syncwarp();
        const int kend = min(ce, pos + 1);
        float mx = -INFINITY;
        for (int j = lane; j < ce - cs; j += 32) {
            const int key = cs + j;
            float sc = -INFINITY;
            if (key < kend) {
                sc = 0.f;
                const float* kr = kc + (size_t)key * HD;
                for (int d = 0; d < HD; ++d) sc = fmaf(q_w[d], kr[d], sc);
            }
            p_w[j] = sc;
            mx = fmaxf(mx, sc);
        }
        mx = warp_max(mx);
        float l = 0.f;
        for (int j = lane; j < ce - cs; j += 32) {
            const float p = (mx == -INFINITY || p_w[j] == -INFINITY) ? 0.f : exp2f(p_w[j] - mx);
            p_w[j] = p;
            l += p;
        }
        l = warp_sum(l);
        __syncwarp();
        float* dst = a.part + (((size_t)r * a.hq + h * G + gq) * a.n_chunks_max + c) * (HD + kPartPad);
        for (int d = lane; d < HD; d += 32) {
            float acc = 0.f;
            for (int j = 0; j < kend - cs; ++j) acc = fmaf(p_w[j], vc[(size_t)(cs + j) * HD + d], acc);
            dst[kPartPad + d] = acc;
        }
        if (lane == 0) {
            dst[0] = mx;
            dst[1] = l;
        }
        __syncwarp();
    }
}

// ------------------------------------------------------------------ merge
// out[r][hq_idx * hd + d] = sum_c 2^(m_c - M) o_c[d] / sum_c 2^(m_c - M) l_c over
// the chunks 0 .. chunk_of(pos_r) of row r.  Fixed order for every term: the
// max is exact in any order; l is summed per thread (chunks c = t mod 256)
// and then in thread order, o per warp (chunks c = w mod 8) and then in warp
// order.  The chunk count depends only on the row's position, so a row gives
// the same bits in a 1-row pass and in a gamma+1-row pass.
constexpr int kMergeWarps = 8;
template <typename WT, int HD>
__global__ void __launch_bounds__(kMergeWarps * 32) attn_merge_kernel(const AttnArgs a) {
    if (a.stop && *a.stop) return;   // a draft pass after the dynamic exit
    extern __shared__ float wsh[];  // [nch] chunk weights
    __shared__ float red[kMergeWarps + 1];
    __shared__ float osh[kMergeWarps][HD];
    constexpr int NT = kMergeWarps * 32;
    const int hq_idx = blockIdx.x, r = blockIdx.y;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");   // the next projections may launch
    asm volatile("griddepcontrol.wait;" ::: "memory");                // the partials are complete
    const int pos = a.p0 + r;
    const int nch = attn_chunk_of(pos) + 1;
    constexpr int S = HD + kPartPad;
    const float* base = a.part + ((size_t)r * a.hq + hq_idx) * a.n_chunks_max * S;
    constexpr int PER = HD / 32;   // dims per lane
    constexpr int PF = 8;          // this warp's first chunks: o loaded while the maxima are reduced
    float pre[PF][PER];
#pragma unroll
    for (int k = 0; k < PF; ++k) {
        const int c = warp + kMergeWarps * k;
        const float* src = base + (size_t)c * S + kPartPad + PER * lane;
        if (c < nch) {
            if constexpr (PER == 4) {
                const float4 v = *reinterpret_cast<const float4*>(src);
                pre[k][0] = v.x;
                pre[k][1] = v.y;
                pre[k][2] = v.z;
                pre[k][3] = v.w;
            } else {
#pragma unroll
                for (int i = 0; i < PER; ++i) pre[k][i] = src[i];
            }
        }
    }
    // (m, l) of this thread's chunks c = tid, tid + NT, ... (one round below 256 chunks)
    constexpr int MC = 2;
    float mc[MC], lc[MC];
#pragma unroll
    for (int k = 0; k < MC; ++k) {
        const int c = tid + NT * k;
        mc[k] = c < nch ? base[(size_t)c * S] : -INFINITY;
        lc[k] = c < nch ? base[(size_t)c * S + 1] : 0.f;
    }
    float mx = -INFINITY;
#pragma unroll
    for (int k = 0; k < MC; ++k) mx = fmaxf(mx, mc[k]);
    for (int c = tid + NT * MC; c < nch; c += NT) mx = fmaxf(mx, base[(size_t)c * S]);
    mx = warp_max(mx);
    if (lane == 0) red[warp] = mx;
    __syncthreads();
    mx = red[0];
#pragma unroll
    for (int w = 1; w < kMergeWarps; ++w) mx = fmaxf(mx, red[w]);
    float ls = 0.f;
#pragma unroll
    for (int k = 0; k < MC; ++k) {
        const int c = tid + NT * k;
        if (c < nch) {
            const float w = (mc[k] == -INFINITY) ? 0.f : exp2f(mc[k] - mx);
            wsh[c] = w;
            ls = fmaf(w, lc[k], ls);
        }
    }
    for (int c = tid + NT * MC; c < nch; c += NT) {
        const float m = base[(size_t)c * S];
        const float w = (m == -INFINITY) ? 0.f : exp2f(m - mx);
        wsh[c] = w;
        ls = fmaf(w, base[(size_t)c * S + 1], ls);
    }
    const float L = block_sum<kMergeWarps>(ls, red);  // ends with a barrier: wsh is visible
    float o[PER];
#pragma unroll
    for (int i = 0; i < PER; ++i) o[i] = 0.f;
#pragma unroll
    for (int k = 0; k < PF; ++k) {
        const int c = warp + kMergeWarps * k;
        if (c < nch) {
            const float w = wsh[c];
#pragma unroll
            for (int i = 0; i < PER; ++i) o[i] = fmaf(w, pre[k][i], o[i]);
        }
    }
#pragma unroll 8
    for (int c = warp + kMergeWarps * PF; c < nch; c += kMergeWarps) {   // unrolled: several loads in flight
        const float w = wsh[c];
        const float* src = base + (size_t)c * S + kPartPad + PER * lane;
        if constexpr (PER == 4) {
            const float4 v = *reinterpret_cast<const float4*>(src);
            o[0] = fmaf(w, v.x, o[0]);
            o[1] = fmaf(w, v.y, o[1]);
            o[2] = fmaf(w, v.z, o[2]);
            o[3] = fmaf(w, v.w, o[3]);
        } else {
#pragma unroll
            for (int i = 0; i < PER; ++i) o[i] = fmaf(w, src[i], o[i]);
        }
    }
#pragma unroll
    for (int i = 0; i < PER; ++i) osh[warp][PER * lane + i] = o[i];
    __syncthreads();
    WT* out = reinterpret_cast<WT*>(a.out);
    for (int d = tid; d < HD; d += blockDim.x) {
        float O = osh[0][d];
#pragma unroll
        for (int w = 1; w < kMergeWarps; ++w) O += osh[w][d];
        out[(size_t)r * a.out_ld + hq_idx * HD + d] = from_float<WT>(O / L);
    }
}

// --------------------------------------------------------------- launchers
static size_t attn_bf16_smem(int HD, int NQ) {
    const size_t ring = (size_t)kWarpStages * 2 * kWarpKeys * HD * 2;
    return 1024 + kAttnWarps * ring + sizeof(__nv_bfloat16) * (size_t)8 * NQ * (HD + 8);
}

static cudaLaunchAttribute pdl_attr() {
    cudaLaunchAttribute at;
    at.id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at.val.programmaticStreamSerializationAllowed = 1;
    return at;
}

cudaError_t launch_attn_prep(const AttnArgs& a, cudaStream_t s) {
    if (a.q == nullptr || a.R < 1 || a.p0 + a.R > a.max_seq) return cudaErrorInvalidValue;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(a.R, (a.hq + a.hk + 3) / 4);
    cfg.blockDim = dim3(128);
    cfg.stream = s;
    cudaLaunchAttribute attr[1] = {pdl_attr()};
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (a.hd == 128) return cudaLaunchKernelEx(&cfg, attn_prep_kernel<128>, a);
    if (a.hd == 64) return cudaLaunchKernelEx(&cfg, attn_prep_kernel<64>, a);
    return cudaErrorInvalidValue;
}

cudaError_t launch_attention(int dtype, const AttnArgs& a, cudaStream_t s) {
    const int nch = attn_num_chunks(a.p0 + a.R);
    if (nch > a.n_chunks_max || a.p0 + a.R > a.max_seq) return cudaErrorInvalidValue;
    dim3 grid(a.hk, nch);
    if (dtype == 1) {
        if (a.q == nullptr || a.err == nullptr) return cudaErrorInvalidValue;
        // query rows per round: 8 NQ (24 at most); each round is its own CTA,
        // the rounds of one KV head adjacent in x
        const int M = (a.hq / a.hk) * a.R;
        const int NQ = M <= 8 ? 1 : M <= 16 ? 2 : 3;
        const int rounds = (M + 8 * NQ - 1) / (8 * NQ);
        const size_t smem = attn_bf16_smem(a.hd, NQ);
        auto run = [&](auto kern) -> cudaError_t {
            cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
            if (e != cudaSuccess) return e;
            cudaLaunchConfig_t cfg = {};
            cfg.gridDim = dim3(a.hk * rounds, nch);
            cfg.blockDim = dim3(128);
            cfg.dynamicSmemBytes = smem;
            cfg.stream = s;
            cudaLaunchAttribute attr[1] = {pdl_attr()};
            cfg.attrs = attr;
            cfg.numAttrs = 1;
            return cudaLaunchKernelEx(&cfg, kern, a);
        };
        if (a.hd == 128) return NQ == 1 ? run(attn_bf16_kernel<128, 1>)
                              : NQ == 2 ? run(attn_bf16_kernel<128, 2>) : run(attn_bf16_kernel<128, 3>);
        if (a.hd == 64) return NQ == 1 ? run(attn_bf16_kernel<64, 1>)
                             : NQ == 2 ? run(attn_bf16_kernel<64, 2>) : run(attn_bf16_kernel<64, 3>);
        return cudaErrorInvalidValue;
    }
    const size_t smem = sizeof(float) * kAttnWarps * ((size_t)a.hd + 2048);
    auto run = [&](auto kern) -> cudaError_t {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        kern<<<grid, 128, smem, s>>>(a);
        return cudaGetLastError();
    };
    if (a.hd == 128) return run(attn_f32_kernel<128>);
    if (a.hd == 64) return run(attn_f32_kernel<64>);
    return cudaErrorInvalidValue;
}

cudaError_t launch_attn_merge(int dtype, const AttnArgs& a, cudaStream_t s) {
    dim3 grid(a.hq, a.R);
    const int nch = attn_num_chunks(a.p0 + a.R);
    const size_t smem = sizeof(float) * (size_t)nch;
    if (nch > a.n_chunks_max || smem > 48 * 1024) return cudaErrorInvalidValue;
    if (dtype == 1) {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = grid;
        cfg.blockDim = dim3(kMergeWarps * 32);
        cfg.dynamicSmemBytes = smem;
        cfg.stream = s;
        cudaLaunchAttribute attr[1] = {pdl_attr()};
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        if (a.hd == 128) return cudaLaunchKernelEx(&cfg, attn_merge_kernel<__nv_bfloat16, 128>, a);
        return cudaLaunchKernelEx(&cfg, attn_merge_kernel<__nv_bfloat16, 64>, a);
    } else {
        if (a.hd == 128) attn_merge_kernel<float, 128><<<grid, kMergeWarps * 32, smem, s>>>(a);
        else attn_merge_kernel<float, 64><<<grid, kMergeWarps * 32, smem, s>>>(a);
    }
    return cudaGetLastError();
}

}  // namespace ks
