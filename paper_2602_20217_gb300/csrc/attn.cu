// Causal GQA attention over the KV cache for R <= 16 query rows (the Attn
// sublayer of Sec. 2 inside a draft step or the gamma+1-row verify pass).
//
// Split-KV ("flash-decode") over a fixed partition of the key axis into
// chunks whose boundaries are absolute positions (attn_chunk_start): 128 keys
// below 8192, 512 keys below 32768, 2048 keys beyond.  One CTA per (KV head,
// chunk); the largest chunks are scheduled first.  Keys past a row's own
// position are masked to -inf (their exp2 is exactly 0) and chunks past it are
// skipped by the merge, so the arithmetic applied to one query row does not
// depend on how many rows share the pass: greedy decoding and the verify pass
// produce bit-identical attention outputs.
//
// Per CTA: the new rows' K (QK-RMSNorm, RoPE) and V are written to the cache
// by the CTA whose chunk holds their position; the G x R query vectors are
// normalised, rotated and pre-scaled by log2(e)/sqrt(hd).  bf16 models: K/V
// tiles of 64 keys stream through a cp.async ring; for up to two 16-row query
// tiles at a time the four warps split each tile (warp w: Q K^T for keys
// 16 w.., P V for head dims w HD/4..) on mma.sync.m16n8k16, with an fp32
// online softmax in the log2 domain over the whole chunk whose row maxima and
// sums are combined across warps in warp order.  fp32 models: CUDA-core dot products.  Partials (m, l, o) per
// (row, query head, chunk) are merged by attn_merge_kernel in a fixed order.
// bf16 launches use programmatic dependent launch: the attention kernel loads
// its first tile of old keys before waiting for the projections that produce
// its queries, and both kernels let their successor launch early.
#include "common.cuh"
#include "internal.h"

namespace ks {

constexpr int kAttnWarps = 4;
constexpr int kPartPad = 4;  // partial row: m, l, 2 pad, o[hd] (16-byte aligned o)
constexpr int kKeyTile = 64;
constexpr int kKvStages = 3;   // bf16: K/V tiles in the cp.async ring (two in flight while computing)

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

// ----------------------------------------------------------- bf16 kernel
// Shared layout (bf16, row pitch hd + 8 elements = 16 B padding):
//   Qs [mpad][P], then kKvStages stages of { Ks [64][HD], Vs [64][HD] }
//   (K / V rows unpadded and chunk-swizzled, see kv_off).
template <int HD>
__global__ void __launch_bounds__(128) attn_bf16_kernel(const AttnArgs a) {
    if (a.stop && *a.stop) return;   // a draft pass after the dynamic exit
    constexpr int NPL = HD / 32;
    constexpr int P = HD + 8;
    constexpr int NDT = HD / 8;  // dim tiles of 8
    constexpr int KT = kKeyTile;
    extern __shared__ __align__(16) unsigned char smem[];

    const int h = blockIdx.x, c = my_chunk(a);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int g = lane >> 2, t = lane & 3;
    const int G = a.hq / a.hk;
    const int M = G * a.R;
    const int mtiles = (M + 15) >> 4;
    const int mpad = mtiles * 16;
    const int cs = attn_chunk_start(c);
    const int ce = min(attn_chunk_start(c + 1), a.p0 + a.R);  // valid keys [cs, ce)
    const int ntiles = (ce - cs + KT - 1) / KT;

    __nv_bfloat16* Qs = reinterpret_cast<__nv_bfloat16*>(smem);
    __nv_bfloat16* KV = Qs + (size_t)mpad * P;  // stage s: K at KV + s*2*KT*HD, V after it

    // The merge kernel may launch now; it reads the partials only after this
    // grid completes.
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

    const __nv_bfloat16* kg = reinterpret_cast<const __nv_bfloat16*>(a.kcache) + (size_t)h * a.max_seq * HD;
    const __nv_bfloat16* vg = reinterpret_cast<const __nv_bfloat16*>(a.vcache) + (size_t)h * a.max_seq * HD;
    constexpr int CPR = HD / 8;  // 16-byte pieces per row
    auto load_tile = [&](int ti) {
        __nv_bfloat16* Ks = KV + (size_t)(ti % kKvStages) * 2 * KT * HD;
        __nv_bfloat16* Vs = Ks + (size_t)KT * HD;
        const int k0 = cs + ti * KT;
        for (int i = tid; i < KT * CPR; i += blockDim.x) {
            const int row = i / CPR, col = (i - row * CPR) * 8;
            const bool ok = k0 + row < ce;
            const size_t off = ok ? (size_t)(k0 + row) * HD + col : 0;
            cp_async16(Ks + kv_off<HD>(row, col), kg + off, ok);
            cp_async16(Vs + kv_off<HD>(row, col), vg + off, ok);
        }
        cp_async_commit();
    };
    // Keys before p0 were written by earlier launches (complete before the
    // projections that precede this kernel could start), so the first tiles
    // of old keys go out before waiting for the projections.
    const int pre = min(kKvStages - 1, ntiles);   // tiles loaded ahead of the loop
    int loaded = 0;
    while (loaded < pre && cs + (loaded + 1) * KT <= a.p0) load_tile(loaded++);
    asm volatile("griddepcontrol.wait;" ::: "memory");

    // 1. new K/V rows of this chunk -> cache (generic stores, then barrier)
    write_new_kv<__nv_bfloat16, NPL>(a, h, cs, ce);
    __syncthreads();
    while (loaded < pre) load_tile(loaded++);

    // 2. queries: m = r * G + gq, scaled into the log2 domain, bf16
    const float qscale = kLog2e * rsqrtf((float)HD);
    const __nv_bfloat16* qn = reinterpret_cast<const __nv_bfloat16*>(a.q_norm);
    constexpr int QB = 4;
    for (int m0 = warp * QB; m0 < mpad; m0 += kAttnWarps * QB) {
        const float* src[QB];
        bool valid[QB];
        int pos[QB];
#pragma unroll
        for (int j = 0; j < QB; ++j) {
            const int m = m0 + j;
            valid[j] = m < M;
            const int r = valid[j] ? m / G : 0, gq = valid[j] ? m - r * G : 0;
            src[j] = a.qkv + (size_t)r * a.qkv_ld + (h * G + gq) * HD;
            pos[j] = a.p0 + r;
        }
        float q[QB][NPL];
        head_vectors<__nv_bfloat16, NPL, QB>(src, valid, pos, qn, a.eps, a.rope, q);
#pragma unroll
        for (int j = 0; j < QB; ++j) {
            const int m = m0 + j;
            if (m >= mpad) continue;
#pragma unroll
            for (int i = 0; i < NPL; ++i)
                Qs[m * P + lane + 32 * i] = __float2bfloat16_rn(valid[j] ? q[j][i] * qscale : 0.f);
        }
    }

    // 3. rounds of up to two m-tiles.  In a round the four warps split every
    //    64-key tile: warp w scores keys 16 w .. 16 w + 15 (Q K^T) and
    //    accumulates head dims w HD/4 .. (w + 1) HD/4 of P V over all 64 keys.
    //    Row maxima and row sums meet in shared memory and are combined in
    //    warp order, so a row's arithmetic is the same for every R.
    constexpr int WD = HD / kAttnWarps;   // head dims per warp
    constexpr int WNT = WD / 8;           // n8 tiles of P V per warp
    constexpr int PP = KT + 8;            // pitch of the probability tile
    __shared__ __align__(16) __nv_bfloat16 Ps[2][16 * PP];
    __shared__ float red_max[2][kAttnWarps][16];
    __shared__ float red_sum[2][kAttnWarps][16];
    for (int mt0 = 0; mt0 < mtiles; mt0 += 2) {
        const int nm = min(2, mtiles - mt0);
        if (mt0 > 0)   // a new round streams the chunk again
            for (int j = 0; j < pre; ++j) load_tile(j);
        uint32_t qf[2][HD / 16][4];
        int rpos[2][2];
        float o[2][WNT][4];
        float mrow[2][2], lrow[2][2];
#pragma unroll
        for (int u = 0; u < 2; ++u)
#pragma unroll
            for (int hh = 0; hh < 2; ++hh) {
                mrow[u][hh] = -INFINITY;
                lrow[u][hh] = 0.f;
                rpos[u][hh] = -1;
            }
#pragma unroll
        for (int u = 0; u < 2; ++u)
#pragma unroll
            for (int i = 0; i < WNT; ++i) o[u][i][0] = o[u][i][1] = o[u][i][2] = o[u][i][3] = 0.f;
        bool qloaded = false;

        for (int ti = 0; ti < ntiles; ++ti) {
            // tile ti + kKvStages - 1 goes into the slot tile ti - 1 used
            if (ti + kKvStages - 1 < ntiles) {
                load_tile(ti + kKvStages - 1);
                cp_async_wait<kKvStages - 1>();
            } else if (ti + 1 < ntiles) {
                cp_async_wait<1>();   // tile ti + 1 may stay in flight
            } else {
                cp_async_wait<0>();
            }
            __syncthreads();  // tile ti (and, first time, Qs) visible
            if (!qloaded) {
#pragma unroll
                for (int u = 0; u < 2; ++u) {
                    if (u >= nm) break;
                    const int mt = mt0 + u;
#pragma unroll
                    for (int ks = 0; ks < HD / 16; ++ks) {
                        const int mi = lane >> 3;
                        const int row = mt * 16 + (mi & 1) * 8 + (lane & 7);
                        const int col = ks * 16 + (mi >> 1) * 8;
                        ldmatrix_x4(qf[u][ks], Qs + row * P + col);
                    }
#pragma unroll
                    for (int hh = 0; hh < 2; ++hh) {
                        const int m = mt * 16 + g + 8 * hh;
                        rpos[u][hh] = (m < M) ? a.p0 + m / G : -1;  // padding rows see no key
                    }
                }
                qloaded = true;
            }
            const __nv_bfloat16* Ks = KV + (size_t)(ti % kKvStages) * 2 * KT * HD;
            const __nv_bfloat16* Vs = Ks + (size_t)KT * HD;
            const int kk = 16 * warp;               // this warp's keys in the tile
            const int kbase = cs + ti * KT + kk;
            // (a) scores of this warp's 16 keys, masked; row maxima to smem
            float sc[2][2][4];
#pragma unroll
            for (int u = 0; u < 2; ++u)
#pragma unroll
                for (int j = 0; j < 2; ++j) sc[u][j][0] = sc[u][j][1] = sc[u][j][2] = sc[u][j][3] = 0.f;
            // each K fragment is loaded once and applied to both m-tiles
#pragma unroll
            for (int ks = 0; ks < HD / 16; ++ks) {
                uint32_t kb[4];
                const int mi = lane >> 3;
                const int krow = kk + (mi >> 1) * 8 + (lane & 7);
                const int kcol = ks * 16 + (mi & 1) * 8;
                ldmatrix_x4(kb, Ks + kv_off<HD>(krow, kcol));
#pragma unroll
                for (int u = 0; u < 2; ++u) {
                    if (u < nm) {
                        mma_bf16(sc[u][0], qf[u][ks][0], qf[u][ks][1], qf[u][ks][2], qf[u][ks][3], kb[0], kb[1]);
                        mma_bf16(sc[u][1], qf[u][ks][0], qf[u][ks][1], qf[u][ks][2], qf[u][ks][3], kb[2], kb[3]);
                    }
                }
            }
#pragma unroll
            for (int u = 0; u < 2; ++u) {
                if (u >= nm) break;
#pragma unroll
                for (int hh = 0; hh < 2; ++hh) {
                    float tmax = -INFINITY;
#pragma unroll
                    for (int j = 0; j < 2; ++j)
#pragma unroll
                        for (int e = 0; e < 2; ++e) {
                            const int key = kbase + j * 8 + 2 * t + e;
                            float& v = sc[u][j][2 * hh + e];
                            if (key > rpos[u][hh] || key >= ce) v = -INFINITY;
                            tmax = fmaxf(tmax, v);
                        }
                    tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, 1));
                    tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, 2));
                    if (t == 0) red_max[u][warp][g + 8 * hh] = tmax;
                }
            }
            __syncthreads();
            // (b) the tile's row maximum, probabilities to smem, row sums to smem
            float alpha[2][2];
#pragma unroll
            for (int u = 0; u < 2; ++u) {
                if (u >= nm) break;
#pragma unroll
                for (int hh = 0; hh < 2; ++hh) {
                    const int row = g + 8 * hh;
                    const float tile_max = fmaxf(fmaxf(red_max[u][0][row], red_max[u][1][row]),
                                                 fmaxf(red_max[u][2][row], red_max[u][3][row]));
                    const float mnew = fmaxf(mrow[u][hh], tile_max);
                    float psum = 0.f;
                    if (mnew == -INFINITY) {
                        alpha[u][hh] = 1.f;
#pragma unroll
                        for (int j = 0; j < 2; ++j) sc[u][j][2 * hh] = sc[u][j][2 * hh + 1] = 0.f;
                    } else {
                        alpha[u][hh] = exp2f(mrow[u][hh] - mnew);
#pragma unroll
                        for (int j = 0; j < 2; ++j)
#pragma unroll
                            for (int e = 0; e < 2; ++e) {
                                float& v = sc[u][j][2 * hh + e];
                                v = exp2f(v - mnew);
                                psum += v;
                            }
                    }
                    mrow[u][hh] = mnew;
                    psum += __shfl_xor_sync(0xffffffffu, psum, 1);
                    psum += __shfl_xor_sync(0xffffffffu, psum, 2);
                    if (t == 0) red_sum[u][warp][row] = psum;
#pragma unroll
                    for (int j = 0; j < 2; ++j)
                        *reinterpret_cast<uint32_t*>(&Ps[u][row * PP + kk + 8 * j + 2 * t]) =
                            pack_bf16(sc[u][j][2 * hh], sc[u][j][2 * hh + 1]);
                }
            }
            __syncthreads();
            // (c) l and o rescaled; O += P V over the 64 keys for this warp's dims
#pragma unroll
            for (int u = 0; u < 2; ++u) {
                if (u >= nm) break;
#pragma unroll
                for (int hh = 0; hh < 2; ++hh) {
                    const int row = g + 8 * hh;
                    const float tsum = ((red_sum[u][0][row] + red_sum[u][1][row]) + red_sum[u][2][row]) +
                                       red_sum[u][3][row];
                    lrow[u][hh] = lrow[u][hh] * alpha[u][hh] + tsum;
#pragma unroll
                    for (int i = 0; i < WNT; ++i) {
                        o[u][i][2 * hh] *= alpha[u][hh];
                        o[u][i][2 * hh + 1] *= alpha[u][hh];
                    }
                }
            }
            // each V fragment is loaded once and applied to both m-tiles
#pragma unroll
            for (int kq = 0; kq < KT / 16; ++kq) {
                uint32_t pa[2][4];
#pragma unroll
                for (int u = 0; u < 2; ++u) {
                    if (u < nm) {
                        const int mi = lane >> 3;
                        const int row = (mi & 1) * 8 + (lane & 7);
                        const int col = kq * 16 + (mi >> 1) * 8;
                        ldmatrix_x4(pa[u], &Ps[u][row * PP + col]);
                    }
                }
#pragma unroll
                for (int dq = 0; dq < WNT / 2; ++dq) {
                    uint32_t vb[4];
                    const int mi = lane >> 3;
                    const int vrow = kq * 16 + (mi & 1) * 8 + (lane & 7);
                    const int vcol = warp * WD + dq * 16 + (mi >> 1) * 8;
                    ldmatrix_x4_trans(vb, Vs + kv_off<HD>(vrow, vcol));
#pragma unroll
                    for (int u = 0; u < 2; ++u) {
                        if (u < nm) {
                            mma_bf16(o[u][2 * dq], pa[u][0], pa[u][1], pa[u][2], pa[u][3], vb[0], vb[1]);
                            mma_bf16(o[u][2 * dq + 1], pa[u][0], pa[u][1], pa[u][2], pa[u][3], vb[2], vb[3]);
                        }
                    }
                }
            }
            __syncthreads();  // everyone is done with tile ti (and Ps, red_*) before reuse
        }
        // this chunk's partials: m and l by warp 0, each warp its dims of o
#pragma unroll
        for (int u = 0; u < 2; ++u) {
            if (u >= nm) break;
#pragma unroll
            for (int hh = 0; hh < 2; ++hh) {
                const int m = (mt0 + u) * 16 + g + 8 * hh;
                if (m >= M) continue;
                const int r = m / G, gq = m - r * G;
                float* dst = a.part + (((size_t)r * a.hq + h * G + gq) * a.n_chunks_max + c) * (HD + kPartPad);
                if (warp == 0 && t == 0) {
                    dst[0] = mrow[u][hh];
                    dst[1] = lrow[u][hh];
                }
#pragma unroll
                for (int i = 0; i < WNT; ++i) {
                    dst[kPartPad + warp * WD + i * 8 + 2 * t] = o[u][i][2 * hh];
                    dst[kPartPad + warp * WD + i * 8 + 2 * t + 1] = o[u][i][2 * hh + 1];
                }
            }
        }
    }
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
// max is exact in any order; l and o are summed per thread (stride 128 over
// chunks) or per warp (chunks c = w mod 4) and then in thread / warp order.
// The chunk count depends only on the row's position, so a row gives the
// same bits in a 1-row pass and in a gamma+1-row pass.
template <typename WT, int HD>
__global__ void __launch_bounds__(128) attn_merge_kernel(const AttnArgs a) {
    if (a.stop && *a.stop) return;   // a draft pass after the dynamic exit
    extern __shared__ float wsh[];  // [nch] chunk weights
    __shared__ float red[kAttnWarps + 1];
    __shared__ float osh[kAttnWarps][HD];
    const int hq_idx = blockIdx.x, r = blockIdx.y;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");   // the next projections may launch
    asm volatile("griddepcontrol.wait;" ::: "memory");                // the partials are complete
    const int pos = a.p0 + r;
    const int nch = attn_chunk_of(pos) + 1;
    constexpr int S = HD + kPartPad;
    const float* base = a.part + ((size_t)r * a.hq + hq_idx) * a.n_chunks_max * S;
    float mx = -INFINITY;
    for (int c = tid; c < nch; c += blockDim.x) mx = fmaxf(mx, base[(size_t)c * S]);
    mx = warp_max(mx);
    if (lane == 0) red[warp] = mx;
    __syncthreads();
    mx = fmaxf(fmaxf(red[0], red[1]), fmaxf(red[2], red[3]));
    float ls = 0.f;
    for (int c = tid; c < nch; c += blockDim.x) {
        const float m = base[(size_t)c * S];
        const float w = (m == -INFINITY) ? 0.f : exp2f(m - mx);
        wsh[c] = w;
        ls = fmaf(w, base[(size_t)c * S + 1], ls);
    }
    const float L = block_sum<kAttnWarps>(ls, red);  // ends with a barrier: wsh is visible
    constexpr int PER = HD / 32;                     // dims per lane
    float o[PER];
#pragma unroll
    for (int i = 0; i < PER; ++i) o[i] = 0.f;
#pragma unroll 8
    for (int c = warp; c < nch; c += kAttnWarps) {   // unrolled: several chunks' loads in flight
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
        const float O = ((osh[0][d] + osh[1][d]) + osh[2][d]) + osh[3][d];
        out[(size_t)r * a.out_ld + hq_idx * HD + d] = from_float<WT>(O / L);
    }
}

// --------------------------------------------------------------- launchers
static size_t attn_bf16_smem(int HD, int mpad) {
    const int P = HD + 8;
    return sizeof(__nv_bfloat16) * ((size_t)mpad * P + (size_t)kKvStages * 2 * kKeyTile * HD);
}

cudaError_t launch_attention(int dtype, const AttnArgs& a, cudaStream_t s) {
    const int nch = attn_num_chunks(a.p0 + a.R);
    if (nch > a.n_chunks_max || a.p0 + a.R > a.max_seq) return cudaErrorInvalidValue;
    dim3 grid(a.hk, nch);
    if (dtype == 1) {
        const int M = (a.hq / a.hk) * a.R;
        const int mpad = ((M + 15) / 16) * 16;
        const size_t smem = attn_bf16_smem(a.hd, mpad);
        auto run = [&](auto kern) -> cudaError_t {
            cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
            if (e != cudaSuccess) return e;
            cudaLaunchConfig_t cfg = {};
            cfg.gridDim = grid;
            cfg.blockDim = dim3(128);
            cfg.dynamicSmemBytes = smem;
            cfg.stream = s;
            cudaLaunchAttribute attr[1];
            attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
            attr[0].val.programmaticStreamSerializationAllowed = 1;
            cfg.attrs = attr;
            cfg.numAttrs = 1;
            return cudaLaunchKernelEx(&cfg, kern, a);
        };
        if (a.hd == 128) return run(attn_bf16_kernel<128>);
        if (a.hd == 64) return run(attn_bf16_kernel<64>);
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
    if (smem > 48 * 1024) return cudaErrorInvalidValue;
    if (dtype == 1) {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = grid;
        cfg.blockDim = dim3(128);
        cfg.dynamicSmemBytes = smem;
        cfg.stream = s;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        if (a.hd == 128) return cudaLaunchKernelEx(&cfg, attn_merge_kernel<__nv_bfloat16, 128>, a);
        return cudaLaunchKernelEx(&cfg, attn_merge_kernel<__nv_bfloat16, 64>, a);
    } else {
        if (a.hd == 128) attn_merge_kernel<float, 128><<<grid, 128, smem, s>>>(a);
        else attn_merge_kernel<float, 64><<<grid, 128, smem, s>>>(a);
    }
    return cudaGetLastError();
}

}  // namespace ks
