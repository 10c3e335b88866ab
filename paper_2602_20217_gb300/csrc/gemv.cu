// Skinny GEMM kernels for the decode / verify passes (R <= 16 activation rows).
//
// Y[r][n] = sum_k W[n][k] A[r][k]: the per-token projections of the Attn and
// MLP sublayers and the LM head (Sec. 2 decoder; every pass of a1 / a2).  At
// R <= 16 rows the work is a stream over the weights (at most 16 flop per
// weight byte pair), so the kernels are built to keep HBM busy:
//  * every lane streams 16-byte chunks of two weight rows with
//    ld.global.nc.L1::no_allocate, several steps unrolled so each warp keeps
//    2 x U x 512 bytes in flight;
//  * bf16 models: the weight chunks are fed as the A operand of
//    mma.sync.m16n8k16 (16 weight rows x 16 k) and the activation rows as B
//    (16 k x 8 rows).  The k-slots of A and B are permuted identically so a
//    lane's 8 contiguous weights and 8 contiguous activations are one MMA
//    pair; column j of the result depends only on activation row j, so one
//    row computed alone (greedy decode) and the same row inside a gamma+1 row
//    verify pass are bit-identical;
//  * fp32 models (the tiny parity workload) use CUDA-core FMAs in the same
//    tile structure;
//  * K is split over ksplit CTAs when there are too few row tiles to fill
//    152 SMs; fp32 partials are summed in slice order by the last CTA to
//    arrive (an atomic ticket, no waiting), so results do not depend on
//    arrival order;
//  * prologue: optional RMSNorm of the fp32 residual (computed by every CTA
//    over the full row in a fixed order); epilogues: plain store (QKV),
//    residual add with optional history capture (W_o, W_down), SwiGLU
//    (gate and up rows paired in one warp), LM head with argmax.
#include "common.cuh"
#include "internal.h"

#include <climits>

namespace ks {

constexpr int kGemvWarps = 4;
constexpr int kRowsPerCta = 16 * kGemvWarps;  // output features per CTA
constexpr int kMaxRows = 16;

static int div_up(int a, int b) { return (a + b - 1) / b; }

int gemv_grid_x(int N) { return div_up(N, kRowsPerCta); }

void gemv_plan(GemvArgs& a, int epi) {
    // Depends on (N, K) only, never on R: the split decides the summation
    // order, which must be the same for 1 row and for gamma + 1 rows.
    const int gx = gemv_grid_x(a.N);
    int s = 1;
    if (epi != EPI_LMHEAD) {
        const int target = 2 * 152;
        s = div_up(target, gx);
        if (s > 16) s = 16;
        if (s < 1) s = 1;
    }
    int kc = div_up(div_up(a.K, s), 64) * 64;
    if (kc < 64) kc = 64;
    a.kc = kc;
    a.ksplit = div_up(a.K, kc);
}

size_t gemv_partial_floats(int N, int K, int R, int epi) {
    GemvArgs a{};
    a.N = N;
    a.K = K;
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
    if (a.norm_gain != nullptr) {
        const float* x = reinterpret_cast<const float*>(a.in);
        const WT* gain = reinterpret_cast<const WT*>(a.norm_gain);
        float ss[kMaxRows];
#pragma unroll
        for (int r = 0; r < kMaxRows; ++r) {
            float s = 0.f;
            if (r < R) {
                const float* xr = x + (size_t)r * a.in_ld;
                for (int k = tid; k < a.K; k += blockDim.x) s = fmaf(xr[k], xr[k], s);
            }
            ss[r] = warp_sum(s);
        }
        const int lane = tid & 31, w = tid >> 5;
        if (lane == 0) {
#pragma unroll
            for (int r = 0; r < kMaxRows; ++r) red[w * kMaxRows + r] = ss[r];
        }
        __syncthreads();
        if (tid < R) {
            float s = 0.f;
            for (int i = 0; i < kGemvWarps; ++i) s += red[i * kMaxRows + tid];
            red[kGemvWarps * kMaxRows + tid] = rsqrtf(s / (float)a.K + a.eps);
        }
        __syncthreads();
        for (int idx = tid; idx < R * kc; idx += blockDim.x) {
            const int r = idx / kc, k = idx - r * kc;
            const int kg = kbeg + k;
            float v = 0.f;
            if (kg < a.K) v = (x[(size_t)r * a.in_ld + kg] * red[kGemvWarps * kMaxRows + r]) * to_float(gain[kg]);
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

// -------------------------------------------------------------- main loops
// bf16: each warp owns 16 weight rows (and, for SwiGLU, the 16 paired up
// rows).  Lane (g = lane / 4, t = lane % 4) loads 8 weights of rows g and
// g + 8 at k = 32 s + 8 t and the 8 matching activations of row g of each
// 8-row group.
template <int NT, bool PAIR, int U>
KS_DEV void mma_rows(const __nv_bfloat16* w0, const __nv_bfloat16* w1, const __nv_bfloat16* u0,
                     const __nv_bfloat16* u1, bool ok0, bool ok1, const __nv_bfloat16* act,
                     int pitch, int R, int kc, int kvalid, float (&acc)[NT][4],
                     float (&accu)[NT][4]) {
    const int lane = threadIdx.x & 31, g = lane >> 2, t = lane & 3;
    const uint4 z = make_uint4(0, 0, 0, 0);
    const int nsteps = kc >> 5;
    for (int s0 = 0; s0 < nsteps; s0 += U) {
        uint4 a0[U], a1[U], c0[U], c1[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int k = (s0 + u) * 32 + 8 * t;
            const bool kin = k < kvalid;
            a0[u] = (kin && ok0) ? ldg_stream(w0 + k) : z;
            a1[u] = (kin && ok1) ? ldg_stream(w1 + k) : z;
            if (PAIR) {
                c0[u] = (kin && ok0) ? ldg_stream(u0 + k) : z;
                c1[u] = (kin && ok1) ? ldg_stream(u1 + k) : z;
            }
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int k = (s0 + u) * 32 + 8 * t;
            const bool kin = (s0 + u) < nsteps;
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) {
                const int r = nt * 8 + g;
                const uint4 b = (kin && r < R) ? lds128(act + r * pitch + k) : z;
                mma_bf16(acc[nt], a0[u].x, a1[u].x, a0[u].y, a1[u].y, b.x, b.y);
                mma_bf16(acc[nt], a0[u].z, a1[u].z, a0[u].w, a1[u].w, b.z, b.w);
                if (PAIR) {
                    mma_bf16(accu[nt], c0[u].x, c1[u].x, c0[u].y, c1[u].y, b.x, b.y);
                    mma_bf16(accu[nt], c0[u].z, c1[u].z, c0[u].w, c1[u].w, b.z, b.w);
                }
            }
        }
    }
}

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
    } else if (EPI == EPI_SWIGLU) {
        WT* act = reinterpret_cast<WT*>(a.act);
        act[(size_t)r * a.act_ld + n] = from_float<WT>(silu(v) * vu);
    }
}

// ------------------------------------------------------------------ kernel
template <typename WT, int NT, int EPI>
__global__ void __launch_bounds__(128) gemv_kernel(const GemvArgs a) {
    constexpr bool PAIR = (EPI == EPI_SWIGLU);
    extern __shared__ __align__(16) unsigned char smem[];
    __shared__ float red[kGemvWarps * kMaxRows + kMaxRows];
    __shared__ float wbest_v[kGemvWarps][kMaxRows];
    __shared__ int wbest_i[kGemvWarps][kMaxRows];
    __shared__ int is_last;

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int g = lane >> 2, t = lane & 3;
    const int kbeg = blockIdx.y * a.kc;
    const int kvalid = min(a.kc, a.K - kbeg);
    const int pitch = (sizeof(WT) == 2) ? (a.kc + 32) : (a.kc + 4);
    WT* act = reinterpret_cast<WT*>(smem);

    stage_activations<WT>(a, act, pitch, kbeg, red);

    const int n_base = blockIdx.x * kRowsPerCta + warp * 16;
    float acc[NT][4], accu[NT][4];
#pragma unroll
    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int i = 0; i < 4; ++i) acc[nt][i] = accu[nt][i] = 0.f;

    if constexpr (sizeof(WT) == 2) {
        const __nv_bfloat16* W = reinterpret_cast<const __nv_bfloat16*>(a.W);
        const int n0 = n_base + g, n1 = n_base + g + 8;
        const bool ok0 = n0 < a.N, ok1 = n1 < a.N;
        const __nv_bfloat16* w0 = W + (size_t)(ok0 ? n0 : 0) * a.K + kbeg;
        const __nv_bfloat16* w1 = W + (size_t)(ok1 ? n1 : 0) * a.K + kbeg;
        const __nv_bfloat16* u0 = PAIR ? w0 + (size_t)a.N * a.K : nullptr;
        const __nv_bfloat16* u1 = PAIR ? w1 + (size_t)a.N * a.K : nullptr;
        constexpr int U = (PAIR ? 4 : 8) / NT;
        mma_rows<NT, PAIR, U>(w0, w1, u0, u1, ok0, ok1,
                              reinterpret_cast<const __nv_bfloat16*>(act), pitch, a.R, a.kc,
                              kvalid, acc, accu);
    } else {
        float* tile = reinterpret_cast<float*>(smem + sizeof(WT) * (size_t)a.R * pitch) +
                      warp * 2 * 16 * 16;
        fma_rows<NT, PAIR>(reinterpret_cast<const float*>(a.W), a.K, a.N, n_base, kbeg,
                           reinterpret_cast<const float*>(act), pitch, a.R, a.kc, kvalid, tile,
                           acc, accu);
    }

    // Fragment ownership: acc[nt][0] = (n_base+g, row nt*8+2t), [1] = (n_base+g, +1),
    // [2] = (n_base+g+8, nt*8+2t), [3] = (n_base+g+8, +1).
    if (EPI == EPI_LMHEAD) {
        const float NEG = -INFINITY;
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
#pragma unroll
            for (int c = 0; c < 2; ++c) {
                const int r = nt * 8 + 2 * t + c;
                float bv = NEG;
                int bi = INT_MAX;
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int n = n_base + g + 8 * h;
                    const float v = acc[nt][2 * h + c];
                    if (n < a.N && r < a.R) {
                        a.logits[(size_t)r * a.logits_ld + n] = v;
                        if (better(v, n, bv, bi)) { bv = v; bi = n; }
                    }
                }
#pragma unroll
                for (int o = 4; o < 32; o <<= 1) {
                    const float ov = __shfl_xor_sync(0xffffffffu, bv, o);
                    const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
                    if (better(ov, oi, bv, bi)) { bv = ov; bi = oi; }
                }
                if (g == 0 && r < kMaxRows) {
                    wbest_v[warp][r] = bv;
                    wbest_i[warp][r] = bi;
                }
            }
        }
        __syncthreads();
        if (tid < a.R) {
            float bv = NEG;
            int bi = INT_MAX;
            for (int w = 0; w < kGemvWarps; ++w)
                if (better(wbest_v[w][tid], wbest_i[w][tid], bv, bi)) {
                    bv = wbest_v[w][tid];
                    bi = wbest_i[w][tid];
                }
            a.amax_val[blockIdx.x * kMaxRows + tid] = bv;
            a.amax_idx[blockIdx.x * kMaxRows + tid] = bi;
        }
        __threadfence();
        __syncthreads();
        if (tid == 0) {
            const int prev = atomicAdd(&a.counters[gridDim.x], 1);
            is_last = (prev == (int)gridDim.x - 1);
        }
        __syncthreads();
        if (!is_last) return;
        __threadfence();
        // The last CTA: one warp per row scans every CTA's candidate.
        for (int r = warp; r < a.R; r += kGemvWarps) {
            float bv = NEG;
            int bi = INT_MAX;
            for (int c = lane; c < (int)gridDim.x; c += 32) {
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
        if (tid == 0) a.counters[gridDim.x] = 0;
        return;
    }

    if (a.ksplit == 1) {
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int n = n_base + g + 8 * (i >> 1);
                const int r = nt * 8 + 2 * t + (i & 1);
                if (n < a.N && r < a.R) apply_epilogue<WT, EPI>(a, n, r, acc[nt][i], accu[nt][i]);
            }
        return;
    }

    // Split K: publish partials, take a ticket; the last CTA of this column
    // sums the slices in slice order and applies the epilogue.
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
    if (tid == 0) {
        const int prev = atomicAdd(&a.counters[blockIdx.x], 1);
        is_last = (prev == a.ksplit - 1);
    }
    __syncthreads();
    if (!is_last) return;
    __threadfence();
    const int row0 = blockIdx.x * kRowsPerCta;
    for (int idx = tid; idx < kRowsPerCta * a.R; idx += blockDim.x) {
        const int r = idx / kRowsPerCta;
        const int n = row0 + (idx - r * kRowsPerCta);
        if (n >= a.N) continue;
        float v = 0.f, vu = 0.f;
        for (int s = 0; s < a.ksplit; ++s) {
            const float* p = a.partial + ((size_t)s * a.R + r) * NP;
            v += __ldcg(p + n);
            if (PAIR) vu += __ldcg(p + a.N + n);
        }
        apply_epilogue<WT, EPI>(a, n, r, v, vu);
    }
    if (tid == 0) a.counters[blockIdx.x] = 0;
}

// ---------------------------------------------------------------- launcher
template <typename WT, int EPI>
static cudaError_t launch_t(const GemvArgs& a, cudaStream_t s) {
    const int pitch = (sizeof(WT) == 2) ? (a.kc + 32) : (a.kc + 4);
    size_t smem = sizeof(WT) * (size_t)a.R * pitch;
    if (sizeof(WT) == 4) smem += sizeof(float) * kGemvWarps * 2 * 16 * 16;
    dim3 grid(gemv_grid_x(a.N), a.ksplit);
    auto run = [&](auto kern) -> cudaError_t {
        if (smem > 48 * 1024) {
            cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                 (int)smem);
            if (e != cudaSuccess) return e;
        }
        kern<<<grid, 128, smem, s>>>(a);
        return cudaGetLastError();
    };
    if (a.R <= 8) return run(gemv_kernel<WT, 1, EPI>);
    return run(gemv_kernel<WT, 2, EPI>);
}

cudaError_t launch_gemv(int dtype, int epi, const GemvArgs& a, cudaStream_t s) {
    if (a.R < 1 || a.R > kMaxRows) return cudaErrorInvalidValue;
    if (dtype == 1) {
        switch (epi) {
            case EPI_STORE: return launch_t<__nv_bfloat16, EPI_STORE>(a, s);
            case EPI_RESID: return launch_t<__nv_bfloat16, EPI_RESID>(a, s);
            case EPI_SWIGLU: return launch_t<__nv_bfloat16, EPI_SWIGLU>(a, s);
            default: return launch_t<__nv_bfloat16, EPI_LMHEAD>(a, s);
        }
    }
    switch (epi) {
        case EPI_STORE: return launch_t<float, EPI_STORE>(a, s);
        case EPI_RESID: return launch_t<float, EPI_RESID>(a, s);
        case EPI_SWIGLU: return launch_t<float, EPI_SWIGLU>(a, s);
        default: return launch_t<float, EPI_LMHEAD>(a, s);
    }
}

}  // namespace ks
