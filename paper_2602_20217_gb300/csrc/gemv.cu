// Skinny GEMM kernel for fp32 models (the tiny parity workload), plus the
// TMA descriptor helper used by the bf16 chain kernel.
//
// Y[r][n] = sum_k W[n][k] A[r][k] for R <= 16 rows: the per-token
// projections of the Attn and MLP sublayers and the LM head (Sec. 2 decoder;
// every pass of a1 / a2).  One CTA per (64-feature group, K slice); each
// warp computes 16 features with CUDA-core dot products and hands its results
// over in the mma fragment layout the bf16 path uses, so both share one set
// of epilogues: plain store (QKV), residual add with optional history capture
// and partial sums of squares (W_o, W_down), SwiGLU (gate and up rows paired
// in one warp), LM head logits with a per-row argmax (ties to the lowest id).
// K slices are added in slice order by the last CTA of a group (an atomic
// ticket, no waiting): results depend only on (N, K), never on R.  The
// optional RMSNorm prologue builds each row's sum of squares from the
// per-16-feature partials that the residual's producer wrote, in group order.
#include "common.cuh"
#include "internal.h"

#include <cudaTypedefs.h>

#include <climits>

namespace ks {

constexpr int kGemvWarps = 4;
constexpr int kRowsPerCta = 16 * kGemvWarps;  // output features per group (CTA or work item)
constexpr int kMaxRows = 16;
// counters: [0] next work item, [1] finished CTAs, [2 + g] ticket of group g

__host__ __device__ __forceinline__ int div_up(int a, int b) { return (a + b - 1) / b; }

int gemv_grid_x(int N) { return div_up(N, kRowsPerCta); }
int gemv_groups(int N, int dtype) { return dtype == 1 ? div_up(N, 16) : div_up(N, kRowsPerCta); }

int sm_count() {
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
    if (a.stop && *a.stop) return;   // a draft pass after the dynamic exit
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

// ---------------------------------------------------------------- launcher
static PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
    static PFN_cuTensorMapEncodeTiled_v12000 encode = nullptr;
    if (encode == nullptr) {
        void* fn = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) !=
                cudaSuccess ||
            q != cudaDriverEntryPointSuccess || fn == nullptr)
            return nullptr;
        encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    }
    return encode;
}

bool make_tma_map(CUtensorMap* map, const void* base, uint64_t rows, uint64_t K, uint32_t box_rows) {
    auto encode = tensor_map_encoder();
    if (!encode || K % 8 != 0 || (reinterpret_cast<uintptr_t>(base) & 15) != 0) return false;
    const cuuint64_t dims[2] = {K, rows};
    const cuuint64_t strides[1] = {K * 2};
    const cuuint32_t box[2] = {256, box_rows};
    const cuuint32_t estr[2] = {1, 1};
    return encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool make_weight_map(CUtensorMap* map, const void* base, uint64_t rows, uint64_t K, uint32_t chunks) {
    auto encode = tensor_map_encoder();
    if (!encode || K % 8 != 0 || (reinterpret_cast<uintptr_t>(base) & 15) != 0) return false;
    const cuuint32_t estr[3] = {1, 1, 1};
    if (K % 64 == 0) {
        // {64 columns, rows, K / 64 chunks}: a box is `chunks` chunks of 16 rows
        const cuuint64_t dims[3] = {64, rows, K / 64};
        const cuuint64_t strides[2] = {K * 2, 128};
        const cuuint32_t box[3] = {64, 16, chunks};
        return encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
                      CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                      CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
    }
    const cuuint64_t dims[2] = {K, rows};
    const cuuint64_t strides[1] = {K * 2};
    const cuuint32_t box[2] = {64, 16};
    return encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool make_stage_map(CUtensorMap* map, const void* base, uint64_t rows, uint64_t K, uint32_t box_rows,
                    uint32_t chunks) {
    if (K % 256 != 0) return make_tma_map(map, base, rows, K, box_rows);
    auto encode = tensor_map_encoder();
    if (!encode || (reinterpret_cast<uintptr_t>(base) & 15) != 0) return false;
    // [rows][K] viewed as {256 columns, rows, K / 256 chunks}: one box holds
    // `chunks` consecutive 256-column chunks of box_rows rows, chunk-major
    const cuuint64_t dims[3] = {256, rows, K / 256};
    const cuuint64_t strides[2] = {K * 2, 512};
    const cuuint32_t box[3] = {256, box_rows, chunks};
    const cuuint32_t estr[3] = {1, 1, 1};
    return encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
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
    // fp32 models only; bf16 projections run in the chain kernel
    if (a.R < 1 || a.R > kMaxRows || a.dtype != dtype || dtype != 0) return cudaErrorInvalidValue;
    switch (epi) {
        case EPI_STORE: return launch_f32<EPI_STORE>(a, s);
        case EPI_RESID: return launch_f32<EPI_RESID>(a, s);
        case EPI_SWIGLU: return launch_f32<EPI_SWIGLU>(a, s);
        default: return launch_f32<EPI_LMHEAD>(a, s);
    }
}

}  // namespace ks
