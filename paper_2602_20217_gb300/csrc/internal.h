// Internal interfaces between the translation units of libknapspec.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace ks {

// ------------------------------------------------------------------ GEMV
// Y[r][n] = sum_k W[n][k] * A[r][k] for r < R rows ("skinny GEMM"), with a
// fused prologue (optional RMSNorm of an fp32 residual input) and epilogue.
enum GemvEpi { EPI_STORE = 0, EPI_RESID = 1, EPI_SWIGLU = 2, EPI_LMHEAD = 3 };

struct GemvArgs {
    const void* W;          // [N (or 2N for SwiGLU)][K], row stride K, model dtype
    int N;                  // output features (SwiGLU: d_ff; rows n and N + n pair up)
    int K;
    int R;                  // activation rows, 1..16
    int ksplit;             // K slices (grid.y); set by gemv_plan
    int kc;                 // K per slice (multiple of 64)
    const void* in;         // fp32 residual [R][in_ld] when norm_gain != null, else model dtype [R][in_ld]
    int in_ld;
    const void* norm_gain;  // RMSNorm gain [K] (model dtype) or null
    float eps;
    float* out; int out_ld;                    // EPI_STORE (fp32)
    float* resid; int resid_ld;                // EPI_RESID: resid[r][n] += y
    float* capture; long long capture_ld;      // EPI_RESID: optional copy of the new residual
    void* act; int act_ld;                     // EPI_SWIGLU: silu(gate) * up, model dtype
    float* logits; int logits_ld;              // EPI_LMHEAD
    float* amax_val; int* amax_idx;            // EPI_LMHEAD per-CTA partials [grid.x][16]
    int* tokens;                               // EPI_LMHEAD argmax per row
    float* partial;                            // split-K partials [ksplit][R][N or 2N]
    int* counters;                             // per-CTA-column arrival counters (+1 global)
};

void gemv_plan(GemvArgs& a, int epi);           // choose ksplit / kc from (N, K) only
size_t gemv_partial_floats(int N, int K, int R, int epi);
int gemv_grid_x(int N);
cudaError_t launch_gemv(int dtype, int epi, const GemvArgs& a, cudaStream_t s);

// ------------------------------------------------------------- attention
struct AttnArgs {
    const float* qkv;       // [R][(hq + 2 hk) hd] fp32 projections (pre-norm, pre-RoPE)
    int qkv_ld;
    int R;
    int p0;                 // position of row 0; row r is at p0 + r
    int hq, hk, hd;
    void* kcache;           // [hk][max_seq][hd] model dtype (this layer)
    void* vcache;
    int max_seq;
    const float* rope;      // [max_seq][hd/2][2] (cos, sin) fp32
    const void* q_norm;     // [hd] or null (model dtype)
    const void* k_norm;
    float eps;
    int chunk;              // keys per CTA (fixed; split boundaries are absolute)
    float* part;            // [R][hq][n_chunks_max][hd + 2] (m, l, o[hd])
    int n_chunks_max;
    void* out;              // [R][hq hd] model dtype: merged attention output
    int out_ld;
};

cudaError_t launch_attention(int dtype, const AttnArgs& a, cudaStream_t s);
cudaError_t launch_attn_merge(int dtype, const AttnArgs& a, cudaStream_t s);
constexpr int kAttnChunk = 128;

// ---------------------------------------------------------------- select
cudaError_t launch_cosine(const void* X, const void* Y, int dtype, int64_t n_pairs, int rows,
                          int d, int64_t pair_stride, const int32_t* row_index, float* out,
                          cudaStream_t s);

// Last error text for ks_last_error (thread-local).
void set_error(const char* fmt, ...);

}  // namespace ks
