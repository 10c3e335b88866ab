// The hidden-state dynamic program of Alg. 1 (Sec. 3.4) on the device: the
// per-sublayer bookkeeping kernels.  The sublayer evaluations themselves are
// ordinary decoder passes (model.cu) over one state's history rows.
//
// State j (skipped weight j = 0 .. J-1) holds r rows of d floats.  For
// sublayer i:
//   dp_cos_kernel     sigma of every execute candidate E[j] and of every
//                     state G[j] against the target's X^(i) rows;
//   dp_select_kernel  the pull form: g[i, j] = E[j] when its cosine is >= the
//                     skip candidate G[j - w_i]'s (ties execute), valid when
//                     its source is valid and its cosine >= tau; column 0 is
//                     X^(i); records the choice and the validity word that
//                     gates the next evaluations;
//   dp_gather_kernel  copies the chosen rows into the next state buffer.
// dp_backtrack_kernel rebuilds each terminal state's layer set from the
// choices (at j = 0 every remaining sublayer is executed).
#include "common.cuh"
#include "internal.h"

#include <cfloat>

namespace ks {

namespace {

constexpr int kCosThreads = 256;

// mean over the r rows of cos(A_r, B_r); A: a state's contiguous rows, B: the
// history plane's rows hidx[0..r).  One CTA per state, fixed reduction order.
__global__ void __launch_bounds__(kCosThreads) dp_cos_kernel(const float* A, long long a_stride, const float* B,
                                                             const int32_t* hidx, int r, int d, float* sig) {
    const float* a = A + (size_t)blockIdx.x * a_stride;
    __shared__ float red[3][kCosThreads / 32 + 1];
    float acc = 0.f;
    for (int row = 0; row < r; ++row) {
        const float* x = a + (size_t)row * d;
        const float* y = B + (size_t)hidx[row] * d;
        float xy = 0.f, xx = 0.f, yy = 0.f;
        for (int k = threadIdx.x; k < d; k += kCosThreads) {
            const float u = x[k], v = y[k];
            xy = fmaf(u, v, xy);
            xx = fmaf(u, u, xx);
            yy = fmaf(v, v, yy);
        }
        xy = block_sum<kCosThreads / 32>(xy, red[0]);
        xx = block_sum<kCosThreads / 32>(xx, red[1]);
        yy = block_sum<kCosThreads / 32>(yy, red[2]);
        acc += xy / (sqrtf(xx) * sqrtf(yy));
    }
    if (threadIdx.x == 0) sig[blockIdx.x] = acc / (float)r;
}

// One thread per skipped weight j.  valid_*: 0 valid, 1 invalid (the value
// the decoder kernels read as their stop word).  choice: 0 execute, 1 skip,
// 2 invalid.  src: the row source of the new state (-1: X^(i), else 2 j' for
// E[j'], 2 j' + 1 for G[j']).
__global__ void dp_select_kernel(int J, int w, float tau, const int* valid_prev, const float* sig_e,
                                 const float* sig_s, int* valid_cur, float* sig_cur, uint8_t* choice, int* src) {
    const int j = threadIdx.x;
    if (j >= J) return;
    const bool e_ok = valid_prev[j] == 0;
    const bool s_ok = j >= w && valid_prev[j - w] == 0;
    const float se = j == 0 ? 1.f : sig_e[j];
    const float ss = s_ok ? sig_s[j - w] : -FLT_MAX;
    int c = 2, s = 0;
    float sg = 0.f;
    if (e_ok && (!s_ok || se >= ss)) {
        c = 0;
        sg = se;
        s = j == 0 ? -1 : 2 * j;
    } else if (s_ok) {
        c = 1;
        sg = ss;
        s = 2 * (j - w) + 1;
    }
    if (c != 2 && !(sg >= tau)) c = 2;
    valid_cur[j] = c == 2 ? 1 : 0;
    sig_cur[j] = sg;
    choice[j] = (uint8_t)c;
    src[j] = s;
}

// grid (J, ceil(d / 256)): row block of state j from its source
__global__ void __launch_bounds__(256) dp_gather_kernel(const int* src, const int* valid_cur, const float* E,
                                                        const float* G_prev, long long stride, const float* X,
                                                        const int32_t* hidx, int r, int d, float* G_cur) {
    const int j = blockIdx.x;
    if (valid_cur[j]) return;
    const int k = blockIdx.y * 256 + threadIdx.x;
    if (k >= d) return;
    const int s = src[j];
    float* out = G_cur + (size_t)j * stride;
    for (int row = 0; row < r; ++row) {
        float v;
        if (s < 0) v = X[(size_t)hidx[row] * d + k];
        else if (s & 1) v = G_prev[(size_t)(s >> 1) * stride + (size_t)row * d + k];
        else v = E[(size_t)(s >> 1) * stride + (size_t)row * d + k];
        out[(size_t)row * d + k] = v;
    }
}

// one thread per candidate: candidate c is terminal state js[c]
__global__ void dp_backtrack_kernel(int n_cand, const int* js, int n_items, int J, const uint8_t* choices,
                                    const int* w, uint8_t* masks) {
    const int c = blockIdx.x * blockDim.x + threadIdx.x;
    if (c >= n_cand) return;
    int j = js[c];
    uint8_t* m = masks + (size_t)c * n_items;
    for (int i = n_items; i >= 1; --i) {
        const uint8_t ch = choices[(size_t)(i - 1) * J + j];
        if (j == 0 || ch == 0) {
            m[i - 1] = 1;
        } else {
            m[i - 1] = 0;
            j -= w[i - 1];
        }
    }
}

// the terminal candidates in executed-weight order (j descending) and their count
__global__ void dp_candidates_kernel(int J, const int* valid, int* js, int* n_cand) {
    if (threadIdx.x != 0) return;
    int n = 0;
    for (int j = J - 1; j >= 0; --j)
        if (valid[j] == 0) js[n++] = j;
    *n_cand = n;
}

}  // namespace

cudaError_t launch_dp_cos(const float* A, long long stride, int n, const float* B, const int32_t* hidx, int r, int d,
                          float* sig, cudaStream_t s) {
    if (n < 1) return cudaSuccess;
    dp_cos_kernel<<<n, kCosThreads, 0, s>>>(A, stride, B, hidx, r, d, sig);
    return cudaGetLastError();
}

cudaError_t launch_dp_select(int J, int w, float tau, const int* valid_prev, const float* sig_e, const float* sig_s,
                             int* valid_cur, float* sig_cur, uint8_t* choice, int* src, cudaStream_t s) {
    if (J < 1 || J > 1024) return cudaErrorInvalidValue;
    dp_select_kernel<<<1, J, 0, s>>>(J, w, tau, valid_prev, sig_e, sig_s, valid_cur, sig_cur, choice, src);
    return cudaGetLastError();
}

cudaError_t launch_dp_gather(int J, const int* src, const int* valid_cur, const float* E, const float* G_prev,
                             long long stride, const float* X, const int32_t* hidx, int r, int d, float* G_cur,
                             cudaStream_t s) {
    dp_gather_kernel<<<dim3(J, (d + 255) / 256), 256, 0, s>>>(src, valid_cur, E, G_prev, stride, X, hidx, r, d,
                                                              G_cur);
    return cudaGetLastError();
}

cudaError_t launch_dp_backtrack(const int* js, int n_cand, int n_items, int J, const uint8_t* choices, const int* w,
                                uint8_t* masks, cudaStream_t s) {
    if (n_cand < 1) return cudaSuccess;
    dp_backtrack_kernel<<<(n_cand + 127) / 128, 128, 0, s>>>(n_cand, js, n_items, J, choices, w, masks);
    return cudaGetLastError();
}

cudaError_t launch_dp_candidates(int J, const int* valid, int* js, int* n_cand, cudaStream_t s) {
    dp_candidates_kernel<<<1, 32, 0, s>>>(J, valid, js, n_cand);
    return cudaGetLastError();
}

}  // namespace ks
