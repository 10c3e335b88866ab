// Sampling-mode speculative decoding on the device (Sec. 2.1, sampling
// branch; nucleus sampling of the Sec. 4 experiments).
//
// filter_kernel: per row of logits, the distribution a token is drawn from:
// logits / T, the top_k largest (ties: lower id first), softmax over them,
// then the shortest prefix in descending probability whose cumulative
// probability reaches top_p, renormalised.  One CTA per row:
//   1. the exact k-th largest logit by a radix select over order-preserving
//      32-bit keys (four 8-bit passes, histograms in shared memory);
//   2. the candidates: every key above it, then the keys equal to it in id
//      order (a block scan over contiguous id ranges) until k are taken;
//   3. ranks by (key desc, id asc), softmax, top-p and renormalisation by one
//      thread in support order (at most 64 terms), so the arithmetic has one
//      fixed order.
// In a draft pass the same kernel draws the draft token with its uniform and
// keeps the support as the draft distribution q of that position.
//
// spec_accept_kernel: the acceptance of Sec. 2.1 over the drafts in order:
// draft t is accepted when u <= min(1, p_t(x) / q_t(x)); at the first
// rejection the token is drawn from norm(max(0, p_t - q_t)) over p_t's
// support (from p_t if that has no mass); after gamma acceptances one more
// token is drawn from p_gamma.
//
// Uniforms: Philox4x64 with 10 rounds (Salmon, Moraes, Dror, Shaw, SC 2011),
// key (seed, 0), counter (step, row, purpose, 0); u = the top 24 bits of the
// first output word / 2^24.  Purposes: 0 draft sample of position t, 1
// acceptance test of draft t, 2 the step's residual or bonus sample.
#include "common.cuh"
#include "internal.h"

#include <cfloat>

namespace ks {

namespace {

constexpr unsigned long long kPhiloxM0 = 0xD2E7470EE14C6C93ull;
constexpr unsigned long long kPhiloxM1 = 0xCA5A826395121157ull;
constexpr unsigned long long kPhiloxW0 = 0x9E3779B97F4A7C15ull;
constexpr unsigned long long kPhiloxW1 = 0xBB67AE8584CAA73Bull;
constexpr int kFilterThreads = 512;

KS_DEV unsigned long long philox_word0(unsigned long long c0, unsigned long long c1, unsigned long long c2,
                                       unsigned long long c3, unsigned long long k0, unsigned long long k1) {
#pragma unroll
    for (int r = 0; r < 10; ++r) {
        if (r) {
            k0 += kPhiloxW0;
            k1 += kPhiloxW1;
        }
        const unsigned long long hi0 = __umul64hi(kPhiloxM0, c0), lo0 = kPhiloxM0 * c0;
        const unsigned long long hi1 = __umul64hi(kPhiloxM1, c2), lo1 = kPhiloxM1 * c2;
        const unsigned long long n0 = hi1 ^ c1 ^ k0, n2 = hi0 ^ c3 ^ k1;
        c0 = n0;
        c1 = lo1;
        c2 = n2;
        c3 = lo0;
    }
    return c0;
}

KS_DEV float uniform(unsigned long long seed, unsigned long long step, int row, int purpose) {
    const unsigned long long x = philox_word0(step, (unsigned long long)row, (unsigned long long)purpose, 0ull,
                                              seed, 0ull);
    return (float)(unsigned)(x >> 40) * (1.0f / 16777216.0f);
}

// larger float -> larger key (no NaNs in logits)
KS_DEV unsigned order_key(float v) {
    const unsigned b = __float_as_uint(v);
    return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

KS_DEV float prob_in(const int* ids, const float* probs, int n, int tok) {
    for (int j = 0; j < n; ++j)
        if (ids[j] == tok) return probs[j];
    return 0.f;
}

// inverse CDF over an ordered support: the first entry whose cumulative
// probability exceeds u (the last one if rounding leaves u above the total)
KS_DEV int draw(const int* ids, const float* probs, int n, float u) {
    float c = 0.f;
    for (int j = 0; j < n; ++j) {
        c += probs[j];
        if (u < c) return ids[j];
    }
    return ids[n - 1];
}

__global__ void __launch_bounds__(kFilterThreads) filter_kernel(const FilterArgs a) {
    const int row = blockIdx.x;
    const float* l = a.logits + (size_t)row * a.ld;
    const int V = a.vocab, tid = threadIdx.x;
    const int K = min(a.top_k, min(V, kSampleMaxK));
    __shared__ unsigned hist[256];
    __shared__ unsigned s_prefix, s_mask;
    __shared__ int s_remaining, s_nc;
    __shared__ int c_id[kSampleMaxK];
    __shared__ unsigned c_key[kSampleMaxK];
    __shared__ int o_id[kSampleMaxK];
    __shared__ float o_pr[kSampleMaxK];
    __shared__ int scan[kFilterThreads];
    if (tid == 0) {
        s_prefix = 0u;
        s_mask = 0u;
        s_remaining = K;
        s_nc = 0;
    }
    // 1. k-th largest key, 8 bits at a time from the top
    for (int shift = 24; shift >= 0; shift -= 8) {
        for (int i = tid; i < 256; i += kFilterThreads) hist[i] = 0u;
        __syncthreads();
        const unsigned prefix = s_prefix, mask = s_mask;
        for (int i = tid; i < V; i += kFilterThreads) {
            const unsigned key = order_key(l[i]);
            if ((key & mask) == prefix) atomicAdd(&hist[(key >> shift) & 255u], 1u);
        }
        __syncthreads();
        if (tid == 0) {
            int rem = s_remaining;
            unsigned above = 0u;
            for (int dgt = 255; dgt >= 0; --dgt) {
                if (above + hist[dgt] >= (unsigned)rem) {
                    s_remaining = rem - (int)above;
                    s_prefix = prefix | ((unsigned)dgt << shift);
                    s_mask = mask | (255u << shift);
                    break;
                }
                above += hist[dgt];
            }
        }
        __syncthreads();
    }
    const unsigned thr = s_prefix;     // the k-th largest key
    const int n_eq = s_remaining;      // how many keys equal to it are taken
    // 2a. keys above the threshold (fewer than K): any order, sorted below
    for (int i = tid; i < V; i += kFilterThreads) {
        const unsigned key = order_key(l[i]);
        if (key > thr) {
            const int slot = atomicAdd(&s_nc, 1);
            c_id[slot] = i;
            c_key[slot] = key;
        }
    }
    __syncthreads();
    const int n_above = s_nc;
    // 2b. keys equal to the threshold, lowest ids first: contiguous id ranges
    // per thread, an exclusive scan of their counts gives each its slots
    const int chunk = (V + kFilterThreads - 1) / kFilterThreads;
    const int lo = tid * chunk, hi = min(V, lo + chunk);
    int cnt = 0;
    for (int i = lo; i < hi; ++i) cnt += order_key(l[i]) == thr;
    scan[tid] = cnt;
    __syncthreads();
    if (tid == 0) {
        int run = 0;
        for (int j = 0; j < kFilterThreads; ++j) {
            const int v = scan[j];
            scan[j] = run;
            run += v;
        }
    }
    __syncthreads();
    int slot = scan[tid];
    for (int i = lo; i < hi && slot < n_eq; ++i)
        if (order_key(l[i]) == thr) {
            c_id[n_above + slot] = i;
            c_key[n_above + slot] = thr;
            ++slot;
        }
    __syncthreads();
    // 3. rank by (key desc, id asc)
    if (tid < K) {
        const unsigned kj = c_key[tid];
        const int ij = c_id[tid];
        int rank = 0;
        for (int i = 0; i < K; ++i) rank += (c_key[i] > kj) || (c_key[i] == kj && c_id[i] < ij);
        o_id[rank] = ij;
    }
    __syncthreads();
    if (tid == 0) {
        // softmax of l / T over the k candidates, then top-p, in support order
        const float m = l[o_id[0]] * a.inv_t;
        float s = 0.f;
        for (int j = 0; j < K; ++j) {
            o_pr[j] = expf(l[o_id[j]] * a.inv_t - m);
            s += o_pr[j];
        }
        int keep = K;
        float c = 0.f;
        for (int j = 0; j < K; ++j) {
            o_pr[j] = o_pr[j] / s;
            c += o_pr[j];
            if (c >= a.top_p) {
                keep = j + 1;
                break;
            }
        }
        float s2 = 0.f;
        for (int j = 0; j < keep; ++j) s2 += o_pr[j];
        int* ids = a.ids + (size_t)(a.slot0 + row) * kSampleMaxK;
        float* pr = a.probs + (size_t)(a.slot0 + row) * kSampleMaxK;
        for (int j = 0; j < keep; ++j) {
            ids[j] = o_id[j];
            pr[j] = o_pr[j] / s2;
        }
        a.n[a.slot0 + row] = keep;
        if (a.token_out) *a.token_out = draw(ids, pr, keep, uniform(a.seed, a.step, a.slot0 + row, 0));
    }
}

__global__ void spec_accept_kernel(const AcceptSampleArgs a) {
    if (threadIdx.x != 0) return;
    const int g = a.gamma;
    const float u_last = uniform(a.seed, a.step, 0, 2);
    int acc = g, rep = -1;
    for (int t = 0; t < g; ++t) {
        const int* pi = a.p_ids + (size_t)t * kSampleMaxK;
        const float* pp = a.p_probs + (size_t)t * kSampleMaxK;
        const int* qi = a.q_ids + (size_t)t * kSampleMaxK;
        const float* qp = a.q_probs + (size_t)t * kSampleMaxK;
        const int pn = a.p_n[t], qn = a.q_n[t];
        const int x = a.rows[1 + t];
        const float px = prob_in(pi, pp, pn, x), qx = prob_in(qi, qp, qn, x);
        if (qx > 0.f && uniform(a.seed, a.step, t, 1) <= fminf(1.f, px / qx)) continue;
        // rejected: draw from norm(max(0, p - q)) over p's support, else from p
        float r[kSampleMaxK];
        float s = 0.f;
        for (int j = 0; j < pn; ++j) {
            r[j] = fmaxf(0.f, pp[j] - prob_in(qi, qp, qn, pi[j]));
            s += r[j];
        }
        if (s > 0.f) {
            for (int j = 0; j < pn; ++j) r[j] = r[j] / s;
            rep = draw(pi, r, pn, u_last);
        } else {
            rep = draw(pi, pp, pn, u_last);
        }
        acc = t;
        break;
    }
    if (rep < 0) {
        rep = draw(a.p_ids + (size_t)g * kSampleMaxK, a.p_probs + (size_t)g * kSampleMaxK, a.p_n[g], u_last);
    }
    a.result[0] = acc;
    a.result[1] = g;
    for (int i = 0; i < acc; ++i) a.result[2 + i] = a.rows[1 + i];
    a.result[2 + acc] = rep;
    a.rows[0] = rep;
}

}  // namespace

cudaError_t launch_filter(const FilterArgs& a, int rows, cudaStream_t s) {
    if (rows < 1 || a.top_k < 1 || !(a.inv_t > 0.f) || !(a.top_p > 0.f) || a.vocab < 1)
        return cudaErrorInvalidValue;
    filter_kernel<<<rows, kFilterThreads, 0, s>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_spec_accept(const AcceptSampleArgs& a, cudaStream_t s) {
    if (a.gamma < 0) return cudaErrorInvalidValue;
    spec_accept_kernel<<<1, 32, 0, s>>>(a);
    return cudaGetLastError();
}

}  // namespace ks
