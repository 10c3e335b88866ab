// a4 and a5 of the hot path: history cosines and knapsack mask selection.
//
// ks_cosine  - Sec. 2's matrix cosine, one CTA per pair; each warp takes rows
//              in turn, the row terms are summed in row order by one thread.
// ks_select_mask - Sec. 3.4 integer weight normalisation (App. C latency
//              model) and the exact 0/1 knapsack of Sec. 3.3 over the 2L
//              sublayers: items processed in order 1..2L, all capacities of
//              an item in parallel across the CTA, int64 fixed-point values,
//              an item taken only on strict improvement, then a backtrack
//              from item 2L that returns the optimal mask with the smallest
//              bitmask value.  One CTA: the table is 2L x (B + 1) with B a few
//              hundred units, so the solve is a few microseconds.
#include "../../include/knapspec.h"
#include "common.cuh"
#include "internal.h"

#include <cmath>

namespace ks {

constexpr int kCosThreads = 256;

template <typename T>
__global__ void __launch_bounds__(kCosThreads) cosine_kernel(const T* X, const T* Y, int rows, int d,
                                                             int64_t pair_stride, const int32_t* row_index,
                                                             float* out) {
    extern __shared__ float rowcos[];
    const int p = blockIdx.x;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const T* Xp = X + (size_t)p * pair_stride;
    const T* Yp = Y + (size_t)p * pair_stride;
    for (int i = warp; i < rows; i += kCosThreads / 32) {
        const int64_t ri = row_index ? row_index[i] : i;
        const T* x = Xp + ri * d;
        const T* y = Yp + ri * d;
        float xy = 0.f, xx = 0.f, yy = 0.f;
        for (int k = lane; k < d; k += 32) {
            const float a = to_float(x[k]), b = to_float(y[k]);
            xy = fmaf(a, b, xy);
            xx = fmaf(a, a, xx);
            yy = fmaf(b, b, yy);
        }
        xy = warp_sum(xy);
        xx = warp_sum(xx);
        yy = warp_sum(yy);
        if (lane == 0) rowcos[i] = xy / (sqrtf(xx) * sqrtf(yy));
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        float s = 0.f;
        for (int i = 0; i < rows; ++i) s += rowcos[i];
        out[p] = s / (float)rows;
    }
}

cudaError_t launch_cosine(const void* X, const void* Y, int dtype, int64_t n_pairs, int rows, int d,
                          int64_t pair_stride, const int32_t* row_index, float* out, cudaStream_t s) {
    const size_t smem = sizeof(float) * (size_t)rows;
    if (smem > 48 * 1024) return cudaErrorInvalidValue;
    if (dtype == KS_DTYPE_BF16)
        cosine_kernel<__nv_bfloat16><<<(unsigned)n_pairs, kCosThreads, smem, s>>>(
            reinterpret_cast<const __nv_bfloat16*>(X), reinterpret_cast<const __nv_bfloat16*>(Y), rows, d,
            pair_stride, row_index, out);
    else
        cosine_kernel<float><<<(unsigned)n_pairs, kCosThreads, smem, s>>>(
            reinterpret_cast<const float*>(X), reinterpret_cast<const float*>(Y), rows, d, pair_stride,
            row_index, out);
    return cudaGetLastError();
}

// ----------------------------------------------------------------- knapsack
constexpr int kMaxItems = 256;
constexpr int kMaxTpt = 128;   // ks_select_tpt passes at most KS_TPT_MAX_CANDIDATES; the DP stage more
constexpr int kKnapThreads = 512;

struct KnapArgs {
    int kind;                 // 0 latency model, 1 explicit units
    double c1, c2, c3;
    long long n;              // context length
    int n_items;
    int budget;               // used when budget_frac < 0
    double budget_frac;       // >= 0: budget = floor(frac * sum w)
    int units[kMaxItems];
    const float* sims;
    uint8_t* mask;
    double* objective;
    int32_t* weights_out;
    int32_t* budget_out;      // optional: the budget used
    long long* best;          // scratch [2][cap + 1]
    uint8_t* take;            // scratch [n_items][cap + 1]
    int cap;                  // capacity of the scratch tables
    int n_frontier;           // > 0: also backtrack the optima of budgets floor(sum w (j + 1) / n_frontier)
    uint8_t* frontier;        // [n_frontier][n_items] masks of those budgets
};

__global__ void __launch_bounds__(kKnapThreads) knapsack_kernel(const KnapArgs a) {
    __shared__ int w[kMaxItems];
    __shared__ long long q[kMaxItems];
    __shared__ int B;
    __shared__ long long SW;
    const int tid = threadIdx.x;
    const int N = a.n_items;
    if (tid == 0) {
        int wa = 1, wm = 1;
        if (a.kind == 0) {
            // Sec. 3.4: Delta = min(t_Attn(n), t_MLP), w = round(t / Delta), >= 1
            // explicit _rn intrinsics: no FMA contraction, the same two
            // roundings as c2 * n + c3 evaluated left to right
            const double ta = __dadd_rn(__dmul_rn(a.c2, (double)a.n), a.c3);
            const double tm = a.c1;
            const double delta = fmin(ta, tm);
            wa = (int)llround(__ddiv_rn(ta, delta));
            wm = (int)llround(__ddiv_rn(tm, delta));
            if (wa < 1) wa = 1;
            if (wm < 1) wm = 1;
        }
        long long sum = 0;
        for (int i = 0; i < N; ++i) {
            // 0-based item i is sublayer i + 1: even i -> Attn, odd i -> MLP
            w[i] = (a.kind == 0) ? ((i % 2 == 0) ? wa : wm) : a.units[i];
            sum += w[i];
        }
        SW = sum;
        long long b = a.budget;
        if (a.budget_frac >= 0.0) b = (long long)floor(__dmul_rn(a.budget_frac, (double)sum));
        if (b > a.cap) b = a.cap;
        if (b < 0) b = 0;
        B = (int)b;
        if (a.budget_out) *a.budget_out = (int)b;
    }
    for (int i = tid; i < N; i += blockDim.x) {
        // q_i = round((1 - sigma_i) * 2^30), half away from zero, in double
        const double v = __dmul_rn(__dsub_rn(1.0, (double)a.sims[i]), 1073741824.0);
        q[i] = llround(v);
    }
    __syncthreads();
    const int cap1 = B + 1;
    long long* cur = a.best;
    long long* nxt = a.best + (a.cap + 1);
    for (int c = tid; c < cap1; c += blockDim.x) cur[c] = 0;
    __syncthreads();
    for (int i = 0; i < N; ++i) {
        const int wi = w[i];
        const long long qi = q[i];
        uint8_t* tk = a.take + (size_t)i * (a.cap + 1);
        for (int c = tid; c < cap1; c += blockDim.x) {
            long long v = cur[c];
            uint8_t t = 0;
            if (c >= wi) {
                const long long cand = cur[c - wi] + qi;
                if (cand > v) {
                    v = cand;
                    t = 1;
                }
            }
            nxt[c] = v;
            tk[c] = t;
        }
        __syncthreads();
        long long* tmp = cur;
        cur = nxt;
        nxt = tmp;
    }
    if (tid == 0) {
        int c = B;
        for (int i = N - 1; i >= 0; --i) {
            const uint8_t t = a.take[(size_t)i * (a.cap + 1) + c];
            a.mask[i] = t;
            if (t) c -= w[i];
        }
        if (a.objective) *a.objective = (double)cur[B] / 1073741824.0;
    }
    // The TPT stage's candidate set: the optimum of each frontier budget,
    // backtracked from the same table (the DP up to capacity c does not
    // depend on larger capacities).
    for (int j = tid; j < a.n_frontier; j += blockDim.x) {
        int c = (int)((SW * (long long)(j + 1)) / a.n_frontier);
        if (c > B) c = B;
        uint8_t* fm = a.frontier + (size_t)j * N;
        for (int i = N - 1; i >= 0; --i) {
            const uint8_t t = a.take[(size_t)i * (a.cap + 1) + c];
            fm[i] = t;
            if (t) c -= w[i];
        }
    }
    if (a.weights_out)
        for (int i = tid; i < N; i += blockDim.x) a.weights_out[i] = w[i];
}

size_t select_scratch_bytes(int n_items, int cap) {
    const size_t best = sizeof(long long) * 2 * ((size_t)cap + 1);
    const size_t take = (size_t)n_items * ((size_t)cap + 1);
    return ((best + take + 255) / 256) * 256;
}

cudaError_t launch_select(const ks_latency* lat, const float* sims, int64_t n, int n_items, int budget,
                          double budget_frac, uint8_t* mask, double* objective, int32_t* weights,
                          int32_t* budget_out, void* scratch, int cap, cudaStream_t s, int n_frontier,
                          uint8_t* frontier) {
    KnapArgs a{};
    a.kind = lat->kind;
    a.c1 = lat->c1;
    a.c2 = lat->c2;
    a.c3 = lat->c3;
    a.n = n;
    a.n_items = n_items;
    a.budget = budget;
    a.budget_frac = budget_frac;
    if (lat->kind == 1)
        for (int i = 0; i < n_items; ++i) a.units[i] = lat->units[i];
    a.sims = sims;
    a.mask = mask;
    a.objective = objective;
    a.weights_out = weights;
    a.budget_out = budget_out;
    a.cap = cap;
    a.best = reinterpret_cast<long long*>(scratch);
    a.take = reinterpret_cast<uint8_t*>(scratch) + sizeof(long long) * 2 * ((size_t)cap + 1);
    a.n_frontier = n_frontier;
    a.frontier = frontier;
    knapsack_kernel<<<1, kKnapThreads, 0, s>>>(a);
    return cudaGetLastError();
}

// ---------------------------------------------------------------- TPT stage
// Alg. 2 after the frontier: Eq. 4's acceptance of each candidate on the
// history rows (its predicted tokens against the full layer set's), then the
// grid search of Eq. 3 over candidates (in order) x gamma = 1..D, a pair
// replacing the best only when its TPT is strictly larger.  Double
// arithmetic with explicit round-to-nearest operations in a fixed order.
struct TptArgs {
    int kind;                 // 0 latency model, 1 explicit units
    double c1, c2, c3;
    long long n;
    int units[kMaxItems];
    int n_items, n_layers;
    int K, r, D;
    const uint8_t* frontier;  // [K][n_items]
    const int32_t* tokens;    // [(K + 1) r]: candidate j's rows at j r, the full set's at K r
    uint8_t* mask_out;        // [n_items] the chosen candidate
    int32_t* info;            // [0] chosen candidate, [1] gamma
    double* out;              // [0] TPT, [1 + j] alpha of candidate j
};

__global__ void __launch_bounds__(256) tpt_kernel(const TptArgs a) {
    __shared__ double alpha[kMaxTpt];
    __shared__ int sel;
    const int tid = threadIdx.x;
    for (int j = tid; j < a.K; j += blockDim.x) {
        int cnt = 0;
        for (int i = 0; i < a.r; ++i) cnt += a.tokens[(size_t)j * a.r + i] == a.tokens[(size_t)a.K * a.r + i];
        alpha[j] = __ddiv_rn((double)cnt, (double)a.r);
        a.out[1 + j] = alpha[j];
    }
    __syncthreads();
    if (tid == 0) {
        double ta = 0.0, tm = 0.0, tt = 0.0;
        if (a.kind == 0) {
            ta = __dadd_rn(__dmul_rn(a.c2, (double)a.n), a.c3);
            tm = a.c1;
            tt = __dmul_rn((double)a.n_layers, __dadd_rn(ta, tm));
        } else {
            for (int i = 0; i < a.n_items; ++i) tt = __dadd_rn(tt, (double)a.units[i]);
        }
        int bj = -1, bg = 0;
        double bv = 0.0;
        for (int j = 0; j < a.K; ++j) {
            const uint8_t* m = a.frontier + (size_t)j * a.n_items;
            double td = 0.0;
            if (a.kind == 0) {
                int na = 0, nm = 0;
                for (int i = 0; i < a.n_items; ++i)
                    if (m[i]) (i % 2 == 0 ? na : nm)++;
                td = __dadd_rn(__dmul_rn((double)na, ta), __dmul_rn((double)nm, tm));
            } else {
                for (int i = 0; i < a.n_items; ++i)
                    if (m[i]) td = __dadd_rn(td, (double)a.units[i]);
            }
            double e = 1.0, p = 1.0;
            for (int g = 1; g <= a.D; ++g) {
                p = __dmul_rn(p, alpha[j]);
                e = __dadd_rn(e, p);   // Eq. 1 summed term by term
                const double v = __ddiv_rn(e, __dadd_rn(__dmul_rn((double)g, td), tt));
                if (v > bv) {
                    bv = v;
                    bj = j;
                    bg = g;
                }
            }
        }
        a.info[0] = bj;
        a.info[1] = bg;
        a.out[0] = bv;
        sel = bj;
    }
    __syncthreads();
    for (int i = tid; i < a.n_items; i += blockDim.x) a.mask_out[i] = a.frontier[(size_t)sel * a.n_items + i];
}

cudaError_t launch_tpt(const ks_latency* lat, int64_t n, int n_items, int n_layers, int K, int r, int D,
                       const uint8_t* frontier, const int32_t* tokens, uint8_t* mask_out, int32_t* info,
                       double* out, cudaStream_t s) {
    if (K < 1 || K > kMaxTpt || r < 1 || D < 1 || n_items > kMaxItems) return cudaErrorInvalidValue;
    TptArgs a{};
    a.kind = lat->kind;
    a.c1 = lat->c1;
    a.c2 = lat->c2;
    a.c3 = lat->c3;
    a.n = n;
    if (lat->kind == 1)
        for (int i = 0; i < n_items; ++i) a.units[i] = lat->units[i];
    a.n_items = n_items;
    a.n_layers = n_layers;
    a.K = K;
    a.r = r;
    a.D = D;
    a.frontier = frontier;
    a.tokens = tokens;
    a.mask_out = mask_out;
    a.info = info;
    a.out = out;
    tpt_kernel<<<1, 256, 0, s>>>(a);
    return cudaGetLastError();
}

}  // namespace ks

// Sec. 3.4 / App. C: the integer weights are round(t / Delta) with Delta =
// min(t_Attn(n), t_MLP), t_Attn(n) = c2 n + c3, t_MLP = c1.  Both times must
// be positive, and the larger may be at most 65535 times the smaller (the
// limit of explicit units), or the quotient would not be a valid weight.
bool ks::latency_valid(const ks_latency* lat, int32_t n_sublayers, int64_t context_len) {
    if (!lat) return false;
    if (lat->kind == 0) {
        if (!(lat->c1 > 0.0) || !(lat->c2 >= 0.0) || !(lat->c3 >= 0.0) || !std::isfinite(lat->c1) ||
            !std::isfinite(lat->c2) || !std::isfinite(lat->c3) || context_len < 0)
            return false;
        const double ta = lat->c2 * (double)context_len + lat->c3;
        if (!(ta > 0.0) || !std::isfinite(ta)) return false;
        const double hi = std::fmax(ta, lat->c1), lo = std::fmin(ta, lat->c1);
        return hi / lo <= 65535.0;
    }
    if (lat->kind == 1) {
        if (!lat->units) return false;
        for (int i = 0; i < n_sublayers; ++i)
            if (lat->units[i] < 1 || lat->units[i] > 65535) return false;
        return true;
    }
    return false;
}

namespace ks {

// ------------------------------------------------ allocation-free variant
// Work tables of ks_select_mask_static: one array for the whole process on
// every device that loads the library, sized for KS_SELECT_STATIC_MAX_BUDGET
// units and kMaxItems sublayers (about 1.1 MB).  Host code may not use the
// symbol as an address; the device address comes from cudaGetSymbolAddress.
constexpr int kStaticCap = KS_SELECT_STATIC_MAX_BUDGET;
constexpr size_t kStaticScratchBytes =
    ((sizeof(long long) * 2 * ((size_t)kStaticCap + 1) + (size_t)kMaxItems * ((size_t)kStaticCap + 1)) + 255) / 256 *
    256;
static __device__ __align__(256) unsigned char g_select_scratch[kStaticScratchBytes];

// Device address of g_select_scratch on the current device.  Looked up on
// every call (cheap once the module is loaded), so a new primary context
// after cudaDeviceReset gets the address of its own copy of the array.
static cudaError_t static_scratch(void** out) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_select_scratch);
    if (e != cudaSuccess) return e;
    *out = p;
    return cudaSuccess;
}

}  // namespace ks

// ------------------------------------------------------------------- C ABI
using namespace ks;

extern "C" ks_status ks_select_mask_static(const ks_latency* lat, const float* sims, int64_t context_len,
                                           int32_t n_sublayers, int32_t budget_units, uint8_t* mask_out,
                                           double* objective_out, int32_t* weights_out, void* stream) {
    if (!sims || !mask_out) {
        set_error("ks_select_mask_static: null pointer");
        return KS_ERR_INVALID_ARG;
    }
    if (n_sublayers < 2 || n_sublayers > kMaxItems || (n_sublayers & 1) || context_len < 0) {
        set_error("ks_select_mask_static: bad n_sublayers / context_len");
        return KS_ERR_INVALID_ARG;
    }
    if (budget_units < 0 || budget_units > kStaticCap) {
        set_error("ks_select_mask_static: budget_units %d outside 0..%d (the size of the built-in tables)",
                  budget_units, kStaticCap);
        return KS_ERR_INVALID_ARG;
    }
    if (!latency_valid(lat, n_sublayers, context_len)) {
        set_error("ks_select_mask_static: bad latency model (times must be positive, ratio at most 65535)");
        return KS_ERR_INVALID_ARG;
    }
    void* scratch = nullptr;
    cudaError_t e = static_scratch(&scratch);
    if (e != cudaSuccess) {
        set_error("ks_select_mask_static: cudaGetSymbolAddress: %s", cudaGetErrorString(e));
        return KS_ERR_CUDA;
    }
    e = launch_select(lat, sims, context_len, n_sublayers, budget_units, -1.0, mask_out, objective_out, weights_out,
                      nullptr, scratch, budget_units, reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) {
        set_error("ks_select_mask_static: %s", cudaGetErrorString(e));
        return KS_ERR_CUDA;
    }
    return KS_OK;
}

extern "C" ks_status ks_cosine(const void* X, const void* Y, int32_t dtype, int64_t n_pairs, int32_t rows,
                               int32_t d, int64_t pair_stride, const int32_t* row_index, float* out,
                               void* stream) {
    if (!X || !Y || !out) {
        set_error("ks_cosine: null pointer");
        return KS_ERR_INVALID_ARG;
    }
    if (n_pairs < 1 || n_pairs > (1 << 30) || rows < 1 || rows > 8192 || d < 1 || pair_stride < 0 ||
        (dtype != KS_DTYPE_F32 && dtype != KS_DTYPE_BF16)) {
        set_error("ks_cosine: bad size or dtype");
        return KS_ERR_INVALID_ARG;
    }
    cudaError_t e = launch_cosine(X, Y, dtype, n_pairs, rows, d, pair_stride, row_index, out,
                                  reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) {
        set_error("ks_cosine: %s", cudaGetErrorString(e));
        return KS_ERR_CUDA;
    }
    return KS_OK;
}

extern "C" ks_status ks_fit_latency(const double* n, const double* t_attn, int32_t count, const double* t_mlp,
                                    int32_t count_mlp, ks_latency* out) {
    if (!n || !t_attn || !t_mlp || !out || count < 2 || count_mlp < 1) {
        set_error("ks_fit_latency: need at least two attention points and one MLP time");
        return KS_ERR_INVALID_ARG;
    }
    // App. C: t_Attn(n) = c2 n + c3 by least squares, t_MLP = c1 (the mean)
    double sn = 0.0, st = 0.0, c1 = 0.0;
    for (int k = 0; k < count; ++k) {
        if (!std::isfinite(n[k]) || !std::isfinite(t_attn[k]) || n[k] < 0.0) {
            set_error("ks_fit_latency: bad sample %d", k);
            return KS_ERR_INVALID_ARG;
        }
        sn += n[k];
        st += t_attn[k];
    }
    for (int k = 0; k < count_mlp; ++k) c1 += t_mlp[k];
    c1 /= count_mlp;
    const double nb = sn / count, tb = st / count;
    double sxx = 0.0, sxy = 0.0;
    for (int k = 0; k < count; ++k) {
        sxx += (n[k] - nb) * (n[k] - nb);
        sxy += (n[k] - nb) * (t_attn[k] - tb);
    }
    if (!(sxx > 0.0)) {
        set_error("ks_fit_latency: the context lengths must not all be equal");
        return KS_ERR_INVALID_ARG;
    }
    double c2 = sxy / sxx, c3 = tb - c2 * nb;
    // the model's coefficients are non-negative: a negative intercept refits
    // through the origin, a negative slope leaves the mean as the intercept
    if (c3 < 0.0) {
        double snn = 0.0, snt = 0.0;
        for (int k = 0; k < count; ++k) {
            snn += n[k] * n[k];
            snt += n[k] * t_attn[k];
        }
        c2 = snt / snn;
        c3 = 0.0;
    }
    if (c2 < 0.0) {
        c2 = 0.0;
        c3 = tb;
    }
    if (!(c1 > 0.0) || !std::isfinite(c1) || !std::isfinite(c2) || !std::isfinite(c3)) {
        set_error("ks_fit_latency: the fitted model is not valid (t_MLP must be positive)");
        return KS_ERR_INVALID_ARG;
    }
    out->kind = 0;
    out->c1 = c1;
    out->c2 = c2;
    out->c3 = c3;
    out->units = nullptr;
    return KS_OK;
}

extern "C" size_t ks_select_scratch_bytes(int32_t n_sublayers, int32_t budget_units) {
    if (n_sublayers < 2 || n_sublayers > kMaxItems || budget_units < 0 || budget_units > 65535) return 0;
    return select_scratch_bytes(n_sublayers, budget_units);
}


extern "C" ks_status ks_select_mask(const ks_latency* lat, const float* sims, int64_t context_len,
                                    int32_t n_sublayers, int32_t budget_units, uint8_t* mask_out,
                                    double* objective_out, int32_t* weights_out, void* scratch,
                                    size_t scratch_bytes, void* stream) {
    if (!sims || !mask_out || !scratch) {
        set_error("ks_select_mask: null pointer");
        return KS_ERR_INVALID_ARG;
    }
    if (n_sublayers < 2 || n_sublayers > kMaxItems || (n_sublayers & 1) || budget_units < 0 ||
        budget_units > 65535 || context_len < 0) {
        set_error("ks_select_mask: bad n_sublayers / budget / context_len");
        return KS_ERR_INVALID_ARG;
    }
    if (!latency_valid(lat, n_sublayers, context_len)) {
        set_error("ks_select_mask: bad latency model (times must be positive, ratio at most 65535)");
        return KS_ERR_INVALID_ARG;
    }
    if ((reinterpret_cast<uintptr_t>(scratch) & 15) != 0) {
        set_error("ks_select_mask: scratch must be 16-byte aligned");
        return KS_ERR_INVALID_ARG;
    }
    if (scratch_bytes < select_scratch_bytes(n_sublayers, budget_units)) {
        set_error("ks_select_mask: scratch too small");
        return KS_ERR_WORKSPACE;
    }
    cudaError_t e = launch_select(lat, sims, context_len, n_sublayers, budget_units, -1.0, mask_out,
                                  objective_out, weights_out, nullptr, scratch, budget_units,
                                  reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) {
        set_error("ks_select_mask: %s", cudaGetErrorString(e));
        return KS_ERR_CUDA;
    }
    return KS_OK;
}
