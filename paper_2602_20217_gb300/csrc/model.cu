// Model runtime and C ABI of libknapspec: workspace layout, the skip-masked
// forward pass (Sec. 2), draft (a1), verify + greedy acceptance (a2, a3,
// Sec. 2.1), the history ring (Sec. 3.4), and the speculative loop that
// re-selects the draft mask with the knapsack (a4, a5).
//
// All device memory is the caller's workspace; this file carves it up.  The
// host loop launches one kernel per matrix product (5 per layer plus the
// attention split/merge pair) on the caller's stream; draft tokens stay on
// the device between steps and one stream synchronisation per verify step
// returns the accepted tokens.
#include "../../include/knapspec.h"
#include "common.cuh"
#include "internal.h"

#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <algorithm>
#include <cstring>
#include <vector>

namespace ks {

static thread_local char g_err[512] = "";

void set_error(const char* fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, sizeof(g_err), fmt, ap);
    va_end(ap);
}


constexpr int kSelectCap = 65535;
constexpr int kKlasses = 11;
enum { K_QKV = 0, K_ATTN, K_MERGE, K_OPROJ, K_GATEUP, K_DOWN, K_LMHEAD, K_EMBED, K_ACCEPT, K_CHAIN, K_PREP };

// ------------------------------------------------------------ small kernels
// x[r] = embed[tok[r]] (fp32); optionally copied to the history plane 0.
// Block (r, b) covers features [256 b, 256 b + 256) of row r; it also writes
// the bf16 x * gain input of the next projection and the 16-feature sums of
// squares ss[q][r] that its RMSNorm uses.
template <typename WT>
__global__ void __launch_bounds__(256) embed_kernel(const WT* embed, const int32_t* tok, int d, int vocab, float* x,
                                                    float* capture, float* ss, __nv_bfloat16* xg,
                                                    const WT* next_gain, const int* stop) {
    if (stop && *stop) return;   // a draft pass after the dynamic exit
    const int r = blockIdx.x;
    const int k = blockIdx.y * 256 + threadIdx.x;
    int t = tok[r];
    if (t < 0 || t >= vocab) t = 0;
    float v = 0.f;
    if (k < d) {
        v = to_float(embed[(size_t)t * d + k]);
        x[(size_t)r * d + k] = v;
        if (capture) capture[(size_t)r * d + k] = v;
        if (xg) xg[(size_t)r * d + k] = __float2bfloat16_rn(v * to_float(next_gain[k]));
    }
    // lanes 0-15 and 16-31 of each warp form one 16-feature group
    float s = v * v;
#pragma unroll
    for (int o = 8; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    const int lane = threadIdx.x & 31;
    if ((lane & 15) == 0 && k < d) ss[(k / kSsGroup) * 16 + r] = s;
}

// The pass input taken from rows already in x (the hidden-state DP's states):
// the 16-feature sums of squares and, for bf16 models, x * gain in bf16, as
// the embedding kernel leaves them.
template <typename WT>
__global__ void __launch_bounds__(256) rows_prep_kernel(const float* x, int d, float* ss, __nv_bfloat16* xg,
                                                        const WT* gain, const int* stop) {
    if (stop && *stop) return;
    const int r = blockIdx.x;
    const int k = blockIdx.y * 256 + threadIdx.x;
    float v = 0.f;
    if (k < d) {
        v = x[(size_t)r * d + k];
        if (xg) xg[(size_t)r * d + k] = __float2bfloat16_rn(v * to_float(gain[k]));
    }
    float s = v * v;
#pragma unroll
    for (int o = 8; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    const int lane = threadIdx.x & 31;
    if ((lane & 15) == 0 && k < d) ss[(k / kSsGroup) * 16 + r] = s;
}

// Greedy acceptance (Sec. 2.1): drafts = rows[1..gamma], z = target argmax of
// rows[0..gamma].  a = longest prefix with drafts[i] == z[i]; the new tokens
// are drafts[0..a-1] followed by z[a], which becomes the pending rows[0].
// After a dynamic-exit draft only the n_drafted drafts that were produced are
// compared (the pass still scored gamma + 1 rows; the rest are ignored).
// result = {a, drafts compared, tokens[0..a]}.
__global__ void accept_kernel(int32_t* rows, const int32_t* z, int gamma, const int32_t* n_drafted,
                              int32_t* result) {
    if (threadIdx.x != 0) return;
    const int g = n_drafted ? min(gamma, *n_drafted) : gamma;
    int a = 0;
    while (a < g && rows[1 + a] == z[a]) ++a;
    result[0] = a;
    result[1] = g;
    for (int i = 0; i < a; ++i) result[2 + i] = rows[1 + i];
    result[2 + a] = z[a];
    rows[0] = z[a];
}

// Dynamic drafting exit (Sec. 3.5): the confidence of draft pass t's token is
// its softmax probability, 1 / sum_i exp(l_i - l_max), over the pass's logits
// (row 0); l_max is the logit of the argmax token the LM head wrote.  Each of
// kTop1Ctas CTAs sums exp(l_i - l_max) over a fixed slice of the vocabulary
// in a fixed order; the last CTA to finish adds the slices in slice order, so
// the value is the same in every run.  It records the confidence, counts the
// pass as drafted, and raises the stop flag below tau, which makes the later
// draft passes of the step return at once.
constexpr int kTop1Ctas = 64;
constexpr int kTop1Threads = 256;
__global__ void __launch_bounds__(kTop1Threads) top1_kernel(const float* logits, int vocab, const int32_t* token,
                                                            float tau, int t, int* stop, int* n_drafted,
                                                            float* conf, float* part, int* ticket) {
    if (*stop) return;
    __shared__ float red[kTop1Threads / 32 + 1];
    __shared__ int last;
    const float lmax = logits[*token];
    const int per = (vocab + kTop1Ctas - 1) / kTop1Ctas;
    const int lo = blockIdx.x * per, hi = min(vocab, lo + per);
    float s = 0.f;
    for (int i = lo + (int)threadIdx.x; i < hi; i += kTop1Threads) s += expf(logits[i] - lmax);
    s = block_sum<kTop1Threads / 32>(s, red);
    if (threadIdx.x == 0) {
        part[blockIdx.x] = s;
        __threadfence();
        last = atomicAdd(ticket, 1) == kTop1Ctas - 1;
    }
    __syncthreads();
    if (!last || threadIdx.x != 0) return;
    __threadfence();
    float S = 0.f;
    for (int c = 0; c < kTop1Ctas; ++c) S += __ldcg(&part[c]);
    const float p1 = 1.f / S;
    conf[t] = p1;
    *n_drafted = t + 1;
    if (p1 < tau) *stop = 1;
    *ticket = 0;
}

// TPT stage, Eq. 4 inputs: row b of a batch is overall row q = row0 + b, i.e.
// candidate j = q / r (j == K: the full layer set) on history row i = q % r.
// Its draft state is X^(2L) minus X^(s) - X^(s-1) for every sublayer s the
// candidate skips, in order s = 1 .. 2L; written as the LM head's input: the
// fp32 residual, its bf16 x * final gain, and the 16-feature sums of squares.
template <typename WT>
__global__ void __launch_bounds__(256) tpt_states_kernel(const float* hist, long long plane, const int32_t* hidx,
                                                         int r, int row0, int nsub, const uint8_t* masks, int K,
                                                         int d, const WT* gain, float* x, float* ss,
                                                         __nv_bfloat16* xg) {
    const int b = blockIdx.x;
    const int q = row0 + b;
    const int j = q / r, i = q - j * r;
    const uint8_t* mask = (j < K) ? masks + (size_t)j * nsub : nullptr;
    const int k = blockIdx.y * 256 + threadIdx.x;
    float h = 0.f;
    if (k < d) {
        const float* base = hist + (size_t)hidx[i] * d + k;
        h = base[(size_t)nsub * plane];
        if (mask)
            for (int sl = 1; sl <= nsub; ++sl)
                if (!mask[sl - 1]) h -= base[(size_t)sl * plane] - base[(size_t)(sl - 1) * plane];
        x[(size_t)b * d + k] = h;
        if (xg) xg[(size_t)b * d + k] = __float2bfloat16_rn(h * to_float(gain[k]));
    }
    float sq = h * h;   // lanes 0-15 and 16-31 of each warp form one 16-feature group
#pragma unroll
    for (int o = 8; o > 0; o >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, o);
    const int lane = threadIdx.x & 31;
    if ((lane & 15) == 0 && k < d) ss[(k / kSsGroup) * 16 + b] = sq;
}

// ------------------------------------------------------------------ helpers
static size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

struct Layout {
    size_t kv, rope, x, ss, xg, qkv, attn_out, act, attn_part, gemv_part, counters, logits, amax_val,
        amax_idx, tok, hist, hist_snap, hist_idx, sims, mask, obj, wts, select, chain_ctr, best, tpt_masks,
        tpt_tok, tpt_info, tpt_out, dyn, samp, slice, qbuf, total;
    int n_chunks_max;
    size_t gemv_part_floats;
    int counters_n;
    int hist_slots;
};

static bool config_ok(const ks_config* c) {
    if (!c) return false;
    if (c->n_layers < 1 || c->n_layers > 128) return false;
    if (c->d_model < 8 || c->d_model % 8) return false;
    if (c->n_q_heads < 1 || c->n_kv_heads < 1 || c->n_q_heads % c->n_kv_heads) return false;
    if (c->n_q_heads / c->n_kv_heads > 16) return false;
    if (c->head_dim != 64 && c->head_dim != 128) return false;
    if (c->d_ff < 8 || c->d_ff % 8) return false;
    // the chain kernel's per-block counters: at most 64 blocks of a phase's
    // output (512 columns for gate/up inputs, 1024 otherwise)
    if (c->d_model > 64 * 512 || c->d_ff > 64 * 1024) return false;
    if (c->vocab < 1) return false;
    if (c->dtype != KS_DTYPE_F32 && c->dtype != KS_DTYPE_BF16) return false;
    // bf16 attention addresses cache rows with 32-bit TMA coordinates
    if (c->dtype == KS_DTYPE_BF16 && 2.0 * c->n_layers * c->n_kv_heads * (double)c->max_seq > 2147483647.0)
        return false;
    if (c->max_seq < 2 || c->max_rows < 2 || c->max_rows > 16) return false;
    if (c->hist_steps < 1 || c->hist_steps > 64) return false;
    if (c->hist_init_rows < 1 || c->hist_init_rows > c->max_rows) return false;
    if (!(c->rms_eps > 0.f) || !(c->rope_theta > 1.0)) return false;
    return true;
}

static Layout make_layout(const ks_config* c) {
    Layout L{};
    const size_t es = c->dtype == KS_DTYPE_BF16 ? 2 : 4;
    const int d = c->d_model, hd = c->head_dim, R = c->max_rows;
    const int nqkv = (c->n_q_heads + 2 * c->n_kv_heads) * hd;
    const int nsub = 2 * c->n_layers;
    L.n_chunks_max = attn_num_chunks(c->max_seq);
    L.hist_slots = c->hist_steps + 1;
    size_t gp = 0;
    gp = std::max(gp, gemv_partial_floats(nqkv, d, R, EPI_STORE, c->dtype));
    gp = std::max(gp, gemv_partial_floats(d, c->n_q_heads * hd, R, EPI_RESID, c->dtype));
    gp = std::max(gp, gemv_partial_floats(c->d_ff, d, R, EPI_SWIGLU, c->dtype));
    gp = std::max(gp, gemv_partial_floats(d, c->d_ff, R, EPI_RESID, c->dtype));
    gp = std::max(gp, gemv_partial_floats(c->vocab, d, R, EPI_LMHEAD, c->dtype));
    L.gemv_part_floats = gp;
    int gx = gemv_grid_x(c->vocab);
    gx = std::max(gx, gemv_grid_x(nqkv));
    gx = std::max(gx, gemv_grid_x(c->d_ff));
    gx = std::max(gx, gemv_grid_x(d));
    L.counters_n = gx + 2;

    size_t off = 0;
    auto take = [&](size_t bytes) {
        size_t o = off;
        off = align_up(off + bytes, 256);
        return o;
    };
    L.kv = take(2 * (size_t)c->n_layers * c->n_kv_heads * (size_t)c->max_seq * hd * es);
    L.rope = take(sizeof(float) * (size_t)c->max_seq * hd);
    L.x = take(sizeof(float) * (size_t)R * d);
    L.ss = take(sizeof(float) * 16 * (size_t)((d + kSsGroup - 1) / kSsGroup));
    L.xg = take(sizeof(__nv_bfloat16) * (size_t)R * d);
    L.qkv = take(sizeof(float) * (size_t)R * nqkv);
    L.attn_out = take(es * (size_t)R * c->n_q_heads * hd);
    L.act = take(es * (size_t)R * c->d_ff);
    L.attn_part = take(sizeof(float) * (size_t)R * c->n_q_heads * L.n_chunks_max * (hd + 4));
    L.gemv_part = take(sizeof(float) * std::max<size_t>(gp, 1));
    L.counters = take(sizeof(int) * (size_t)L.counters_n);
    L.logits = take(sizeof(float) * (size_t)R * c->vocab);
    L.amax_val = take(sizeof(float) * (size_t)gemv_groups(c->vocab, c->dtype) * 16);
    L.amax_idx = take(sizeof(int) * (size_t)gemv_groups(c->vocab, c->dtype) * 16);
    // tokens: rows[R+1] | target[R] | result[R+3] | err | prompt/out[max_seq]
    L.tok = take(sizeof(int) * ((size_t)3 * R + 8 + c->max_seq));
    L.hist = take(sizeof(float) * (size_t)(nsub + 1) * L.hist_slots * R * d);
    L.hist_snap = take(sizeof(float) * (size_t)(nsub + 1) * R * d);  // the prefill's history entry
    L.hist_idx = take(sizeof(int) * (size_t)L.hist_slots * R);
    L.sims = take(sizeof(float) * nsub);
    L.mask = take(nsub);
    L.obj = take(sizeof(double) * 2);
    L.wts = take(sizeof(int) * (nsub + 2));
    L.select = take(select_scratch_bytes(nsub, kSelectCap));
    // bf16: two sets of chain counters
    L.chain_ctr = take(sizeof(int) * 2 * chain_counter_ints());
    L.best = take(sizeof(unsigned long long) * 16);
    // TPT stage: candidate masks, predicted tokens of every (candidate + full
    // set) x history row, the choice and its figures
    L.tpt_masks = take((size_t)KS_TPT_MAX_CANDIDATES * nsub);
    L.tpt_tok = take(sizeof(int32_t) * (KS_TPT_MAX_CANDIDATES + 1) * (size_t)L.hist_slots * R);
    L.tpt_info = take(sizeof(int32_t) * 4);
    L.tpt_out = take(sizeof(double) * (KS_TPT_MAX_CANDIDATES + 1));
    // dynamic exit: confidence[max_rows] | slice sums[kTop1Ctas] | ticket
    L.dyn = take(sizeof(float) * ((size_t)R + kTop1Ctas) + sizeof(int));
    // sampling: q and p distributions, [R][kSampleMaxK] ids and probs plus [R] sizes each
    L.samp = take(2 * ((size_t)R * kSampleMaxK * (sizeof(int) + sizeof(float)) + sizeof(int) * R));
    // chain kernel K-slices: partial sums [2][640][2][16][16] floats, then tickets [2][640]
    L.slice = take(sizeof(float) * 2 * kChainSliceMaxItems * 512 + sizeof(int) * 2 * kChainSliceMaxItems);
    // bf16 attention: the pass's prepared queries [hk][G R][hd]
    L.qbuf = take(sizeof(__nv_bfloat16) * (size_t)R * c->n_q_heads * hd);
    L.total = off;
    return L;
}

}  // namespace ks

using namespace ks;

struct KlassTiming {
    bool on = false;
    std::vector<cudaEvent_t> ev;  // pairs
    size_t used = 0;
    double bytes = 0.0;           // weight bytes the timed launches had to stream
};

struct ks_model {
    ks_config cfg;
    int dtype;
    size_t es;
    int nsub;
    const void* embed;
    const void* lm_head;
    const void* final_norm;
    std::vector<const void*> attn_norm, w_qkv, w_o, q_norm, k_norm, mlp_norm, w_gate_up, w_down;
    cudaStream_t stream;
    char* ws;
    size_t ws_bytes;
    Layout lay;
    // carved pointers
    char* kv;
    float *rope, *x, *ss, *qkv, *attn_part, *gemv_part, *logits, *amax_val, *hist, *hist_snap, *sims;
    __nv_bfloat16* xg;
    void *attn_out, *act, *select;
    int *counters, *amax_idx, *rows, *target, *result, *err, *seq, *hist_idx;
    uint8_t* mask_dev;
    ChainArgs* chain = nullptr;  // bf16: parameter block of the chain launches (host)
    int* chain_ctr;           // two counter sets, alternating between chain launches
    unsigned long long* best; // LM head argmax keys of the chain kernel
    uint8_t* tpt_masks;       // TPT stage buffers
    int32_t* tpt_tok;
    int32_t* tpt_info;
    double* tpt_out;
    float* conf;              // dynamic exit: confidence of each draft pass of the step
    float* top1_part;         // dynamic exit: slice sums
    int* top1_ticket;
    int* stop;                // dynamic exit: set once a draft token is below tau_conf
    int* n_drafted;           // dynamic exit: draft passes of the step that ran
    float* slice_part;        // chain kernel: K-slice partial sums
    int* slice_ticket;
    __nv_bfloat16* qbuf;      // bf16 attention: prepared queries of the pass
    CUtensorMap map_kv;       // bf16 attention: the KV cache as rows of hd elements
    bool last_dynamic = false;
    bool last_sampled = false;   // the drafts on the device were sampled (ks_draft_sample)
    int *q_ids, *q_n, *p_ids, *p_n;   // sampling mode: draft / target distributions [16][kSampleMaxK]
    float *q_probs, *p_probs;
    int last_scored = 0;      // drafts compared by the last verify
    int chain_parity = 0;
    double* obj_dev;
    int* wts_dev;
    // pinned host staging
    int32_t* h_buf;
    size_t h_buf_ints;
    // decoding state
    bool have_seq = false;
    int p = 0;
    int pending = 0;
    int prompt_len = 0;       // state right after the last prefill, for ks_rewind
    int prompt_pending = 0;
    int prompt_rows = 0;
    int last_gamma = -1;
    int last_pass_rows = 0;
    std::vector<int> slot_off, slot_cnt;  // history ring rows per slot
    int hist_next = 0;
    int64_t launches = 0;
    int64_t h2d = 0, d2h = 0;
    // bf16: TMA maps of every weight matrix and of the three projection inputs
    std::vector<CUtensorMap> map_qkv, map_o, map_gu, map_down;
    CUtensorMap map_lm, map_xg[16], map_xg2[16], map_attn_out[16], map_act[16];  // [R - 1]: boxes of R rows
    KlassTiming timing[kKlasses];
};

// ----------------------------------------------------------------- plumbing
static ks_status cuda_fail(cudaError_t e, const char* what) {
    set_error("%s: %s", what, cudaGetErrorString(e));
    return KS_ERR_CUDA;
}

#define KS_CUDA(call, what)                                   \
    do {                                                      \
        cudaError_t e_ = (call);                              \
        if (e_ != cudaSuccess) return cuda_fail(e_, what);    \
    } while (0)

template <class F>
static ks_status launch(ks_model* m, int klass, F&& f, const char* what, double bytes = 0.0) {
    KlassTiming& T = m->timing[klass];
    if (T.on) T.bytes += bytes;
    cudaEvent_t e0 = nullptr, e1 = nullptr;
    if (T.on) {
        if (T.used + 2 > T.ev.size()) {
            for (int i = 0; i < 64; ++i) {
                cudaEvent_t e;
                KS_CUDA(cudaEventCreate(&e), "cudaEventCreate");
                T.ev.push_back(e);
            }
        }
        e0 = T.ev[T.used];
        e1 = T.ev[T.used + 1];
        T.used += 2;
        KS_CUDA(cudaEventRecord(e0, m->stream), "cudaEventRecord");
    }
    cudaError_t e = f();
    if (e != cudaSuccess) return cuda_fail(e, what);
    m->launches++;
    if (T.on) KS_CUDA(cudaEventRecord(e1, m->stream), "cudaEventRecord");
    return KS_OK;
}

#define KS_TRY(expr)                   \
    do {                               \
        ks_status s_ = (expr);         \
        if (s_ != KS_OK) return s_;    \
    } while (0)

static float* hist_plane(ks_model* m, int plane) {
    const size_t plane_elems = (size_t)m->lay.hist_slots * m->cfg.max_rows * m->cfg.d_model;
    return m->hist + (size_t)plane * plane_elems;
}

static void* kcache(ks_model* m, int layer) {
    const size_t per = (size_t)m->cfg.n_kv_heads * m->cfg.max_seq * m->cfg.head_dim * m->es;
    return m->kv + (size_t)(2 * layer) * per;
}
static void* vcache(ks_model* m, int layer) {
    const size_t per = (size_t)m->cfg.n_kv_heads * m->cfg.max_seq * m->cfg.head_dim * m->es;
    return m->kv + (size_t)(2 * layer + 1) * per;
}

// One pass of f^(S) over R consecutive rows at positions p0..p0+R-1.
// tok: device token ids of the rows.  mask: host uint8[2L] or null (all).
// capture_slot >= 0: write X^(i) of every row into the history slot (all
// sublayers must run).  argmax: device int32[R] for the LM head argmax, or
// null to skip the LM head.
static ks_status forward(ks_model* m, const int32_t* tok, int R, int p0, const uint8_t* mask,
                         int capture_slot, int32_t* argmax, const int* stop = nullptr) {
    const ks_config& c = m->cfg;
    const int d = c.d_model, hd = c.head_dim;
    const int nqkv = (c.n_q_heads + 2 * c.n_kv_heads) * hd;
    const int dt = m->dtype;
    const bool bf = dt == KS_DTYPE_BF16;
    const int ssg = (d + kSsGroup - 1) / kSsGroup;
    cudaStream_t s = m->stream;
    auto cap_ptr = [&](int plane) -> float* {
        if (capture_slot < 0) return nullptr;
        return hist_plane(m, plane) + (size_t)capture_slot * c.max_rows * d;
    };
    auto runs = [&](int i) { return !mask || mask[i - 1]; };  // 1-based sublayer i
    // gain of the RMSNorm that reads the residual after sublayer i (0 = embed):
    // the next sublayer that runs, else the final norm
    auto next_gain = [&](int i) -> const void* {
        for (int k = i + 1; k <= 2 * c.n_layers; ++k)
            if (runs(k)) return (k % 2 == 1) ? m->attn_norm[(k - 1) / 2] : m->mlp_norm[(k - 1) / 2];
        return m->final_norm;
    };
    // input of a normalised projection
    auto norm_input = [&](GemvArgs& g, const void* gain) {
        g.ss_in = m->ss;
        g.ss_groups = ssg;
        g.eps = c.rms_eps;
        if (bf) {
            g.in = m->xg;       // x * gain in bf16, scaled by 1 / rms in the epilogue
            g.in_ld = d;
        } else {
            g.in = m->x;        // fp32 kernel normalises while staging
            g.in_ld = d;
            g.norm_gain = gain;
        }
    };
    auto resid_output = [&](GemvArgs& g, int after) {
        g.resid = m->x;
        g.resid_ld = d;
        g.ss_out = m->ss;
        g.capture = cap_ptr(after);
        g.capture_ld = d;
        if (bf) {
            g.xg_out = m->xg;
            g.next_gain = next_gain(after);
        }
    };
    auto common = [&](GemvArgs& g, const void* W, int N, int K) {
        g.W = W;
        g.dtype = dt;
        g.N = N;
        g.K = K;
        g.R = R;
        g.partial = m->gemv_part;
        g.counters = m->counters;
        g.err = m->err;
        g.stop = stop;
    };
    KS_TRY(launch(m, K_EMBED, [&]() -> cudaError_t {
        if (!tok) {   // input rows already in x
            if (bf)
                rows_prep_kernel<__nv_bfloat16><<<dim3(R, (d + 255) / 256), 256, 0, s>>>(
                    m->x, d, m->ss, m->xg, reinterpret_cast<const __nv_bfloat16*>(next_gain(0)), stop);
            else
                rows_prep_kernel<float><<<dim3(R, (d + 255) / 256), 256, 0, s>>>(m->x, d, m->ss, nullptr,
                                                                                  nullptr, stop);
            return cudaGetLastError();
        }
        if (bf)
            embed_kernel<__nv_bfloat16><<<dim3(R, (d + 255) / 256), 256, 0, s>>>(
                reinterpret_cast<const __nv_bfloat16*>(m->embed), tok, d, c.vocab, m->x, cap_ptr(0), m->ss, m->xg,
                reinterpret_cast<const __nv_bfloat16*>(next_gain(0)), stop);
        else
            embed_kernel<float><<<dim3(R, (d + 255) / 256), 256, 0, s>>>(reinterpret_cast<const float*>(m->embed), tok, d, c.vocab, m->x,
                                                  cap_ptr(0), m->ss, nullptr, nullptr, stop);
        return cudaGetLastError();
    }, "embed"));

    // attention core of layer l: RoPE / QK-norm, cache write, split-KV, merge
    auto attention = [&](int l) -> ks_status {
        AttnArgs at{};
        at.qkv = m->qkv; at.qkv_ld = nqkv; at.R = R; at.p0 = p0;
        at.hq = c.n_q_heads; at.hk = c.n_kv_heads; at.hd = hd;
        at.kcache = kcache(m, l); at.vcache = vcache(m, l); at.max_seq = c.max_seq;
        at.rope = m->rope;
        at.q_norm = c.qk_norm ? m->q_norm[l] : nullptr;
        at.k_norm = c.qk_norm ? m->k_norm[l] : nullptr;
        at.eps = c.rms_eps;
        at.part = m->attn_part; at.n_chunks_max = m->lay.n_chunks_max;
        at.out = m->attn_out; at.out_ld = c.n_q_heads * hd;
        at.stop = stop;
        at.err = m->err;
        if (bf) {
            at.kvmap = m->map_kv;
            at.kv_row_k = 2 * l * c.n_kv_heads * c.max_seq;
            at.kv_row_v = (2 * l + 1) * c.n_kv_heads * c.max_seq;
            at.q = m->qbuf;
            KS_TRY(launch(m, K_PREP, [&] { return launch_attn_prep(at, s); }, "attention query prep"));
        }
        KS_TRY(launch(m, K_ATTN, [&] { return launch_attention(dt, at, s); }, "attention"));
        KS_TRY(launch(m, K_MERGE, [&] { return launch_attn_merge(dt, at, s); }, "attention merge"));
        return KS_OK;
    };
    for (int l = 0; l < c.n_layers; ++l) {
        if ((!runs(2 * l + 1) || !runs(2 * l + 2)) && capture_slot >= 0) {
            set_error("forward: capture needs every sublayer");
            return KS_ERR_STATE;
        }
    }

    if (bf) {
        // bf16: consecutive projections run as one chain launch; a chain ends
        // at each attention core.  While a projection class is being timed,
        // every projection is its own launch so that it can be timed alone.
        const bool split = m->timing[K_QKV].on || m->timing[K_OPROJ].on || m->timing[K_GATEUP].on ||
                           m->timing[K_DOWN].on || m->timing[K_LMHEAD].on;
        const int L = c.n_layers, F = c.d_ff, hqd = c.n_q_heads * hd;
        if (!m->chain) m->chain = new ChainArgs();
        ChainArgs& ca = *m->chain;
        ca.amap[0] = m->map_xg[R - 1];
        ca.amap[1] = m->map_xg2[R - 1];
        ca.amap[2] = m->map_attn_out[R - 1];
        ca.amap[3] = m->map_act[R - 1];
        ca.R = R;
        ca.n_layers = L; ca.d = d; ca.F = F; ca.nqkv = nqkv; ca.hqd = hqd; ca.vocab = c.vocab;
        ca.eps = c.rms_eps;
        ca.x = m->x; ca.ss = m->ss; ca.xg = m->xg; ca.qkv = m->qkv;
        ca.act = reinterpret_cast<__nv_bfloat16*>(m->act);
        ca.logits = m->logits; ca.best = m->best; ca.tokens = argmax;
        ca.capture = capture_slot >= 0 ? hist_plane(m, 0) + (size_t)capture_slot * c.max_rows * d : nullptr;
        ca.capture_plane = (long long)m->lay.hist_slots * c.max_rows * d;
        ca.err = m->err;
        ca.stop = stop;
        ca.slice_part = m->slice_part;
        ca.slice_ticket = m->slice_ticket;
        int nph = 0, klass = K_CHAIN;
        double bytes = 0.0;
        auto flush = [&]() -> ks_status {
            if (nph == 0) return KS_OK;
            ca.n_phases = nph;
            ca.counters = m->chain_ctr + (size_t)m->chain_parity * chain_counter_ints();
            m->chain_parity ^= 1;
            KS_TRY(launch(m, split ? klass : K_CHAIN, [&] { return launch_chain(ca, s); }, "projections", bytes));
            nph = 0;
            bytes = 0.0;
            return KS_OK;
        };
        auto add = [&](int layer, int kind, const void* gain, int k_class) -> ks_status {
            const double es2 = 2.0;
            const double wb = kind == CH_QKV ? es2 * nqkv * d
                            : kind == CH_O ? es2 * d * hqd
                            : kind == CH_GU ? es2 * 2.0 * F * d
                            : kind == CH_DOWN ? es2 * d * F
                            : es2 * c.vocab * d;
            ca.code[nph] = (uint16_t)(kind == CH_LM ? 4 * L : 4 * layer + kind);
            ca.gain[nph] = reinterpret_cast<const __nv_bfloat16*>(gain);
            ca.wmap[nph] = kind == CH_QKV ? m->map_qkv[layer]
                         : kind == CH_O ? m->map_o[layer]
                         : kind == CH_GU ? m->map_gu[layer]
                         : kind == CH_DOWN ? m->map_down[layer] : m->map_lm;
            ++nph;
            bytes += wb;
            klass = k_class;
            return (split || nph == kChainMaxPhases) ? flush() : KS_OK;
        };
        for (int l = 0; l < L; ++l) {
            if (runs(2 * l + 1)) {
                KS_TRY(add(l, CH_QKV, nullptr, K_QKV));
                KS_TRY(flush());
                KS_TRY(attention(l));
                KS_TRY(add(l, CH_O, next_gain(2 * l + 1), K_OPROJ));
            }
            if (runs(2 * l + 2)) {
                KS_TRY(add(l, CH_GU, nullptr, K_GATEUP));
                KS_TRY(add(l, CH_DOWN, next_gain(2 * l + 2), K_DOWN));
            }
        }
        if (argmax) KS_TRY(add(0, CH_LM, nullptr, K_LMHEAD));
        KS_TRY(flush());
        m->last_pass_rows = R;
        return KS_OK;
    }

    for (int l = 0; l < c.n_layers; ++l) {
        const bool run_attn = runs(2 * l + 1);
        const bool run_mlp = runs(2 * l + 2);
        if (run_attn) {
            GemvArgs g{};
            common(g, m->w_qkv[l], nqkv, d);
            norm_input(g, m->attn_norm[l]);
            g.out = m->qkv;
            g.out_ld = nqkv;
            gemv_plan(g, EPI_STORE);
            KS_TRY(launch(m, K_QKV, [&] { return launch_gemv(dt, EPI_STORE, g, s); }, "qkv"));
            KS_TRY(attention(l));
            GemvArgs o{};
            common(o, m->w_o[l], d, c.n_q_heads * hd);
            o.in = m->attn_out;
            o.in_ld = c.n_q_heads * hd;
            resid_output(o, 2 * l + 1);
            gemv_plan(o, EPI_RESID);
            KS_TRY(launch(m, K_OPROJ, [&] { return launch_gemv(dt, EPI_RESID, o, s); }, "o-proj"));
        }
        if (run_mlp) {
            GemvArgs gu{};
            common(gu, m->w_gate_up[l], c.d_ff, d);
            norm_input(gu, m->mlp_norm[l]);
            gu.act = m->act;
            gu.act_ld = c.d_ff;
            gemv_plan(gu, EPI_SWIGLU);
            KS_TRY(launch(m, K_GATEUP, [&] { return launch_gemv(dt, EPI_SWIGLU, gu, s); }, "gate-up"));
            GemvArgs dn{};
            common(dn, m->w_down[l], d, c.d_ff);
            dn.in = m->act;
            dn.in_ld = c.d_ff;
            resid_output(dn, 2 * l + 2);
            gemv_plan(dn, EPI_RESID);
            KS_TRY(launch(m, K_DOWN, [&] { return launch_gemv(dt, EPI_RESID, dn, s); }, "down"));
        }
    }
    if (argmax) {
        GemvArgs lm{};
        common(lm, m->lm_head, c.vocab, d);
        norm_input(lm, m->final_norm);
        lm.logits = m->logits;
        lm.logits_ld = c.vocab;
        lm.amax_val = m->amax_val;
        lm.amax_idx = m->amax_idx;
        lm.tokens = argmax;
        gemv_plan(lm, EPI_LMHEAD);
        KS_TRY(launch(m, K_LMHEAD, [&] { return launch_gemv(dt, EPI_LMHEAD, lm, s); }, "lm-head"));
    }
    m->last_pass_rows = R;
    return KS_OK;
}

// Wait for the stream, then read the device status word (set when a kernel's
// bounded wait on an asynchronous copy gave up).
static ks_status sync(ks_model* m, const char* what) {
    int32_t* hs = m->h_buf + m->h_buf_ints - 1;
    cudaError_t e = cudaMemcpyAsync(hs, m->err, sizeof(int32_t), cudaMemcpyDeviceToHost, m->stream);
    if (e != cudaSuccess) return cuda_fail(e, what);
    e = cudaStreamSynchronize(m->stream);
    if (e != cudaSuccess) return cuda_fail(e, what);
    if (*hs == 1) {
        set_error("%s: a kernel gave up waiting for an asynchronous copy", what);
        return KS_ERR_TIMEOUT;
    }
    if (*hs != 0) {
        set_error("%s: a kernel's self-check failed (status word %d)", what, *hs);
        return KS_ERR_STATE;
    }
    return KS_OK;
}

// ------------------------------------------------------------------- C ABI
extern "C" {

const char* ks_status_str(ks_status s) {
    switch (s) {
        case KS_OK: return "KS_OK";
        case KS_ERR_INVALID_ARG: return "KS_ERR_INVALID_ARG";
        case KS_ERR_CUDA: return "KS_ERR_CUDA";
        case KS_ERR_WORKSPACE: return "KS_ERR_WORKSPACE";
        case KS_ERR_CAPACITY: return "KS_ERR_CAPACITY";
        case KS_ERR_TIMEOUT: return "KS_ERR_TIMEOUT";
        case KS_ERR_UNSUPPORTED: return "KS_ERR_UNSUPPORTED";
        case KS_ERR_STATE: return "KS_ERR_STATE";
    }
    return "KS_ERR_UNKNOWN";
}

const char* ks_last_error(void) { return g_err; }

size_t ks_workspace_bytes(const ks_config* cfg) {
    if (!config_ok(cfg)) return 0;
    return make_layout(cfg).total;
}

ks_status ks_model_create(const ks_config* cfg, const ks_weights* w, void* workspace, size_t workspace_bytes,
                          void* stream, ks_model** out) {
    if (!out) {
        set_error("ks_model_create: out is null");
        return KS_ERR_INVALID_ARG;
    }
    *out = nullptr;
    if (!config_ok(cfg)) {
        set_error("ks_model_create: invalid or unsupported config");
        return KS_ERR_INVALID_ARG;
    }
    if (!w || !workspace) {
        set_error("ks_model_create: null weights or workspace");
        return KS_ERR_INVALID_ARG;
    }
    if (reinterpret_cast<uintptr_t>(workspace) & 255) {
        set_error("ks_model_create: workspace must be 256-byte aligned");
        return KS_ERR_INVALID_ARG;
    }
    const Layout lay = make_layout(cfg);
    if (workspace_bytes < lay.total) {
        set_error("ks_model_create: workspace %zu < required %zu", workspace_bytes, lay.total);
        return KS_ERR_WORKSPACE;
    }
    const int L = cfg->n_layers;
    auto aligned = [](const void* p) { return p && (reinterpret_cast<uintptr_t>(p) & 15) == 0; };
    if (!aligned(w->embed) || !aligned(w->lm_head) || !aligned(w->final_norm) || !w->attn_norm || !w->w_qkv ||
        !w->w_o || !w->mlp_norm || !w->w_gate_up || !w->w_down || (cfg->qk_norm && (!w->q_norm || !w->k_norm))) {
        set_error("ks_model_create: missing or misaligned weight pointer");
        return KS_ERR_INVALID_ARG;
    }
    for (int l = 0; l < L; ++l) {
        if (!aligned(w->attn_norm[l]) || !aligned(w->w_qkv[l]) || !aligned(w->w_o[l]) || !aligned(w->mlp_norm[l]) ||
            !aligned(w->w_gate_up[l]) || !aligned(w->w_down[l]) ||
            (cfg->qk_norm && (!aligned(w->q_norm[l]) || !aligned(w->k_norm[l])))) {
            set_error("ks_model_create: layer %d weight pointer missing or not 16-byte aligned", l);
            return KS_ERR_INVALID_ARG;
        }
    }
    ks_model* m = new ks_model();
    m->cfg = *cfg;
    m->dtype = cfg->dtype;
    m->es = cfg->dtype == KS_DTYPE_BF16 ? 2 : 4;
    m->nsub = 2 * L;
    m->embed = w->embed;
    m->lm_head = w->lm_head;
    m->final_norm = w->final_norm;
    for (int l = 0; l < L; ++l) {
        m->attn_norm.push_back(w->attn_norm[l]);
        m->w_qkv.push_back(w->w_qkv[l]);
        m->w_o.push_back(w->w_o[l]);
        m->q_norm.push_back(cfg->qk_norm ? w->q_norm[l] : nullptr);
        m->k_norm.push_back(cfg->qk_norm ? w->k_norm[l] : nullptr);
        m->mlp_norm.push_back(w->mlp_norm[l]);
        m->w_gate_up.push_back(w->w_gate_up[l]);
        m->w_down.push_back(w->w_down[l]);
    }
    m->stream = reinterpret_cast<cudaStream_t>(stream);
    m->ws = reinterpret_cast<char*>(workspace);
    m->ws_bytes = workspace_bytes;
    m->lay = lay;
    char* b = m->ws;
    m->kv = b + lay.kv;
    m->rope = reinterpret_cast<float*>(b + lay.rope);
    m->x = reinterpret_cast<float*>(b + lay.x);
    m->ss = reinterpret_cast<float*>(b + lay.ss);
    m->xg = reinterpret_cast<__nv_bfloat16*>(b + lay.xg);
    m->qkv = reinterpret_cast<float*>(b + lay.qkv);
    m->attn_out = b + lay.attn_out;
    m->act = b + lay.act;
    m->attn_part = reinterpret_cast<float*>(b + lay.attn_part);
    m->gemv_part = reinterpret_cast<float*>(b + lay.gemv_part);
    m->counters = reinterpret_cast<int*>(b + lay.counters);
    m->logits = reinterpret_cast<float*>(b + lay.logits);
    m->amax_val = reinterpret_cast<float*>(b + lay.amax_val);
    m->amax_idx = reinterpret_cast<int*>(b + lay.amax_idx);
    int* tok = reinterpret_cast<int*>(b + lay.tok);
    const int R = cfg->max_rows;
    m->rows = tok;
    m->target = tok + (R + 1);
    m->result = tok + (2 * R + 1);
    m->err = tok + (3 * R + 4);
    m->seq = tok + (3 * R + 8);
    m->hist = reinterpret_cast<float*>(b + lay.hist);
    m->hist_snap = reinterpret_cast<float*>(b + lay.hist_snap);
    m->hist_idx = reinterpret_cast<int*>(b + lay.hist_idx);
    m->sims = reinterpret_cast<float*>(b + lay.sims);
    m->mask_dev = reinterpret_cast<uint8_t*>(b + lay.mask);
    m->chain_ctr = reinterpret_cast<int*>(b + lay.chain_ctr);
    m->best = reinterpret_cast<unsigned long long*>(b + lay.best);
    m->tpt_masks = reinterpret_cast<uint8_t*>(b + lay.tpt_masks);
    m->tpt_tok = reinterpret_cast<int32_t*>(b + lay.tpt_tok);
    m->tpt_info = reinterpret_cast<int32_t*>(b + lay.tpt_info);
    m->tpt_out = reinterpret_cast<double*>(b + lay.tpt_out);
    m->conf = reinterpret_cast<float*>(b + lay.dyn);
    m->top1_part = m->conf + cfg->max_rows;
    m->top1_ticket = reinterpret_cast<int*>(m->top1_part + kTop1Ctas);
    m->stop = m->rows + (3 * cfg->max_rows + 5);        // spare words of the token block
    m->n_drafted = m->rows + (3 * cfg->max_rows + 6);
    m->slice_part = reinterpret_cast<float*>(b + lay.slice);
    m->slice_ticket = reinterpret_cast<int*>(m->slice_part + (size_t)2 * kChainSliceMaxItems * 512);
    m->qbuf = reinterpret_cast<__nv_bfloat16*>(b + lay.qbuf);
    {
        char* sb = b + lay.samp;
        const size_t RK = (size_t)cfg->max_rows * kSampleMaxK;
        m->q_ids = reinterpret_cast<int*>(sb);
        m->q_probs = reinterpret_cast<float*>(m->q_ids + RK);
        m->q_n = reinterpret_cast<int*>(m->q_probs + RK);
        m->p_ids = m->q_n + cfg->max_rows;
        m->p_probs = reinterpret_cast<float*>(m->p_ids + RK);
        m->p_n = reinterpret_cast<int*>(m->p_probs + RK);
    }
    m->obj_dev = reinterpret_cast<double*>(b + lay.obj);
    m->wts_dev = reinterpret_cast<int*>(b + lay.wts);
    m->select = b + lay.select;
    m->slot_off.assign(lay.hist_slots, 0);
    m->slot_cnt.assign(lay.hist_slots, 0);
    if (m->dtype == KS_DTYPE_BF16) {
        const int d = cfg->d_model, F = cfg->d_ff, hqd = cfg->n_q_heads * cfg->head_dim;
        const int nqkv = (cfg->n_q_heads + 2 * cfg->n_kv_heads) * cfg->head_dim;
        bool ok = true;
        m->map_qkv.resize(L);
        m->map_o.resize(L);
        m->map_gu.resize(L);
        m->map_down.resize(L);
        for (int l = 0; l < L && ok; ++l) {
            ok = ok && make_weight_map(&m->map_qkv[l], m->w_qkv[l], nqkv, d, 16);
            ok = ok && make_weight_map(&m->map_o[l], m->w_o[l], d, hqd, 16);
            ok = ok && make_weight_map(&m->map_gu[l], m->w_gate_up[l], 2 * (uint64_t)F, d, 8);
            ok = ok && make_weight_map(&m->map_down[l], m->w_down[l], d, F, 16);
        }
        ok = ok && make_weight_map(&m->map_lm, m->lm_head, cfg->vocab, d, 16);
        // [L][K, V][hk][max_seq] rows of hd elements; a box is one 16-key tile
        ok = ok && make_weight_map(&m->map_kv, m->kv,
                                   2 * (uint64_t)L * cfg->n_kv_heads * (uint64_t)cfg->max_seq, cfg->head_dim,
                                   cfg->head_dim / 64);
        for (int b = 0; b < R; ++b) {
            ok = ok && make_stage_map(&m->map_xg[b], m->xg, R, d, b + 1, 4);
            ok = ok && make_stage_map(&m->map_xg2[b], m->xg, R, d, b + 1, 2);
            ok = ok && make_stage_map(&m->map_attn_out[b], m->attn_out, R, hqd, b + 1, 4);
            ok = ok && make_stage_map(&m->map_act[b], m->act, R, F, b + 1, 4);
        }
        if (!ok) {
            set_error("ks_model_create: TMA descriptor encoding failed");
            delete m;
            return KS_ERR_CUDA;
        }
    }

    auto fail = [&](cudaError_t e, const char* what) {
        ks_status st = cuda_fail(e, what);
        if (m->h_buf) cudaFreeHost(m->h_buf);
        delete m;
        return st;
    };
    m->h_buf_ints = (size_t)cfg->max_seq + 4 * (size_t)R + 64 + lay.hist_slots * (size_t)R + 2 * (size_t)L + 64 +
                    4 * (size_t)kDpMaxStates + 4 * (size_t)L + 64;   // + the DP stage's staging
    cudaError_t e = cudaHostAlloc(reinterpret_cast<void**>(&m->h_buf), m->h_buf_ints * sizeof(int32_t),
                                  cudaHostAllocDefault);
    if (e != cudaSuccess) {
        m->h_buf = nullptr;
        return fail(e, "cudaHostAlloc");
    }
    // RoPE table in double, rounded to fp32: [pos][j][cos, sin]
    {
        const int hd = cfg->head_dim, half = hd / 2;
        std::vector<float> tab((size_t)cfg->max_seq * hd);
        std::vector<double> inv(half);
        for (int j = 0; j < half; ++j) inv[j] = std::pow(cfg->rope_theta, -2.0 * j / hd);
        for (int p = 0; p < cfg->max_seq; ++p)
            for (int j = 0; j < half; ++j) {
                const double ang = (double)p * inv[j];
                tab[((size_t)p * half + j) * 2] = (float)std::cos(ang);
                tab[((size_t)p * half + j) * 2 + 1] = (float)std::sin(ang);
            }
        e = cudaMemcpyAsync(m->rope, tab.data(), tab.size() * sizeof(float), cudaMemcpyHostToDevice, m->stream);
        if (e != cudaSuccess) return fail(e, "rope upload");
        e = cudaStreamSynchronize(m->stream);
        if (e != cudaSuccess) return fail(e, "rope upload");
    }
    e = cudaMemsetAsync(m->counters, 0, sizeof(int) * lay.counters_n, m->stream);
    if (e != cudaSuccess) return fail(e, "counter reset");
    // The bf16 attention streams whole 16-key tiles; keys past a row's
    // position are masked (softmax weight exactly 0), which needs finite
    // values there: positions never written hold zeros.
    e = cudaMemsetAsync(m->kv, 0, lay.rope - lay.kv, m->stream);
    if (e != cudaSuccess) return fail(e, "KV cache reset");
    e = cudaMemsetAsync(m->chain_ctr, 0, sizeof(int) * 2 * chain_counter_ints(), m->stream);
    if (e != cudaSuccess) return fail(e, "counter reset");
    e = cudaMemsetAsync(m->best, 0, sizeof(unsigned long long) * 16, m->stream);
    if (e != cudaSuccess) return fail(e, "counter reset");
    e = cudaMemsetAsync(b + lay.tok, 0, sizeof(int) * ((size_t)3 * R + 8 + cfg->max_seq), m->stream);  // incl. err
    if (e != cudaSuccess) return fail(e, "token reset");
    e = cudaMemsetAsync(m->slice_ticket, 0, sizeof(int) * 2 * kChainSliceMaxItems, m->stream);
    if (e != cudaSuccess) return fail(e, "slice reset");
    e = cudaMemsetAsync(b + lay.dyn, 0, sizeof(float) * ((size_t)R + kTop1Ctas) + sizeof(int), m->stream);
    if (e != cudaSuccess) return fail(e, "dynamic-exit reset");
    e = cudaStreamSynchronize(m->stream);
    if (e != cudaSuccess) return fail(e, "create sync");
    *out = m;
    return KS_OK;
}

ks_status ks_model_destroy(ks_model* m) {
    if (!m) return KS_ERR_INVALID_ARG;
    cudaStreamSynchronize(m->stream);
    for (auto& T : m->timing)
        for (auto e : T.ev) cudaEventDestroy(e);
    if (m->h_buf) cudaFreeHost(m->h_buf);
    delete m->chain;
    delete m;
    return KS_OK;
}

// The history after a prefill: one entry holding the last hist_init_rows of
// the prompt's final chunk (lastlen rows captured in slot 0).
static void reset_history(ks_model* m, int lastlen) {
    m->last_gamma = -1;
    m->last_dynamic = false;
    m->last_sampled = false;
    std::fill(m->slot_cnt.begin(), m->slot_cnt.end(), 0);
    const int init = std::min(m->cfg.hist_init_rows, lastlen);
    m->slot_off[0] = lastlen - init;
    m->slot_cnt[0] = init;
    m->hist_next = 1;
}

ks_status ks_prefill(ks_model* m, const int32_t* tokens, int32_t n, int32_t* next_token) {
    if (!m || !tokens || !next_token) {
        set_error("ks_prefill: null argument");
        return KS_ERR_INVALID_ARG;
    }
    const ks_config& c = m->cfg;
    if (n < 1) {
        set_error("ks_prefill: n must be >= 1");
        return KS_ERR_INVALID_ARG;
    }
    if (n + 1 > c.max_seq) {
        set_error("ks_prefill: prompt of %d does not fit max_seq %d", n, c.max_seq);
        return KS_ERR_CAPACITY;
    }
    for (int i = 0; i < n; ++i)
        if (tokens[i] < 0 || tokens[i] >= c.vocab) {
            set_error("ks_prefill: token %d out of range", i);
            return KS_ERR_INVALID_ARG;
        }
    m->have_seq = false;
    m->prompt_len = 0;
    std::memcpy(m->h_buf, tokens, sizeof(int32_t) * n);
    KS_CUDA(cudaMemcpyAsync(m->seq, m->h_buf, sizeof(int32_t) * n, cudaMemcpyHostToDevice, m->stream), "prompt upload");
    m->h2d += sizeof(int32_t) * n;
    const int R = c.max_rows;
    // chunks aligned to the end so the last chunk holds the last R rows
    const int first = n - R * ((n - 1) / R);
    int start = 0;
    int len = first;
    const int init_slot = 0;
    while (start < n) {
        const bool last = (start + len == n);
        KS_TRY(forward(m, m->seq + start, len, start, nullptr, last ? init_slot : -1, last ? m->target : nullptr));
        start += len;
        len = R;
    }
    // pending = argmax of the last prompt row
    const int lastlen = (n <= R) ? n : R;
    KS_CUDA(cudaMemcpyAsync(m->rows, m->target + (lastlen - 1), sizeof(int32_t), cudaMemcpyDeviceToDevice, m->stream),
            "pending");
    KS_CUDA(cudaMemcpyAsync(m->h_buf, m->rows, sizeof(int32_t), cudaMemcpyDeviceToHost, m->stream), "pending");
    m->d2h += sizeof(int32_t);
    KS_TRY(sync(m, "ks_prefill"));
    m->pending = m->h_buf[0];
    *next_token = m->pending;
    m->p = n;
    m->have_seq = true;
    m->prompt_len = n;
    m->prompt_pending = m->pending;
    m->prompt_rows = lastlen;
    // keep the prefill's history entry (slot 0 of every plane) for ks_rewind
    const size_t row_bytes = sizeof(float) * (size_t)c.max_rows * c.d_model;
    KS_CUDA(cudaMemcpy2DAsync(m->hist_snap, row_bytes, m->hist, row_bytes * m->lay.hist_slots, row_bytes,
                              m->nsub + 1, cudaMemcpyDeviceToDevice, m->stream),
            "history snapshot");
    reset_history(m, lastlen);
    return KS_OK;
}

ks_status ks_rewind(ks_model* m, int32_t* next_token) {
    if (!m || !next_token) {
        set_error("ks_rewind: null argument");
        return KS_ERR_INVALID_ARG;
    }
    if (m->prompt_len < 1) {
        set_error("ks_rewind: no prompt (call ks_prefill first)");
        return KS_ERR_STATE;
    }
    // Decode steps write K/V only at positions >= the prompt length, so the
    // prompt's cache is intact; restore the pending token and the history.
    const ks_config& c = m->cfg;
    m->have_seq = false;
    m->h_buf[0] = m->prompt_pending;
    KS_CUDA(cudaMemcpyAsync(m->rows, m->h_buf, sizeof(int32_t), cudaMemcpyHostToDevice, m->stream), "pending");
    m->h2d += sizeof(int32_t);
    const size_t row_bytes = sizeof(float) * (size_t)c.max_rows * c.d_model;
    KS_CUDA(cudaMemcpy2DAsync(m->hist, row_bytes * m->lay.hist_slots, m->hist_snap, row_bytes, row_bytes,
                              m->nsub + 1, cudaMemcpyDeviceToDevice, m->stream),
            "history restore");
    KS_TRY(sync(m, "ks_rewind"));
    m->p = m->prompt_len;
    m->pending = m->prompt_pending;
    m->have_seq = true;
    reset_history(m, m->prompt_rows);
    *next_token = m->pending;
    return KS_OK;
}

ks_status ks_draft(ks_model* m, const uint8_t* mask, int32_t gamma, int32_t* draft_tokens) {
    if (!m || !mask) {
        set_error("ks_draft: null argument");
        return KS_ERR_INVALID_ARG;
    }
    if (!m->have_seq) {
        set_error("ks_draft: no sequence (call ks_prefill first)");
        return KS_ERR_STATE;
    }
    if (gamma < 1 || gamma >= m->cfg.max_rows) {
        set_error("ks_draft: gamma must be in [1, max_rows)");
        return KS_ERR_INVALID_ARG;
    }
    if (m->p + gamma + 1 > m->cfg.max_seq) {
        set_error("ks_draft: KV capacity exceeded");
        return KS_ERR_CAPACITY;
    }
    for (int t = 0; t < gamma; ++t)
        KS_TRY(forward(m, m->rows + t, 1, m->p + t, mask, -1, m->rows + t + 1));
    m->last_gamma = gamma;
    m->last_dynamic = false;
    m->last_sampled = false;
    if (draft_tokens) {
        KS_CUDA(cudaMemcpyAsync(m->h_buf, m->rows + 1, sizeof(int32_t) * gamma, cudaMemcpyDeviceToHost, m->stream),
                "draft download");
        m->d2h += sizeof(int32_t) * gamma;
        KS_TRY(sync(m, "ks_draft"));
        std::memcpy(draft_tokens, m->h_buf, sizeof(int32_t) * gamma);
    }
    return KS_OK;
}

ks_status ks_draft_dynamic(ks_model* m, const uint8_t* mask, int32_t gamma, float tau_conf, int32_t* n_drafted,
                           float* confidence, int32_t* draft_tokens) {
    if (!m || !mask) {
        set_error("ks_draft_dynamic: null argument");
        return KS_ERR_INVALID_ARG;
    }
    if (!m->have_seq) {
        set_error("ks_draft_dynamic: no sequence (call ks_prefill first)");
        return KS_ERR_STATE;
    }
    if (gamma < 1 || gamma >= m->cfg.max_rows || !(tau_conf >= 0.f) || !std::isfinite(tau_conf)) {
        set_error("ks_draft_dynamic: gamma must be in [1, max_rows) and tau_conf finite and >= 0");
        return KS_ERR_INVALID_ARG;
    }
    if (m->p + gamma + 1 > m->cfg.max_seq) {
        set_error("ks_draft_dynamic: KV capacity exceeded");
        return KS_ERR_CAPACITY;
    }
    cudaStream_t s = m->stream;
    // a new step: no pass has run and none has stopped (stop and n_drafted are adjacent)
    KS_CUDA(cudaMemsetAsync(m->stop, 0, 2 * sizeof(int), s), "dynamic-exit reset");
    for (int t = 0; t < gamma; ++t) {
        KS_TRY(forward(m, m->rows + t, 1, m->p + t, mask, -1, m->rows + t + 1, m->stop));
        KS_TRY(launch(m, K_ACCEPT, [&]() -> cudaError_t {
            top1_kernel<<<kTop1Ctas, kTop1Threads, 0, s>>>(m->logits, m->cfg.vocab, m->rows + t + 1, tau_conf, t,
                                                           m->stop, m->n_drafted, m->conf, m->top1_part,
                                                           m->top1_ticket);
            return cudaGetLastError();
        }, "draft confidence"));
    }
    m->last_gamma = gamma;
    m->last_dynamic = true;
    m->last_sampled = false;
    if (n_drafted || confidence || draft_tokens) {
        int32_t* hb = m->h_buf;   // tokens [0, 16), count [16], confidences [32, 48)
        KS_CUDA(cudaMemcpyAsync(hb, m->rows + 1, sizeof(int32_t) * gamma, cudaMemcpyDeviceToHost, s), "draft download");
        KS_CUDA(cudaMemcpyAsync(hb + 16, m->n_drafted, sizeof(int32_t), cudaMemcpyDeviceToHost, s), "draft download");
        KS_CUDA(cudaMemcpyAsync(hb + 32, m->conf, sizeof(float) * gamma, cudaMemcpyDeviceToHost, s), "draft download");
        m->d2h += sizeof(int32_t) * (gamma + 1) + sizeof(float) * gamma;
        KS_TRY(sync(m, "ks_draft_dynamic"));
        const int n = hb[16];
        if (n_drafted) *n_drafted = n;
        if (draft_tokens) std::memcpy(draft_tokens, hb, sizeof(int32_t) * n);
        if (confidence) std::memcpy(confidence, hb + 32, sizeof(float) * n);
    }
    return KS_OK;
}

// a2 + a3; sp != null: the sampling branch of Sec. 2.1 over the drafts of
// the preceding ks_draft_sample (filtered target rows, then the acceptance
// with residual resampling), else greedy acceptance.
static ks_status verify_impl(ks_model* m, const int32_t* draft_tokens, int32_t gamma, const ks_sampling* sp,
                             unsigned long long step, int32_t* n_accepted, int32_t* out_tokens, int32_t* n_out) {
    if (!m || !n_accepted || !out_tokens || !n_out) {
        set_error("ks_verify: null argument");
        return KS_ERR_INVALID_ARG;
    }
    if (!m->have_seq) {
        set_error("ks_verify: no sequence (call ks_prefill first)");
        return KS_ERR_STATE;
    }
    if (gamma < 1 || gamma >= m->cfg.max_rows) {
        set_error("ks_verify: gamma must be in [1, max_rows)");
        return KS_ERR_INVALID_ARG;
    }
    if (m->p + gamma + 1 > m->cfg.max_seq) {
        set_error("ks_verify: KV capacity exceeded");
        return KS_ERR_CAPACITY;
    }
    if (draft_tokens) {
        for (int i = 0; i < gamma; ++i)
            if (draft_tokens[i] < 0 || draft_tokens[i] >= m->cfg.vocab) {
                set_error("ks_verify: draft token %d out of range", i);
                return KS_ERR_INVALID_ARG;
            }
        int32_t* hb = m->h_buf + m->cfg.max_seq;  // separate staging region
        std::memcpy(hb, draft_tokens, sizeof(int32_t) * gamma);
        KS_CUDA(cudaMemcpyAsync(m->rows + 1, hb, sizeof(int32_t) * gamma, cudaMemcpyHostToDevice, m->stream),
                "draft upload");
        m->h2d += sizeof(int32_t) * gamma;
    } else if (m->last_gamma != gamma) {
        set_error("ks_verify: no preceding ks_draft with this gamma");
        return KS_ERR_STATE;
    }
    const int R = gamma + 1;
    const int slot = m->hist_next;
    KS_TRY(forward(m, m->rows, R, m->p, nullptr, slot, m->target));
    if (sp) {
        FilterArgs f{};
        f.logits = m->logits; f.ld = m->cfg.vocab; f.vocab = m->cfg.vocab;
        f.inv_t = 1.f / sp->temperature; f.top_k = sp->top_k; f.top_p = sp->top_p;
        f.ids = m->p_ids; f.probs = m->p_probs; f.n = m->p_n; f.slot0 = 0; f.token_out = nullptr;
        f.seed = sp->seed; f.step = step;
        KS_TRY(launch(m, K_ACCEPT, [&] { return launch_filter(f, R, m->stream); }, "target distributions"));
        AcceptSampleArgs ac{};
        ac.rows = m->rows; ac.gamma = gamma;
        ac.p_ids = m->p_ids; ac.p_probs = m->p_probs; ac.p_n = m->p_n;
        ac.q_ids = m->q_ids; ac.q_probs = m->q_probs; ac.q_n = m->q_n;
        ac.result = m->result; ac.seed = sp->seed; ac.step = step;
        KS_TRY(launch(m, K_ACCEPT, [&] { return launch_spec_accept(ac, m->stream); }, "sampling acceptance"));
    } else {
        KS_TRY(launch(m, K_ACCEPT, [&]() -> cudaError_t {
            accept_kernel<<<1, 32, 0, m->stream>>>(m->rows, m->target, gamma,
                                                   (m->last_dynamic && !draft_tokens) ? m->n_drafted : nullptr,
                                                   m->result);
            return cudaGetLastError();
        }, "accept"));
    }
    int32_t* hb = m->h_buf + m->cfg.max_seq + 2 * m->cfg.max_rows;
    KS_CUDA(cudaMemcpyAsync(hb, m->result, sizeof(int32_t) * (gamma + 3), cudaMemcpyDeviceToHost, m->stream),
            "result download");
    m->d2h += sizeof(int32_t) * (gamma + 3);
    KS_TRY(sync(m, "ks_verify"));
    const int a = hb[0];
    const int scored = hb[1];
    if (a < 0 || scored < 0 || scored > gamma || a > scored) {
        set_error("ks_verify: corrupt acceptance result");
        return KS_ERR_CUDA;
    }
    *n_accepted = a;
    *n_out = a + 1;
    for (int i = 0; i <= a; ++i) out_tokens[i] = hb[2 + i];
    m->pending = hb[2 + a];
    m->p += a + 1;
    m->slot_off[slot] = 0;
    m->slot_cnt[slot] = a + 1;
    m->hist_next = (slot + 1) % m->lay.hist_slots;
    // keep hist_steps entries: drop the entry the next verify will overwrite
    m->slot_cnt[m->hist_next] = 0;
    m->last_gamma = -1;
    m->last_dynamic = false;
    m->last_sampled = false;
    m->last_scored = scored;
    return KS_OK;
}

ks_status ks_verify(ks_model* m, const int32_t* draft_tokens, int32_t gamma, int32_t* n_accepted,
                    int32_t* out_tokens, int32_t* n_out) {
    if (m && !draft_tokens && m->last_sampled) {
        set_error("ks_verify: the preceding drafts were sampled (use ks_verify_sample)");
        return KS_ERR_STATE;
    }
    return verify_impl(m, draft_tokens, gamma, nullptr, 0ull, n_accepted, out_tokens, n_out);
}

static bool sampling_ok(const ks_sampling* sp) {
    return sp && sp->temperature > 0.f && std::isfinite(sp->temperature) && sp->top_k >= 1 &&
           sp->top_p > 0.f && sp->top_p <= 1.f;
}

ks_status ks_draft_sample(ks_model* m, const uint8_t* mask, int32_t gamma, const ks_sampling* sp, uint64_t step,
                          int32_t* draft_tokens) {
    if (!m || !mask || !sp) {
        set_error("ks_draft_sample: null argument");
        return KS_ERR_INVALID_ARG;
    }
    if (!m->have_seq) {
        set_error("ks_draft_sample: no sequence (call ks_prefill first)");
        return KS_ERR_STATE;
    }
    if (gamma < 1 || gamma >= m->cfg.max_rows || !sampling_ok(sp)) {
        set_error("ks_draft_sample: gamma must be in [1, max_rows); temperature > 0, top_k >= 1, 0 < top_p <= 1");
        return KS_ERR_INVALID_ARG;
    }
    if (m->p + gamma + 1 > m->cfg.max_seq) {
        set_error("ks_draft_sample: KV capacity exceeded");
        return KS_ERR_CAPACITY;
    }
    for (int t = 0; t < gamma; ++t) {
        KS_TRY(forward(m, m->rows + t, 1, m->p + t, mask, -1, m->rows + t + 1));
        FilterArgs f{};
        f.logits = m->logits; f.ld = m->cfg.vocab; f.vocab = m->cfg.vocab;
        f.inv_t = 1.f / sp->temperature; f.top_k = sp->top_k; f.top_p = sp->top_p;
        f.ids = m->q_ids; f.probs = m->q_probs; f.n = m->q_n; f.slot0 = t;
        f.token_out = m->rows + t + 1;   // replaces the LM head's argmax
        f.seed = sp->seed; f.step = step;
        KS_TRY(launch(m, K_ACCEPT, [&] { return launch_filter(f, 1, m->stream); }, "draft sample"));
    }
    m->last_gamma = gamma;
    m->last_dynamic = false;
    m->last_sampled = true;
    if (draft_tokens) {
        KS_CUDA(cudaMemcpyAsync(m->h_buf, m->rows + 1, sizeof(int32_t) * gamma, cudaMemcpyDeviceToHost, m->stream),
                "draft download");
        m->d2h += sizeof(int32_t) * gamma;
        KS_TRY(sync(m, "ks_draft_sample"));
        std::memcpy(draft_tokens, m->h_buf, sizeof(int32_t) * gamma);
    }
    return KS_OK;
}

ks_status ks_verify_sample(ks_model* m, int32_t gamma, const ks_sampling* sp, uint64_t step, int32_t* n_accepted,
                           int32_t* out_tokens, int32_t* n_out) {
    if (!m || !sp) {
        set_error("ks_verify_sample: null argument");
        return KS_ERR_INVALID_ARG;
    }
    if (!sampling_ok(sp)) {
        set_error("ks_verify_sample: temperature > 0, top_k >= 1, 0 < top_p <= 1");
        return KS_ERR_INVALID_ARG;
    }
    if (!m->last_sampled || m->last_gamma != gamma) {
        set_error("ks_verify_sample: no preceding ks_draft_sample with this gamma");
        return KS_ERR_STATE;
    }
    return verify_impl(m, nullptr, gamma, sp, step, n_accepted, out_tokens, n_out);
}

ks_status ks_decode_greedy(ks_model* m, int32_t n_tokens, int32_t* out) {
    if (!m || !out || n_tokens < 1) {
        set_error("ks_decode_greedy: bad argument");
        return KS_ERR_INVALID_ARG;
    }
    if (!m->have_seq) {
        set_error("ks_decode_greedy: no sequence (call ks_prefill first)");
        return KS_ERR_STATE;
    }
    if (m->p + n_tokens > m->cfg.max_seq) {
        set_error("ks_decode_greedy: KV capacity exceeded");
        return KS_ERR_CAPACITY;
    }
    // seq[0] = pending; step i feeds seq[i] at p + i and writes seq[i + 1]
    KS_CUDA(cudaMemcpyAsync(m->seq, m->rows, sizeof(int32_t), cudaMemcpyDeviceToDevice, m->stream), "pending");
    for (int i = 0; i + 1 < n_tokens; ++i) KS_TRY(forward(m, m->seq + i, 1, m->p + i, nullptr, -1, m->seq + i + 1));
    KS_CUDA(cudaMemcpyAsync(m->rows, m->seq + (n_tokens - 1), sizeof(int32_t), cudaMemcpyDeviceToDevice, m->stream),
            "pending");
    KS_CUDA(cudaMemcpyAsync(m->h_buf, m->seq, sizeof(int32_t) * n_tokens, cudaMemcpyDeviceToHost, m->stream),
            "tokens download");
    m->d2h += sizeof(int32_t) * n_tokens;
    KS_TRY(sync(m, "ks_decode_greedy"));
    std::memcpy(out, m->h_buf, sizeof(int32_t) * n_tokens);
    m->p += n_tokens - 1;
    m->pending = out[n_tokens - 1];
    m->last_gamma = -1;
    m->last_dynamic = false;
    m->last_sampled = false;
    return KS_OK;
}

ks_status ks_model_position(const ks_model* m, int32_t* committed, int32_t* pending) {
    if (!m || !committed || !pending) return KS_ERR_INVALID_ARG;
    *committed = m->p;
    *pending = m->pending;
    return KS_OK;
}

static int history_rows(ks_model* m, int32_t* idx) {
    int r = 0;
    const int R = m->cfg.max_rows;
    // oldest slot first: the slot after hist_next-1 going around the ring
    for (int k = 1; k <= m->lay.hist_slots; ++k) {
        const int s = (m->hist_next + k) % m->lay.hist_slots;
        for (int i = 0; i < m->slot_cnt[s]; ++i) idx[r++] = s * R + m->slot_off[s] + i;
    }
    return r;
}

// LM head + argmax of R rows whose input (x, xg, ss) is already in place.
static ks_status lm_head_rows(ks_model* m, int R, int32_t* tokens) {
    const ks_config& c = m->cfg;
    const int d = c.d_model, L = c.n_layers;
    cudaStream_t s = m->stream;
    if (m->dtype == KS_DTYPE_BF16) {
        if (!m->chain) m->chain = new ChainArgs();
        ChainArgs& ca = *m->chain;
        ca.amap[0] = m->map_xg[R - 1];
        ca.amap[1] = m->map_xg2[R - 1];
        ca.amap[2] = m->map_attn_out[R - 1];
        ca.amap[3] = m->map_act[R - 1];
        ca.R = R;
        ca.n_layers = L; ca.d = d; ca.F = c.d_ff; ca.hqd = c.n_q_heads * c.head_dim;
        ca.nqkv = (c.n_q_heads + 2 * c.n_kv_heads) * c.head_dim; ca.vocab = c.vocab;
        ca.eps = c.rms_eps;
        ca.x = m->x; ca.ss = m->ss; ca.xg = m->xg; ca.qkv = m->qkv;
        ca.act = reinterpret_cast<__nv_bfloat16*>(m->act);
        ca.logits = m->logits; ca.best = m->best; ca.tokens = tokens;
        ca.capture = nullptr;
        ca.err = m->err;
        ca.stop = nullptr;
        ca.slice_part = m->slice_part;
        ca.slice_ticket = m->slice_ticket;
        ca.n_phases = 1;
        ca.code[0] = (uint16_t)(4 * L);
        ca.gain[0] = nullptr;
        ca.wmap[0] = m->map_lm;
        ca.counters = m->chain_ctr + (size_t)m->chain_parity * chain_counter_ints();
        m->chain_parity ^= 1;
        return launch(m, K_LMHEAD, [&] { return launch_chain(ca, s); }, "tpt lm-head",
                      2.0 * c.vocab * (double)d);
    }
    GemvArgs g{};
    g.W = m->lm_head;
    g.dtype = m->dtype;
    g.N = c.vocab;
    g.K = d;
    g.R = R;
    g.partial = m->gemv_part;
    g.counters = m->counters;
    g.err = m->err;
    g.ss_in = m->ss;
    g.ss_groups = (d + kSsGroup - 1) / kSsGroup;
    g.eps = c.rms_eps;
    g.in = m->x;
    g.in_ld = d;
    g.norm_gain = m->final_norm;
    g.logits = m->logits;
    g.logits_ld = c.vocab;
    g.amax_val = m->amax_val;
    g.amax_idx = m->amax_idx;
    g.tokens = tokens;
    gemv_plan(g, EPI_LMHEAD);
    return launch(m, K_LMHEAD, [&] { return launch_gemv(m->dtype, EPI_LMHEAD, g, s); }, "tpt lm-head");
}

static ks_status history_sims(ks_model* m, int* rows_out);

// The TPT stage on the device (results stay in tpt_* and mask_dev).
static ks_status tpt_stage(ks_model* m, const ks_latency* lat, int K, int D, int* rows_out) {
    const ks_config& c = m->cfg;
    const int nsub = m->nsub, d = c.d_model;
    int r = 0;
    KS_TRY(history_sims(m, &r));
    // frontier: the knapsack over the whole weight sum, backtracked at K budgets
    KS_TRY(launch(m, K_ACCEPT, [&] {
        return launch_select(lat, m->sims, m->p, nsub, 0, 1.0, m->mask_dev, m->obj_dev, m->wts_dev,
                             m->wts_dev + nsub, m->select, kSelectCap, m->stream, K, m->tpt_masks);
    }, "tpt frontier"));
    // predictions of every candidate (and of the full set) on every history row
    const int total = (K + 1) * r;
    const int64_t plane = (int64_t)m->lay.hist_slots * c.max_rows * d;
    const bool bf = m->dtype == KS_DTYPE_BF16;
    for (int row0 = 0; row0 < total; row0 += c.max_rows) {
        const int B = std::min(c.max_rows, total - row0);
        KS_TRY(launch(m, K_EMBED, [&]() -> cudaError_t {
            if (bf)
                tpt_states_kernel<__nv_bfloat16><<<dim3(B, (d + 255) / 256), 256, 0, m->stream>>>(
                    hist_plane(m, 0), plane, m->hist_idx, r, row0, nsub, m->tpt_masks, K, d,
                    reinterpret_cast<const __nv_bfloat16*>(m->final_norm), m->x, m->ss, m->xg);
            else
                tpt_states_kernel<float><<<dim3(B, (d + 255) / 256), 256, 0, m->stream>>>(
                    hist_plane(m, 0), plane, m->hist_idx, r, row0, nsub, m->tpt_masks, K, d,
                    reinterpret_cast<const float*>(m->final_norm), m->x, m->ss, nullptr);
            return cudaGetLastError();
        }, "tpt states"));
        KS_TRY(lm_head_rows(m, B, m->tpt_tok + row0));
    }
    KS_TRY(launch(m, K_ACCEPT, [&] {
        return launch_tpt(lat, m->p, nsub, c.n_layers, K, r, D, m->tpt_masks, m->tpt_tok, m->mask_dev,
                          m->tpt_info, m->tpt_out, m->stream);
    }, "tpt grid"));
    if (rows_out) *rows_out = r;
    return KS_OK;
}

// a4 on the history rows (their indices uploaded to hist_idx) into sims.
static ks_status history_cosines(ks_model* m, float* sims, int* rows_out) {
    int32_t* hidx = m->h_buf + m->cfg.max_seq + 4 * m->cfg.max_rows + 16;
    const int r = history_rows(m, hidx);
    if (r < 1) {
        set_error("history similarities: empty history");
        return KS_ERR_STATE;
    }
    KS_CUDA(cudaMemcpyAsync(m->hist_idx, hidx, sizeof(int32_t) * r, cudaMemcpyHostToDevice, m->stream),
            "history index upload");
    m->h2d += sizeof(int32_t) * r;
    const int d = m->cfg.d_model;
    const int64_t plane = (int64_t)m->lay.hist_slots * m->cfg.max_rows * d;
    cudaError_t e = launch_cosine(hist_plane(m, 0), hist_plane(m, 1), KS_DTYPE_F32, m->nsub, r, d, plane,
                                  m->hist_idx, sims, m->stream);
    if (e != cudaSuccess) return cuda_fail(e, "history cosine");
    m->launches++;
    if (rows_out) *rows_out = r;
    return KS_OK;
}

static ks_status history_sims(ks_model* m, int* rows_out) { return history_cosines(m, m->sims, rows_out); }

ks_status ks_history_similarities(ks_model* m, float* sims, int32_t* rows_used) {
    if (!m || !sims) {
        set_error("ks_history_similarities: null argument");
        return KS_ERR_INVALID_ARG;
    }
    if (!m->have_seq) {
        set_error("ks_history_similarities: no sequence");
        return KS_ERR_STATE;
    }
    int r = 0;
    KS_TRY(history_cosines(m, sims, &r));
    if (rows_used) *rows_used = r;
    return KS_OK;
}

static bool latency_ok(const ks_latency& lat, int nsub, int64_t context_len) {
    return latency_valid(&lat, nsub, context_len);
}

ks_status ks_select_tpt(ks_model* m, const ks_latency* lat, int32_t n_candidates, int32_t max_gamma,
                        uint8_t* mask_out, int32_t* gamma_out, double* tpt_out, double* alphas_out,
                        uint8_t* candidates_out) {
    if (!m || !lat || !mask_out || !gamma_out || !tpt_out) {
        set_error("ks_select_tpt: null argument");
        return KS_ERR_INVALID_ARG;
    }
    if (n_candidates < 1 || n_candidates > KS_TPT_MAX_CANDIDATES || max_gamma < 1 ||
        max_gamma >= m->cfg.max_rows || !latency_ok(*lat, m->nsub, m->p)) {
        set_error("ks_select_tpt: bad argument");
        return KS_ERR_INVALID_ARG;
    }
    if (!m->have_seq) {
        set_error("ks_select_tpt: no sequence (call ks_prefill first)");
        return KS_ERR_STATE;
    }
    KS_TRY(tpt_stage(m, lat, n_candidates, max_gamma, nullptr));
    const int nsub = m->nsub;
    std::vector<double> out(1 + n_candidates);
    int32_t info[2] = {0, 0};
    KS_CUDA(cudaMemcpyAsync(mask_out, m->mask_dev, nsub, cudaMemcpyDeviceToHost, m->stream), "tpt download");
    KS_CUDA(cudaMemcpyAsync(info, m->tpt_info, sizeof(info), cudaMemcpyDeviceToHost, m->stream), "tpt download");
    KS_CUDA(cudaMemcpyAsync(out.data(), m->tpt_out, sizeof(double) * out.size(), cudaMemcpyDeviceToHost, m->stream),
            "tpt download");
    if (candidates_out)
        KS_CUDA(cudaMemcpyAsync(candidates_out, m->tpt_masks, (size_t)n_candidates * nsub, cudaMemcpyDeviceToHost,
                                m->stream),
                "tpt download");
    m->d2h += nsub + sizeof(info) + sizeof(double) * out.size() + (candidates_out ? n_candidates * nsub : 0);
    KS_TRY(sync(m, "ks_select_tpt"));
    *gamma_out = info[1];
    *tpt_out = out[0];
    if (alphas_out)
        for (int j = 0; j < n_candidates; ++j) alphas_out[j] = out[1 + j];
    return KS_OK;
}

// ----------------------------------------------- hidden-state DP (Alg. 1)
// Scratch of ks_select_dp, in this order (256-byte aligned pieces):
//   G0, G1, E: [S][rows][d] fp32 (states of the previous / current sublayer,
//   execute candidates); sig_e, sig_s, sig: [S] fp32; valid0, valid1, src,
//   js: [S] int; n_cand: int; w: [2L] int; choices: [2L][S] u8;
//   kv: K and V of one layer at the history positions, [2][hk][rows][hd] in
//   the model dtype; masks: [S][2L] u8; pred: [S + 1][rows] int;
//   tpt: info[2] int, out[1 + S] double, mask_out[2L] u8.
struct DpScratch {
    float *G0, *G1, *E, *sig_e, *sig_s, *sig;
    int *valid0, *valid1, *src, *js, *n_cand, *w, *pred, *info;
    uint8_t *choices, *masks, *mask_out;
    void* kv;
    double* out;
    size_t bytes;
};

static DpScratch dp_layout(const ks_model* m, int S, int rows, char* base) {
    const ks_config& c = m->cfg;
    const int nsub = 2 * c.n_layers, d = c.d_model;
    size_t off = 0;
    auto take = [&](size_t n) {
        const size_t o = off;
        off += align_up(n, 256);
        return base ? base + o : nullptr;
    };
    DpScratch D{};
    const size_t st = sizeof(float) * (size_t)S * rows * d;
    D.G0 = reinterpret_cast<float*>(take(st));
    D.G1 = reinterpret_cast<float*>(take(st));
    D.E = reinterpret_cast<float*>(take(st));
    D.sig_e = reinterpret_cast<float*>(take(sizeof(float) * S));
    D.sig_s = reinterpret_cast<float*>(take(sizeof(float) * S));
    D.sig = reinterpret_cast<float*>(take(sizeof(float) * S));
    D.valid0 = reinterpret_cast<int*>(take(sizeof(int) * S));
    D.valid1 = reinterpret_cast<int*>(take(sizeof(int) * S));
    D.src = reinterpret_cast<int*>(take(sizeof(int) * S));
    D.js = reinterpret_cast<int*>(take(sizeof(int) * S));
    D.n_cand = reinterpret_cast<int*>(take(sizeof(int)));
    D.w = reinterpret_cast<int*>(take(sizeof(int) * nsub));
    D.choices = reinterpret_cast<uint8_t*>(take((size_t)nsub * S));
    D.kv = take(2 * (size_t)c.n_kv_heads * rows * c.head_dim * m->es);
    D.masks = reinterpret_cast<uint8_t*>(take((size_t)S * nsub));
    D.pred = reinterpret_cast<int*>(take(sizeof(int) * (size_t)(S + 1) * rows));
    D.info = reinterpret_cast<int*>(take(sizeof(int) * 2));
    D.out = reinterpret_cast<double*>(take(sizeof(double) * (1 + (size_t)S)));
    D.mask_out = reinterpret_cast<uint8_t*>(take((size_t)nsub));
    D.bytes = off;
    return D;
}

size_t ks_dp_scratch_bytes(const ks_model* m, int32_t max_states, int32_t max_rows) {
    if (!m || max_states < 1 || max_states > kDpMaxStates || max_rows < 1) return 0;
    return dp_layout(m, max_states, max_rows, nullptr).bytes;
}

// Integer weights of Sec. 3.4 (the knapsack kernel's rule): Delta = min(t_Attn(n),
// t_MLP), w = round(t / Delta) half away from zero, at least 1; units as given.
static void dp_weights(const ks_latency& lat, int64_t n, int nsub, std::vector<int>& w) {
    w.assign(nsub, 1);
    if (lat.kind == 1) {
        for (int i = 0; i < nsub; ++i) w[i] = lat.units[i];
        return;
    }
    volatile double prod = lat.c2 * (double)n;   // two roundings, as the device evaluates c2 n + c3
    const double ta = prod + lat.c3, tm = lat.c1;
    const double delta = std::min(ta, tm);
    const int wa = std::max(1, (int)std::llround(ta / delta)), wm = std::max(1, (int)std::llround(tm / delta));
    for (int i = 0; i < nsub; ++i) w[i] = (i % 2 == 0) ? wa : wm;
}

ks_status ks_select_dp(ks_model* m, const ks_latency* lat, float tau, int32_t max_gamma, int32_t max_states,
                       int32_t max_rows, void* scratch, size_t scratch_bytes, uint8_t* mask_out, int32_t* gamma_out,
                       double* tpt_out, int32_t* n_candidates, int32_t* js_out, double* alphas_out,
                       uint8_t* candidates_out) {
    if (!m || !lat || !scratch || !mask_out || !gamma_out || !tpt_out) {
        set_error("ks_select_dp: null argument");
        return KS_ERR_INVALID_ARG;
    }
    const ks_config& c = m->cfg;
    const int nsub = m->nsub, d = c.d_model, L = c.n_layers;
    if (max_gamma < 1 || max_gamma >= c.max_rows || max_states < 1 || max_states > kDpMaxStates || max_rows < 1 ||
        !std::isfinite(tau) || !latency_ok(*lat, nsub, m->p)) {
        set_error("ks_select_dp: bad argument");
        return KS_ERR_INVALID_ARG;
    }
    if (!m->have_seq) {
        set_error("ks_select_dp: no sequence (call ks_prefill first)");
        return KS_ERR_STATE;
    }
    DpScratch D = dp_layout(m, max_states, max_rows, reinterpret_cast<char*>(scratch));
    if (scratch_bytes < D.bytes || (reinterpret_cast<uintptr_t>(scratch) & 255)) {
        set_error("ks_select_dp: scratch smaller than ks_dp_scratch_bytes or not 256-byte aligned");
        return KS_ERR_WORKSPACE;
    }
    std::vector<int> w;
    dp_weights(*lat, m->p, nsub, w);
    int K = 0;
    for (int x : w) K += x;
    const int S = K / 2 + 1;   // skipped weights 0 .. K / 2
    if (S > max_states) {
        set_error("ks_select_dp: %d states (K = %d) exceed max_states %d", S, K, max_states);
        return KS_ERR_CAPACITY;
    }
    // history rows: the last r committed positions, oldest first
    int32_t* hidx = m->h_buf + c.max_seq + 4 * c.max_rows + 16;
    int r = history_rows(m, hidx);
    if (r < 1) {
        set_error("ks_select_dp: empty history");
        return KS_ERR_STATE;
    }
    if (r > max_rows) {   // keep the most recent max_rows rows
        std::memmove(hidx, hidx + (r - max_rows), sizeof(int32_t) * max_rows);
        r = max_rows;
    }
    const int p0 = m->p - r;
    cudaStream_t s = m->stream;
    KS_CUDA(cudaMemcpyAsync(m->hist_idx, hidx, sizeof(int32_t) * r, cudaMemcpyHostToDevice, s), "dp upload");
    int32_t* hw = m->h_buf + c.max_seq + 4 * c.max_rows + 16 + m->lay.hist_slots * c.max_rows + (nsub + 3) / 4 + 4;
    std::memcpy(hw, w.data(), sizeof(int) * nsub);
    KS_CUDA(cudaMemcpyAsync(D.w, hw, sizeof(int) * nsub, cudaMemcpyHostToDevice, s), "dp upload");
    m->h2d += sizeof(int32_t) * (r + nsub);
    const long long stride = (long long)r * d;
    float *Gp = D.G0, *Gc = D.G1;
    int *vp = D.valid0, *vc = D.valid1;
    // g[0, 0] = X^(0); every other state starts invalid
    {
        std::vector<int> ones(S, 1);
        ones[0] = 0;
        int32_t* hv = hw + nsub;
        std::memcpy(hv, ones.data(), sizeof(int) * S);
        KS_CUDA(cudaMemcpyAsync(vp, hv, sizeof(int) * S, cudaMemcpyHostToDevice, s), "dp init");
        ones[0] = -1;
        std::memcpy(hv + S, ones.data(), sizeof(int) * S);
        KS_CUDA(cudaMemcpyAsync(D.src, hv + S, sizeof(int) * S, cudaMemcpyHostToDevice, s), "dp init");
        KS_TRY(launch(m, K_ACCEPT, [&] {
            return launch_dp_gather(S, D.src, vp, D.E, Gp, stride, hist_plane(m, 0), m->hist_idx, r, d, Gp, s);
        }, "dp init"));
    }
    const size_t kv_row = (size_t)c.head_dim * m->es;
    const size_t kv_plane = (size_t)c.n_kv_heads * r * kv_row;
    std::vector<uint8_t> one(nsub, 0);
    for (int i = 1; i <= nsub; ++i) {
        const bool attn = (i % 2) == 1;
        const int l = (i - 1) / 2;
        std::fill(one.begin(), one.end(), 0);
        one[i - 1] = 1;
        char* kc = reinterpret_cast<char*>(kcache(m, l));
        char* vcach = reinterpret_cast<char*>(vcache(m, l));
        char* kvs = reinterpret_cast<char*>(D.kv);
        const size_t seq_pitch = (size_t)c.max_seq * kv_row;
        if (attn) {   // the target's K/V at the history positions, restored after every state
            KS_CUDA(cudaMemcpy2DAsync(kvs, r * kv_row, kc + (size_t)p0 * kv_row, seq_pitch, r * kv_row, c.n_kv_heads,
                                      cudaMemcpyDeviceToDevice, s), "dp kv save");
            KS_CUDA(cudaMemcpy2DAsync(kvs + kv_plane, r * kv_row, vcach + (size_t)p0 * kv_row, seq_pitch, r * kv_row,
                                      c.n_kv_heads, cudaMemcpyDeviceToDevice, s), "dp kv save");
        }
        for (int j = 1; j < S; ++j) {
            for (int c0 = 0; c0 < r; c0 += c.max_rows) {
                const int R = std::min(c.max_rows, r - c0);
                KS_CUDA(cudaMemcpyAsync(m->x, Gp + (size_t)j * stride + (size_t)c0 * d, sizeof(float) * R * d,
                                        cudaMemcpyDeviceToDevice, s), "dp state in");
                KS_TRY(forward(m, nullptr, R, p0 + c0, one.data(), -1, nullptr, vp + j));
                KS_CUDA(cudaMemcpyAsync(D.E + (size_t)j * stride + (size_t)c0 * d, m->x, sizeof(float) * R * d,
                                        cudaMemcpyDeviceToDevice, s), "dp state out");
            }
            if (attn) {
                KS_CUDA(cudaMemcpy2DAsync(kc + (size_t)p0 * kv_row, seq_pitch, kvs, r * kv_row, r * kv_row,
                                          c.n_kv_heads, cudaMemcpyDeviceToDevice, s), "dp kv restore");
                KS_CUDA(cudaMemcpy2DAsync(vcach + (size_t)p0 * kv_row, seq_pitch, kvs + kv_plane, r * kv_row,
                                          r * kv_row, c.n_kv_heads, cudaMemcpyDeviceToDevice, s), "dp kv restore");
            }
        }
        const float* X = hist_plane(m, i);
        KS_TRY(launch(m, K_ACCEPT, [&] { return launch_dp_cos(D.E, stride, S, X, m->hist_idx, r, d, D.sig_e, s); },
                      "dp cosines"));
        KS_TRY(launch(m, K_ACCEPT, [&] { return launch_dp_cos(Gp, stride, S, X, m->hist_idx, r, d, D.sig_s, s); },
                      "dp cosines"));
        KS_TRY(launch(m, K_ACCEPT, [&] {
            return launch_dp_select(S, w[i - 1], tau, vp, D.sig_e, D.sig_s, vc, D.sig, D.choices + (size_t)(i - 1) * S,
                                    D.src, s);
        }, "dp select"));
        KS_TRY(launch(m, K_ACCEPT, [&] {
            return launch_dp_gather(S, D.src, vc, D.E, Gp, stride, X, m->hist_idx, r, d, Gc, s);
        }, "dp gather"));
        std::swap(Gp, Gc);
        std::swap(vp, vc);
    }
    // terminal candidates, executed weight ascending
    KS_TRY(launch(m, K_ACCEPT, [&] { return launch_dp_candidates(S, vp, D.js, D.n_cand, s); }, "dp candidates"));
    int32_t* hc = hw + nsub;
    KS_CUDA(cudaMemcpyAsync(hc, D.n_cand, sizeof(int), cudaMemcpyDeviceToHost, s), "dp candidates");
    KS_CUDA(cudaMemcpyAsync(hc + 1, D.js, sizeof(int) * S, cudaMemcpyDeviceToHost, s), "dp candidates");
    m->d2h += sizeof(int) * (1 + S);
    KS_TRY(sync(m, "ks_select_dp"));
    const int n_cand = hc[0];
    std::vector<int> js(hc + 1, hc + 1 + n_cand);
    if (n_cand < 1) {
        set_error("ks_select_dp: no state survived the pruning (tau %g)", (double)tau);
        return KS_ERR_STATE;
    }
    KS_TRY(launch(m, K_ACCEPT, [&] {
        return launch_dp_backtrack(D.js, n_cand, nsub, S, D.choices, D.w, D.masks, s);
    }, "dp backtrack"));
    // Eq. 4 inputs: the LM head's argmax of every terminal state's rows and of X^(2L)
    for (int cnd = 0; cnd <= n_cand; ++cnd) {
        for (int c0 = 0; c0 < r; c0 += c.max_rows) {
            const int R = std::min(c.max_rows, r - c0);
            if (cnd < n_cand) {
                KS_CUDA(cudaMemcpyAsync(m->x, Gp + (size_t)js[cnd] * stride + (size_t)c0 * d, sizeof(float) * R * d,
                                        cudaMemcpyDeviceToDevice, s), "dp prediction rows");
            } else {   // the target's rows X^(2L) (gathered like state 0 of sublayer 2L)
                KS_CUDA(cudaMemcpyAsync(m->x, Gp + (size_t)c0 * d, sizeof(float) * R * d, cudaMemcpyDeviceToDevice,
                                        s), "dp prediction rows");
            }
            KS_TRY(launch(m, K_EMBED, [&]() -> cudaError_t {
                if (m->dtype == KS_DTYPE_BF16)
                    rows_prep_kernel<__nv_bfloat16><<<dim3(R, (d + 255) / 256), 256, 0, s>>>(
                        m->x, d, m->ss, m->xg, reinterpret_cast<const __nv_bfloat16*>(m->final_norm), nullptr);
                else
                    rows_prep_kernel<float><<<dim3(R, (d + 255) / 256), 256, 0, s>>>(m->x, d, m->ss, nullptr, nullptr,
                                                                                      nullptr);
                return cudaGetLastError();
            }, "dp prediction prep"));
            KS_TRY(lm_head_rows(m, R, D.pred + (size_t)cnd * r + c0));
        }
    }
    KS_TRY(launch(m, K_ACCEPT, [&] {
        return launch_tpt(lat, m->p, nsub, L, n_cand, r, max_gamma, D.masks, D.pred, D.mask_out, D.info, D.out, s);
    }, "dp tpt grid"));
    std::vector<double> outv(1 + n_cand);
    int32_t info[2] = {0, 0};
    KS_CUDA(cudaMemcpyAsync(mask_out, D.mask_out, nsub, cudaMemcpyDeviceToHost, s), "dp download");
    KS_CUDA(cudaMemcpyAsync(info, D.info, sizeof(info), cudaMemcpyDeviceToHost, s), "dp download");
    KS_CUDA(cudaMemcpyAsync(outv.data(), D.out, sizeof(double) * outv.size(), cudaMemcpyDeviceToHost, s),
            "dp download");
    if (candidates_out)
        KS_CUDA(cudaMemcpyAsync(candidates_out, D.masks, (size_t)n_cand * nsub, cudaMemcpyDeviceToHost, s),
                "dp download");
    m->d2h += nsub + sizeof(info) + sizeof(double) * outv.size() + (candidates_out ? (size_t)n_cand * nsub : 0);
    KS_TRY(sync(m, "ks_select_dp"));
    *gamma_out = info[1];
    *tpt_out = outv[0];
    if (n_candidates) *n_candidates = n_cand;
    if (js_out)
        for (int k = 0; k < n_cand; ++k) js_out[k] = js[k];
    if (alphas_out)
        for (int k = 0; k < n_cand; ++k) alphas_out[k] = outv[1 + k];
    return KS_OK;
}

ks_status ks_generate_speculative(ks_model* m, const ks_spec_params* prm, int32_t n_tokens, int32_t* out,
                                  ks_spec_stats* stats, int32_t* accepted_per_step) {
    if (!m || !prm || !out || n_tokens < 1) {
        set_error("ks_generate_speculative: bad argument");
        return KS_ERR_INVALID_ARG;
    }
    if (!m->have_seq) {
        set_error("ks_generate_speculative: no sequence (call ks_prefill first)");
        return KS_ERR_STATE;
    }
    const int nsub = m->nsub;
    if (prm->gamma < 1 || prm->gamma >= m->cfg.max_rows || prm->policy < 0 || prm->policy > 3 ||
        (prm->policy == 0 && !prm->mask) ||
        (prm->policy == 1 && (prm->resolve_every < 1 || !(prm->budget_frac >= 0.0) || prm->budget_frac > 1.0)) ||
        (prm->policy == 2 && (prm->resolve_every < 1 || prm->tpt_candidates < 1 ||
                              prm->tpt_candidates > KS_TPT_MAX_CANDIDATES || prm->tpt_max_gamma < 1 ||
                              prm->tpt_max_gamma >= m->cfg.max_rows)) ||
        (prm->policy == 3 && (prm->resolve_every < 1 || !prm->dp_scratch || prm->tpt_max_gamma < 1 ||
                              prm->tpt_max_gamma >= m->cfg.max_rows))) {
        set_error("ks_generate_speculative: bad parameters");
        return KS_ERR_INVALID_ARG;
    }
    if (!(prm->tau_conf >= 0.0) || !std::isfinite(prm->tau_conf)) {
        set_error("ks_generate_speculative: tau_conf must be finite and >= 0");
        return KS_ERR_INVALID_ARG;
    }
    const bool sampling = prm->sampling.temperature != 0.f;
    if (sampling && (!sampling_ok(&prm->sampling) || prm->tau_conf > 0.0)) {
        set_error("ks_generate_speculative: sampling needs temperature > 0, top_k >= 1, 0 < top_p <= 1 "
                  "and no dynamic exit");
        return KS_ERR_INVALID_ARG;
    }
    if (prm->policy != 0 && !latency_ok(prm->latency, nsub, m->p)) {
        set_error("ks_generate_speculative: bad latency model");
        return KS_ERR_INVALID_ARG;
    }
    ks_spec_stats st{};
    std::vector<uint8_t> mask(nsub, 1);
    if (prm->policy == 0) std::memcpy(mask.data(), prm->mask, nsub);
    int n = 0;
    out[n++] = m->pending;
    std::vector<int32_t> toks(m->cfg.max_rows + 1);
    int gamma = prm->gamma;
    while (n < n_tokens && (prm->max_steps <= 0 || st.steps < prm->max_steps)) {
        if (prm->policy != 0 && st.steps % prm->resolve_every == 0 && !latency_ok(prm->latency, nsub, m->p)) {
            set_error("ks_generate_speculative: latency model invalid at context %d", m->p);
            return KS_ERR_INVALID_ARG;
        }
        if (prm->policy == 2 && st.steps % prm->resolve_every == 0) {
            // TPT stage: the next mask and draft length
            KS_TRY(tpt_stage(m, &prm->latency, prm->tpt_candidates, prm->tpt_max_gamma, nullptr));
            uint8_t* hm = reinterpret_cast<uint8_t*>(m->h_buf + m->cfg.max_seq + 4 * m->cfg.max_rows + 16 +
                                                     m->lay.hist_slots * m->cfg.max_rows);
            int32_t* hg = m->h_buf + m->cfg.max_seq;
            KS_CUDA(cudaMemcpyAsync(hm, m->mask_dev, nsub, cudaMemcpyDeviceToHost, m->stream), "mask download");
            KS_CUDA(cudaMemcpyAsync(hg, m->tpt_info, sizeof(int32_t) * 2, cudaMemcpyDeviceToHost, m->stream),
                    "gamma download");
            m->d2h += nsub + 2 * sizeof(int32_t);
            KS_TRY(sync(m, "select"));
            std::memcpy(mask.data(), hm, nsub);
            gamma = hg[1];
            st.resolves++;
        }
        if (prm->policy == 3 && st.steps % prm->resolve_every == 0) {
            // Alg. 1 + the Eq. 3 grid: the next mask and draft length
            int32_t gsel = 0;
            double tsel = 0.0;
            KS_TRY(ks_select_dp(m, &prm->latency, prm->dp_tau, prm->tpt_max_gamma, prm->dp_max_states,
                                prm->dp_max_rows, prm->dp_scratch, (size_t)prm->dp_scratch_bytes, mask.data(),
                                &gsel, &tsel, nullptr, nullptr, nullptr, nullptr));
            gamma = gsel;
            st.resolves++;
        }
        if (prm->policy == 1 && st.steps % prm->resolve_every == 0) {
            KS_TRY(ks_history_similarities(m, m->sims, nullptr));
            KS_TRY(launch(m, K_ACCEPT, [&] {
                return launch_select(&prm->latency, m->sims, m->p, nsub, 0, prm->budget_frac, m->mask_dev, m->obj_dev,
                                     m->wts_dev, m->wts_dev + nsub, m->select, kSelectCap, m->stream);
            }, "select"));
            uint8_t* hm = reinterpret_cast<uint8_t*>(m->h_buf + m->cfg.max_seq + 4 * m->cfg.max_rows + 16 +
                                                     m->lay.hist_slots * m->cfg.max_rows);
            KS_CUDA(cudaMemcpyAsync(hm, m->mask_dev, nsub, cudaMemcpyDeviceToHost, m->stream), "mask download");
            m->d2h += nsub;
            KS_TRY(sync(m, "select"));
            std::memcpy(mask.data(), hm, nsub);
            st.resolves++;
        }
        int g = gamma;
        if (m->p + g + 1 > m->cfg.max_seq) g = m->cfg.max_seq - m->p - 1;
        if (g < 1) {
            set_error("ks_generate_speculative: KV capacity exhausted");
            return KS_ERR_CAPACITY;
        }
        int32_t a = 0, no = 0;
        if (sampling) {
            const unsigned long long step = (unsigned long long)st.steps;
            KS_TRY(ks_draft_sample(m, mask.data(), g, &prm->sampling, step, nullptr));
            KS_TRY(ks_verify_sample(m, g, &prm->sampling, step, &a, toks.data(), &no));
        } else {
            if (prm->tau_conf > 0.0)
                KS_TRY(ks_draft_dynamic(m, mask.data(), g, (float)prm->tau_conf, nullptr, nullptr, nullptr));
            else
                KS_TRY(ks_draft(m, mask.data(), g, nullptr));
            KS_TRY(ks_verify(m, nullptr, g, &a, toks.data(), &no));
        }
        if (accepted_per_step) accepted_per_step[st.steps] = a;
        st.steps++;
        st.drafted += m->last_scored;
        st.accepted += a;
        for (int i = 0; i < no && n < n_tokens; ++i) out[n++] = toks[i];
    }
    int na = 0, nm = 0;
    for (int i = 0; i < nsub; ++i)
        if (!mask[i]) (i % 2 == 0 ? na : nm)++;
    st.attn_skipped = na;
    st.mlp_skipped = nm;
    if (stats) *stats = st;
    return KS_OK;
}

ks_status ks_debug_set_status(ks_model* m, int32_t code) {
    if (!m || code < 0 || code > 5) {
        set_error("ks_debug_set_status: bad argument");
        return KS_ERR_INVALID_ARG;
    }
    KS_CUDA(cudaStreamSynchronize(m->stream), "debug status");
    KS_CUDA(cudaMemcpy(m->err, &code, sizeof(int32_t), cudaMemcpyHostToDevice), "debug status");
    return KS_OK;
}

ks_status ks_debug_read(ks_model* m, int32_t what, int32_t layer, int32_t start, int32_t count, void* dst,
                        size_t bytes) {
    if (!m || !dst) return KS_ERR_INVALID_ARG;
    const ks_config& c = m->cfg;
    cudaStream_t s = m->stream;
    KS_TRY(sync(m, "debug sync"));
    if (what == 0 || what == 1) {
        const size_t row = what == 0 ? (size_t)c.vocab : (size_t)c.d_model;
        if (count < 1 || count > c.max_rows || bytes < row * count * sizeof(float)) return KS_ERR_INVALID_ARG;
        KS_CUDA(cudaMemcpy(dst, what == 0 ? m->logits : m->x, row * count * sizeof(float), cudaMemcpyDeviceToHost),
                "debug read");
        return KS_OK;
    }
    if (what == 2 || what == 3) {
        if (layer < 0 || layer >= c.n_layers || start < 0 || count < 1 || start + count > c.max_seq) return KS_ERR_INVALID_ARG;
        const size_t rowb = (size_t)c.head_dim * m->es;
        if (bytes < rowb * count * c.n_kv_heads) return KS_ERR_INVALID_ARG;
        const char* base = reinterpret_cast<const char*>(what == 2 ? kcache(m, layer) : vcache(m, layer));
        KS_CUDA(cudaMemcpy2DAsync(dst, rowb * count, base + (size_t)start * rowb, rowb * c.max_seq, rowb * count,
                                  c.n_kv_heads, cudaMemcpyDeviceToHost, s),
                "debug kv read");
        return sync(m, "debug kv read");
    }
    if (what == 5 || what == 6) {
        // sampling distributions: per slot n, ids[kSampleMaxK], probs[kSampleMaxK] (int32, int32, float)
        if (start < 0 || count < 1 || start + count > c.max_rows ||
            bytes < sizeof(int32_t) * (size_t)count * (1 + 2 * kSampleMaxK))
            return KS_ERR_INVALID_ARG;
        const int* ids = what == 5 ? m->q_ids : m->p_ids;
        const float* pr = what == 5 ? m->q_probs : m->p_probs;
        const int* n = what == 5 ? m->q_n : m->p_n;
        std::vector<int32_t> hn(count), hi((size_t)count * kSampleMaxK);
        std::vector<float> hp((size_t)count * kSampleMaxK);
        KS_CUDA(cudaMemcpy(hn.data(), n + start, sizeof(int32_t) * count, cudaMemcpyDeviceToHost), "debug read");
        KS_CUDA(cudaMemcpy(hi.data(), ids + (size_t)start * kSampleMaxK, sizeof(int32_t) * hi.size(),
                           cudaMemcpyDeviceToHost), "debug read");
        KS_CUDA(cudaMemcpy(hp.data(), pr + (size_t)start * kSampleMaxK, sizeof(float) * hp.size(),
                           cudaMemcpyDeviceToHost), "debug read");
        int32_t* out = reinterpret_cast<int32_t*>(dst);
        for (int r = 0; r < count; ++r) {
            int32_t* o = out + (size_t)r * (1 + 2 * kSampleMaxK);
            o[0] = hn[r];
            std::memcpy(o + 1, hi.data() + (size_t)r * kSampleMaxK, sizeof(int32_t) * kSampleMaxK);
            std::memcpy(o + 1 + kSampleMaxK, hp.data() + (size_t)r * kSampleMaxK, sizeof(float) * kSampleMaxK);
        }
        return KS_OK;
    }
    if (what == 4) {
        std::vector<int32_t> idx(m->lay.hist_slots * c.max_rows);
        const int r = history_rows(m, idx.data());
        if (count == 0) {  // query the row count
            if (bytes < sizeof(int32_t)) return KS_ERR_INVALID_ARG;
            *reinterpret_cast<int32_t*>(dst) = r;
            return KS_OK;
        }
        if (count != r) return KS_ERR_INVALID_ARG;
        const size_t need = sizeof(float) * (size_t)(m->nsub + 1) * r * c.d_model;
        if (bytes < need) return KS_ERR_INVALID_ARG;
        float* o = reinterpret_cast<float*>(dst);
        for (int pl = 0; pl <= m->nsub; ++pl)
            for (int i = 0; i < r; ++i)
                KS_CUDA(cudaMemcpy(o + ((size_t)pl * r + i) * c.d_model, hist_plane(m, pl) + (size_t)idx[i] * c.d_model,
                                   sizeof(float) * c.d_model, cudaMemcpyDeviceToHost),
                        "debug history read");
        return KS_OK;
    }
    return KS_ERR_INVALID_ARG;
}

ks_status ks_kernel_timing(ks_model* m, int32_t klass, int32_t enable) {
    if (!m || klass < 0 || klass >= kKlasses) return KS_ERR_INVALID_ARG;
    KS_TRY(sync(m, "timing"));
    m->timing[klass].on = enable != 0;
    m->timing[klass].used = 0;
    m->timing[klass].bytes = 0.0;
    return KS_OK;
}

ks_status ks_kernel_bytes(const ks_model* m, int32_t klass, double* bytes) {
    if (!m || klass < 0 || klass >= kKlasses || !bytes) return KS_ERR_INVALID_ARG;
    *bytes = m->timing[klass].bytes;
    return KS_OK;
}

ks_status ks_kernel_time(ks_model* m, int32_t klass, int64_t* launches, double* total_ms) {
    if (!m || klass < 0 || klass >= kKlasses || !launches || !total_ms) return KS_ERR_INVALID_ARG;
    KS_TRY(sync(m, "timing"));
    KlassTiming& T = m->timing[klass];
    double tot = 0.0;
    for (size_t i = 0; i < T.used; i += 2) {
        float ms = 0.f;
        KS_CUDA(cudaEventElapsedTime(&ms, T.ev[i], T.ev[i + 1]), "cudaEventElapsedTime");
        tot += ms;
    }
    *launches = (int64_t)(T.used / 2);
    *total_ms = tot;
    return KS_OK;
}

int64_t ks_launch_count(const ks_model* m) { return m ? m->launches : -1; }

ks_status ks_transfer_bytes(const ks_model* m, int64_t* h2d, int64_t* d2h) {
    if (!m || !h2d || !d2h) return KS_ERR_INVALID_ARG;
    *h2d = m->h2d;
    *d2h = m->d2h;
    return KS_OK;
}

}  // extern "C"
