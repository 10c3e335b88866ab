// Plain fp32 CPU oracle of the KnapSpec hot path, single-threaded C++.
// TEST INFRASTRUCTURE ONLY: called by tests/, __graft_entry__.smoke() and the
// bench's CPU baseline, never by the library; it shares no code with the CUDA
// path.  Every loop is the textbook definition, in fp32, with no blocking,
// vectorised library or reordering beyond the order written here; the only
// double-precision steps are the ones the paper's readings fix (RoPE angles,
// latency ratios, knapsack values).
//
// Follows (arXiv 2602.20217):
//  * Sec. 2: f = composition of 2L sublayers f^(2i-1) = Attn_i, f^(2i) = MLP_i,
//    each including its normalisation; f^(S) runs only the sublayers in S,
//    a skipped sublayer being the identity on the residual stream;
//  * Sec. 2.1: greedy speculative decoding - a draft proposes gamma tokens,
//    the target scores pending + drafts in one pass, drafts are accepted while
//    they equal the target's argmax, and the target's token follows;
//  * Sec. 2 (matrix cosine) and Sec. 3.4: sigma_i = cos(X^(i-1), X^(i)) over the
//    history rows of the last m speculation steps;
//  * Sec. 3.3, 3.4 and App. C: latency model t_MLP = c1, t_Attn(n) = c2 n + c3,
//    integer weights round(t / Delta) with Delta = min(t_Attn, t_MLP), and the
//    exact 0/1 knapsack over the sublayers.
// Readings where the paper is silent: Llama/Qwen3 blocks (pre-RMSNorm, fused
// [Wq; Wk; Wv], optional per-head QK RMSNorm, rotate-half RoPE with
// inv_freq_j = theta^(-2j/hd) whose cos/sin are computed in double and rounded
// to fp32, causal GQA with scale 1/sqrt(hd), SwiGLU MLP, final RMSNorm, untied
// LM head); argmax ties go to the lowest id; item value q_i = round((1 -
// sigma_i) 2^30) (half away from zero); the knapsack takes an item only on a
// strict improvement, so the optimum with the smallest bitmask is returned.
#include <cmath>
#include <cstdint>
#include <cstdlib>
#include <cstring>
#include <deque>
#include <vector>

extern "C" {

typedef struct {
    int32_t n_layers, d_model, n_q_heads, n_kv_heads, head_dim, d_ff, vocab, qk_norm;
    float rms_eps;
    double rope_theta;
} ko_config;

// Host fp32 weights (borrowed), row-major [out][in]; per-layer arrays of L pointers.
typedef struct {
    const float* embed;       // [vocab][d]
    const float* lm_head;     // [vocab][d]
    const float* final_norm;  // [d]
    const float* const* attn_norm;   // [d]
    const float* const* w_qkv;       // [(hq + 2 hk) hd][d]
    const float* const* w_o;         // [d][hq hd]
    const float* const* q_norm;      // [hd] or null
    const float* const* k_norm;      // [hd] or null
    const float* const* mlp_norm;    // [d]
    const float* const* w_gate_up;   // [2 F][d]: gate rows, then up rows
    const float* const* w_down;      // [d][F]
} ko_weights;

}  // extern "C"

namespace {

// y[n] = sum_k W[n][k] x[k]
void matvec(const float* W, const float* x, int N, int K, float* y) {
    for (int n = 0; n < N; ++n) {
        const float* w = W + (size_t)n * K;
        float s = 0.f;
        for (int k = 0; k < K; ++k) s += w[k] * x[k];
        y[n] = s;
    }
}

// RMSNorm: x / sqrt(mean(x^2) + eps) * gain
void rms_norm(const float* x, const float* gain, int n, float eps, float* y) {
    float ss = 0.f;
    for (int i = 0; i < n; ++i) ss += x[i] * x[i];
    const float inv = 1.f / std::sqrt(ss / (float)n + eps);
    for (int i = 0; i < n; ++i) y[i] = x[i] * inv * (gain ? gain[i] : 1.f);
}

// Rotate-half RoPE of one head vector at position pos: pair (j, j + hd/2)
// rotated by pos * theta^(-2j/hd) (angle, cos and sin in double, then fp32).
void rope(float* v, int hd, int pos, double theta) {
    const int half = hd / 2;
    for (int j = 0; j < half; ++j) {
        const double ang = (double)pos * std::pow(theta, -2.0 * j / hd);
        const float c = (float)std::cos(ang), s = (float)std::sin(ang);
        const float a = v[j], b = v[j + half];
        v[j] = a * c - b * s;
        v[j + half] = b * c + a * s;
    }
}

float silu(float z) { return z / (1.f + std::exp(-z)); }

}  // namespace

extern "C" {

// f^(2l-1) on R rows x[R][d] at positions pos[R]: x += W_o GQA(RoPE(QKN(q)),
// RoPE(QKN(k)), v) with the inputs from RMSNorm(x).  The rows' K/V are written
// to the caches [hk][n_max][hd] first, so the rows see each other causally.
void ko_attn_sublayer(const ko_config* c, const ko_weights* w, int layer, float* x, int R, const int* pos,
                      float* kcache, float* vcache, int n_max) {
    const int d = c->d_model, hq = c->n_q_heads, hk = c->n_kv_heads, hd = c->head_dim, G = hq / hk;
    const int nqkv = (hq + 2 * hk) * hd;
    std::vector<float> h(d), qkv((size_t)R * nqkv), o((size_t)hq * hd), y(d), sc;
    for (int r = 0; r < R; ++r) {
        rms_norm(x + (size_t)r * d, w->attn_norm[layer], d, c->rms_eps, h.data());
        float* t = qkv.data() + (size_t)r * nqkv;
        matvec(w->w_qkv[layer], h.data(), nqkv, d, t);
        for (int hh = 0; hh < hq + hk; ++hh) {   // query heads, then key heads
            float* v = t + (size_t)hh * hd;
            if (c->qk_norm) {
                std::vector<float> tmp(v, v + hd);
                rms_norm(tmp.data(), hh < hq ? w->q_norm[layer] : w->k_norm[layer], hd, c->rms_eps, v);
            }
            rope(v, hd, pos[r], c->rope_theta);
        }
        for (int j = 0; j < hk; ++j)
            for (int e = 0; e < hd; ++e) {
                kcache[((size_t)j * n_max + pos[r]) * hd + e] = t[(size_t)(hq + j) * hd + e];
                vcache[((size_t)j * n_max + pos[r]) * hd + e] = t[(size_t)(hq + hk + j) * hd + e];
            }
    }
    const float scale = 1.f / std::sqrt((float)hd);
    for (int r = 0; r < R; ++r) {
        const float* t = qkv.data() + (size_t)r * nqkv;
        const int n = pos[r] + 1;   // keys 0 .. pos[r]
        sc.assign(n, 0.f);
        for (int qh = 0; qh < hq; ++qh) {
            const float* q = t + (size_t)qh * hd;
            const float* K = kcache + (size_t)(qh / G) * n_max * hd;
            const float* V = vcache + (size_t)(qh / G) * n_max * hd;
            float mx = -INFINITY;
            for (int k = 0; k < n; ++k) {
                float s = 0.f;
                for (int e = 0; e < hd; ++e) s += q[e] * K[(size_t)k * hd + e];
                sc[k] = s * scale;
                if (sc[k] > mx) mx = sc[k];
            }
            float sum = 0.f;
            for (int k = 0; k < n; ++k) {
                sc[k] = std::exp(sc[k] - mx);
                sum += sc[k];
            }
            float* out = o.data() + (size_t)qh * hd;
            for (int e = 0; e < hd; ++e) out[e] = 0.f;
            for (int k = 0; k < n; ++k) {
                const float p = sc[k] / sum;
                for (int e = 0; e < hd; ++e) out[e] += p * V[(size_t)k * hd + e];
            }
        }
        matvec(w->w_o[layer], o.data(), d, hq * hd, y.data());
        for (int i = 0; i < d; ++i) x[(size_t)r * d + i] += y[i];
    }
}

// f^(2l) on R rows: x += W_down(silu(W_gate h) * W_up h), h = RMSNorm(x).
void ko_mlp_sublayer(const ko_config* c, const ko_weights* w, int layer, float* x, int R) {
    const int d = c->d_model, F = c->d_ff;
    std::vector<float> h(d), gu(2 * (size_t)F), act(F), y(d);
    for (int r = 0; r < R; ++r) {
        rms_norm(x + (size_t)r * d, w->mlp_norm[layer], d, c->rms_eps, h.data());
        matvec(w->w_gate_up[layer], h.data(), 2 * F, d, gu.data());
        for (int f = 0; f < F; ++f) act[f] = silu(gu[f]) * gu[F + f];
        matvec(w->w_down[layer], act.data(), d, F, y.data());
        for (int i = 0; i < d; ++i) x[(size_t)r * d + i] += y[i];
    }
}

// logits[R][vocab] = lm_head RMSNorm_final(x); rows [row0, row1) of the LM head
// only (the rest are left untouched) - the full head is row0 = 0, row1 = vocab.
void ko_final_logits(const ko_config* c, const ko_weights* w, const float* x, int R, float* logits, int row0,
                     int row1) {
    const int d = c->d_model;
    std::vector<float> h(d);
    for (int r = 0; r < R; ++r) {
        rms_norm(x + (size_t)r * d, w->final_norm, d, c->rms_eps, h.data());
        for (int v = row0; v < row1; ++v) {
            const float* wr = w->lm_head + (size_t)v * d;
            float s = 0.f;
            for (int k = 0; k < d; ++k) s += wr[k] * h[k];
            logits[(size_t)r * c->vocab + v] = s;
        }
    }
}

int ko_argmax(const float* v, int n) {   // ties: the lowest index
    int b = 0;
    for (int i = 1; i < n; ++i)
        if (v[i] > v[b]) b = i;
    return b;
}

// Sec. 2 matrix cosine: <X, Y>_F / (||X||_F ||Y||_F) over rows x d values.
double ko_matrix_cos(const float* X, const float* Y, int rows, int d) {
    float xy = 0.f, xx = 0.f, yy = 0.f;
    for (size_t i = 0; i < (size_t)rows * d; ++i) {
        xy += X[i] * Y[i];
        xx += X[i] * X[i];
        yy += Y[i] * Y[i];
    }
    return (double)(xy / (std::sqrt(xx) * std::sqrt(yy)));
}

long long ko_round_half_away(double v) { return v < 0 ? -(long long)std::floor(-v + 0.5) : (long long)std::floor(v + 0.5); }

// Sec. 3.4 with App. C times: Delta = min(ta, tm), w = round(t / Delta) >= 1.
void ko_integer_weights(double ta, double tm, int* wa, int* wm) {
    const double delta = ta < tm ? ta : tm;
    const long long a = ko_round_half_away(ta / delta), m = ko_round_half_away(tm / delta);
    *wa = a < 1 ? 1 : (int)a;
    *wm = m < 1 ? 1 : (int)m;
}

// Sec. 3.3: maximise sum_{i in S} q_i subject to sum_{i in S} w_i <= budget.
// best[i][cap] over items 1..i, item taken only on a strict improvement;
// backtracking from item n picks the optimum with the smallest bitmask.
long long ko_knapsack(const int* w, const long long* q, int n, int budget, uint8_t* mask) {
    std::vector<std::vector<long long>> best(n + 1, std::vector<long long>(budget + 1, 0));
    std::vector<std::vector<uint8_t>> take(n + 1, std::vector<uint8_t>(budget + 1, 0));
    for (int i = 1; i <= n; ++i)
        for (int cap = 0; cap <= budget; ++cap) {
            best[i][cap] = best[i - 1][cap];
            if (w[i - 1] <= cap && best[i - 1][cap - w[i - 1]] + q[i - 1] > best[i][cap]) {
                best[i][cap] = best[i - 1][cap - w[i - 1]] + q[i - 1];
                take[i][cap] = 1;
            }
        }
    int cap = budget;
    for (int i = n; i >= 1; --i) {
        mask[i - 1] = take[i][cap];
        if (take[i][cap]) cap -= w[i - 1];
    }
    return best[n][budget];
}

// Brute force over all 2^n masks (n <= 24): the largest value, ties to the
// smallest bitmask (bit i-1 <-> item i).
long long ko_knapsack_brute(const int* w, const long long* q, int n, int budget, uint8_t* mask) {
    long long bv = -1;
    uint32_t bm = 0;
    for (uint32_t m = 0; m < (1u << n); ++m) {
        long long sw = 0, sv = 0;
        for (int i = 0; i < n; ++i)
            if (m >> i & 1u) {
                sw += w[i];
                sv += q[i];
            }
        if (sw <= budget && sv > bv) {
            bv = sv;
            bm = m;
        }
    }
    for (int i = 0; i < n; ++i) mask[i] = (bm >> i) & 1u;
    return bv;
}

// ------------------------------------------------------------------ session
// One sequence: KV cache, committed length p, pending token (newest known
// token, its K/V not yet in the cache), history of per-sublayer states of the
// committed rows of the last hist_steps verify passes (the prompt's last
// hist_init_rows rows form the first entry).
struct ko_session {
    ko_config c;
    ko_weights w;
    int n_max;
    std::vector<std::vector<float>> k, v;
    int p = 0, pending = -1;
    int hist_steps, hist_init_rows;
    std::deque<std::vector<float>> hist;   // entries [2L+1][rows][d]
    std::deque<int> hist_rows;
};

ko_session* ko_session_create(const ko_config* c, const ko_weights* w, int n_max, int hist_steps,
                              int hist_init_rows) {
    ko_session* s = new ko_session();
    s->c = *c;
    s->w = *w;
    s->n_max = n_max;
    const size_t per = (size_t)c->n_kv_heads * n_max * c->head_dim;
    s->k.assign(c->n_layers, std::vector<float>(per, 0.f));
    s->v.assign(c->n_layers, std::vector<float>(per, 0.f));
    s->hist_steps = hist_steps;
    s->hist_init_rows = hist_init_rows;
    return s;
}

void ko_session_destroy(ko_session* s) { delete s; }

// f^(S) on R consecutive rows at positions pos0..: logits [R][vocab] (may be
// null), states [2L+1][R][d] (X^(i) after sublayer i; may be null).  mask: 2L
// bytes, 1 = run (null = all).  Returns 0, or -1 past the KV capacity.
int ko_forward(ko_session* s, const int* tokens, int R, int pos0, const uint8_t* mask, float* logits,
               float* states) {
    const ko_config& c = s->c;
    const int d = c.d_model, L = c.n_layers;
    if (pos0 + R > s->n_max) return -1;
    std::vector<float> x((size_t)R * d);
    std::vector<int> pos(R);
    for (int r = 0; r < R; ++r) {
        pos[r] = pos0 + r;
        std::memcpy(&x[(size_t)r * d], s->w.embed + (size_t)tokens[r] * d, sizeof(float) * d);
    }
    if (states) std::memcpy(states, x.data(), sizeof(float) * R * d);
    for (int i = 1; i <= 2 * L; ++i) {
        if (!mask || mask[i - 1]) {
            const int l = (i - 1) / 2;
            if (i % 2 == 1)
                ko_attn_sublayer(&c, &s->w, l, x.data(), R, pos.data(), s->k[l].data(), s->v[l].data(), s->n_max);
            else
                ko_mlp_sublayer(&c, &s->w, l, x.data(), R);
        }
        if (states) std::memcpy(states + (size_t)i * R * d, x.data(), sizeof(float) * R * d);
    }
    if (logits) ko_final_logits(&c, &s->w, x.data(), R, logits, 0, c.vocab);
    return 0;
}

static void push_history(ko_session* s, const std::vector<float>& states, int R, int first, int rows) {
    const int d = s->c.d_model, n = 2 * s->c.n_layers + 1;
    std::vector<float> e((size_t)n * rows * d);
    for (int i = 0; i < n; ++i)
        std::memcpy(&e[((size_t)i * rows) * d], &states[((size_t)i * R + first) * d], sizeof(float) * rows * d);
    s->hist.push_back(std::move(e));
    s->hist_rows.push_back(rows);
    while ((int)s->hist.size() > s->hist_steps) {
        s->hist.pop_front();
        s->hist_rows.pop_front();
    }
}

// The prompt in chunks of `chunk` rows; the greedy next token becomes pending.
int ko_prefill(ko_session* s, const int* prompt, int n, int chunk) {
    const int d = s->c.d_model, V = s->c.vocab, n_st = 2 * s->c.n_layers + 1;
    std::vector<float> logits, states;
    int last = 0;
    for (int s0 = 0; s0 < n; s0 += chunk) {
        const int R = n - s0 < chunk ? n - s0 : chunk;
        logits.assign((size_t)R * V, 0.f);
        states.assign((size_t)n_st * R * d, 0.f);
        if (ko_forward(s, prompt + s0, R, s0, nullptr, logits.data(), states.data())) return -1;
        last = R;
    }
    s->p = n;
    s->pending = ko_argmax(&logits[(size_t)(last - 1) * V], V);
    s->hist.clear();
    s->hist_rows.clear();
    const int r0 = s->hist_init_rows < last ? s->hist_init_rows : last;
    push_history(s, states, last, last - r0, r0);
    return s->pending;
}

// One greedy autoregressive step: commit pending, return the new token.
int ko_ar_step(ko_session* s) {
    std::vector<float> logits(s->c.vocab);
    if (ko_forward(s, &s->pending, 1, s->p, nullptr, logits.data(), nullptr)) return -1;
    s->p += 1;
    s->pending = ko_argmax(logits.data(), s->c.vocab);
    return s->pending;
}

// gamma greedy tokens from f^(S) starting at the pending token (Sec. 2.2).
int ko_draft(ko_session* s, const uint8_t* mask, int gamma, int* out) {
    std::vector<float> logits(s->c.vocab);
    int tok = s->pending;
    for (int t = 0; t < gamma; ++t) {
        if (ko_forward(s, &tok, 1, s->p + t, mask, logits.data(), nullptr)) return -1;
        tok = ko_argmax(logits.data(), s->c.vocab);
        out[t] = tok;
    }
    return 0;
}

// Score [pending] + drafts with the target in one pass (Sec. 2.1): a accepted
// drafts, then the target's own token (a + 1 tokens in new_tokens).  Commits
// them and records their states as one history entry.
int ko_verify(ko_session* s, const int* drafts, int gamma, int* a_out, int* new_tokens) {
    const int R = gamma + 1, V = s->c.vocab, d = s->c.d_model, n_st = 2 * s->c.n_layers + 1;
    std::vector<int> rows(R);
    rows[0] = s->pending;
    for (int t = 0; t < gamma; ++t) rows[t + 1] = drafts[t];
    std::vector<float> logits((size_t)R * V), states((size_t)n_st * R * d);
    if (ko_forward(s, rows.data(), R, s->p, nullptr, logits.data(), states.data())) return -1;
    int a = 0;
    while (a < gamma && drafts[a] == ko_argmax(&logits[(size_t)a * V], V)) ++a;
    for (int t = 0; t < a; ++t) new_tokens[t] = drafts[t];
    new_tokens[a] = ko_argmax(&logits[(size_t)a * V], V);
    push_history(s, states, R, 0, a + 1);
    s->p += a + 1;
    s->pending = new_tokens[a];
    *a_out = a;
    return 0;
}

int ko_position(const ko_session* s, int* pending) {
    if (pending) *pending = s->pending;
    return s->p;
}

// Rows held in the history (and, if out != null, X^(0..2L) of them as
// [2L+1][r][d], oldest entry first).
int ko_history(const ko_session* s, float* out) {
    int r = 0;
    for (int n : s->hist_rows) r += n;
    if (!out) return r;
    const int d = s->c.d_model, n_st = 2 * s->c.n_layers + 1;
    int off = 0;
    for (size_t e = 0; e < s->hist.size(); ++e) {
        const int rows = s->hist_rows[e];
        for (int i = 0; i < n_st; ++i)
            std::memcpy(out + ((size_t)i * r + off) * d, &s->hist[e][(size_t)i * rows * d], sizeof(float) * rows * d);
        off += rows;
    }
    return r;
}

}  // extern "C"
