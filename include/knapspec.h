/*
 * knapspec.h - C ABI of a single-GPU (GB300, sm_103a) implementation of the
 * data-parallel hot path of KnapSpec self-speculative decoding
 * (Cha, Kim, Han, Yang, Han: "KnapSpec: Self-Speculative Decoding via
 * Adaptive Layer Selection as a Knapsack Problem", arXiv 2602.20217).
 *
 * The hot path, per speculation step:
 *   a1  draft:   gamma greedy tokens from the skip-masked sub-network f^(S)
 *                (Sec. 2: f^(S) composes the sublayers in S in their order;
 *                f^(2i-1) = Attn_i, f^(2i) = MLP_i, norms included);
 *   a2  verify:  the full target f over the gamma+1 rows in one pass (Sec. 2.1);
 *   a3  accept:  greedy acceptance - keep drafts while they equal the target's
 *                argmax, then append the target's own token (Sec. 2.1, Eq. 1);
 *   a4  cosine:  per-sublayer matrix cosines of the history hidden states
 *                (Sec. 2 definition of cos(X, Y); Sec. 3.4, m = 5 steps);
 *   a5  select:  integer latency weights (Sec. 3.4, App. C) and an exact 0/1
 *                knapsack over the 2L sublayers (Sec. 3.3) -> next draft mask.
 *
 * Conventions for every call:
 *  - All device memory is allocated by the caller.  The library borrows
 *    pointers and never frees them.  A model handle owns host metadata, a
 *    small pinned host staging buffer and CUDA events only.
 *  - "dev" pointers are device addresses; "host" pointers are host memory.
 *  - Weights are row-major [out, in] (y = W x), dtype KS_DTYPE_F32 or
 *    KS_DTYPE_BF16; norm gains have the same dtype.  The residual stream and
 *    all reductions are fp32; bf16 models feed bf16 activations to the
 *    matrix products and keep the KV cache in bf16.
 *  - Every call returns a ks_status and never aborts, traps or exits.
 *    Invalid arguments are rejected before any work is enqueued.  CUDA errors
 *    are reported as KS_ERR_CUDA (the message is kept per thread, see
 *    ks_last_error).  No kernel waits on another launch; the pipeline waits
 *    inside a kernel (TMA barriers) give up after 2 s, record the fact in a
 *    device status word and return, and the next synchronising call reports
 *    KS_ERR_TIMEOUT.  The status word stays set until the model is created
 *    again (every later synchronising call reports it), and the chained
 *    projection kernels of a job enqueued after it was set return at once, so
 *    a long job that hit a timeout ends quickly instead of waiting again.
 *  - One handle is used by one host thread at a time and issues all work on
 *    the stream given at creation.
 *  - Greedy argmax ties resolve to the lowest token id.
 */
#ifndef KNAPSPEC_H
#define KNAPSPEC_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    KS_OK = 0,
    KS_ERR_INVALID_ARG = 1,   /* null/misaligned pointer, bad size, bad shape      */
    KS_ERR_CUDA = 2,          /* a CUDA runtime call or kernel launch failed        */
    KS_ERR_WORKSPACE = 3,     /* the workspace is smaller than required             */
    KS_ERR_CAPACITY = 4,      /* KV capacity (max_seq) or row capacity exceeded     */
    KS_ERR_TIMEOUT = 5,       /* a bounded device-side wait gave up (2 s limit)     */
    KS_ERR_UNSUPPORTED = 6,   /* shape/dtype outside what the kernels implement     */
    KS_ERR_STATE = 7          /* call out of order (e.g. draft before prefill)      */
} ks_status;

enum { KS_DTYPE_F32 = 0, KS_DTYPE_BF16 = 1 };

/* Decoder shape (Sec. 2 with the Llama / Qwen3 block; see the design notes).
 * Supported: head_dim in {64, 128}; n_q_heads % n_kv_heads == 0;
 * d_model, d_ff, head_dim multiples of 8; max_rows <= 16. */
typedef struct {
    int32_t n_layers;        /* L; the model has 2L sublayers                          */
    int32_t d_model;
    int32_t n_q_heads;
    int32_t n_kv_heads;
    int32_t head_dim;
    int32_t d_ff;
    int32_t vocab;
    int32_t qk_norm;         /* 1: per-head RMSNorm on q and k before RoPE (Qwen3)     */
    int32_t dtype;           /* KS_DTYPE_F32 or KS_DTYPE_BF16                          */
    int32_t max_seq;         /* KV capacity in positions                               */
    int32_t max_rows;        /* rows per pass: >= gamma + 1 and the prefill chunk      */
    int32_t hist_steps;      /* m: speculation steps kept in the history (Sec. 3.4)    */
    int32_t hist_init_rows;  /* prompt rows that seed the history at prefill           */
    float rms_eps;
    double rope_theta;       /* rotate-half RoPE, inv_freq_j = theta^(-2j/head_dim)    */
} ks_config;

/* Borrowed device pointers.  Per-layer fields point to host arrays of
 * n_layers device pointers.  q_norm / k_norm may be NULL when qk_norm == 0.
 *   embed      [vocab, d]           lm_head  [vocab, d]     final_norm [d]
 *   attn_norm  [d]                  w_qkv    [(hq + 2 hk) hd, d]  (q; k; v rows)
 *   w_o        [d, hq hd]           q_norm, k_norm [hd]
 *   mlp_norm   [d]                  w_gate_up [2 d_ff, d]  (gate rows, then up rows)
 *   w_down     [d, d_ff]
 * Every device pointer must be 16-byte aligned. */
typedef struct {
    const void* embed;
    const void* lm_head;
    const void* final_norm;
    const void* const* attn_norm;
    const void* const* w_qkv;
    const void* const* w_o;
    const void* const* q_norm;
    const void* const* k_norm;
    const void* const* mlp_norm;
    const void* const* w_gate_up;
    const void* const* w_down;
} ks_weights;

/* Latency model used for the knapsack weights.
 * kind 0: App. C model t_MLP = c1, t_Attn(n) = c2 n + c3, turned into integer
 *         weights by Sec. 3.4: Delta = min(t_Attn(n), t_MLP),
 *         w = round(t / Delta) (half away from zero, at least 1).
 *         Requires c1 > 0, c2 >= 0, c3 >= 0 (finite), t_Attn(n) > 0 at the
 *         context length used, and max(t_Attn, t_MLP) / min(t_Attn, t_MLP)
 *         <= 65535; otherwise the call taking it returns KS_ERR_INVALID_ARG.
 * kind 1: explicit integer units per sublayer, units[2L] (host), 1..65535. */
typedef struct {
    int32_t kind;
    double c1, c2, c3;
    const int32_t* units;
} ks_latency;

/* Least-squares fit of the App. C latency model from a profiling sweep:
 * (c2, c3) minimise sum_k (c2 n[k] + c3 - t_attn[k])^2 over count >= 2
 * samples (n: context lengths, not all equal; t_attn: the Attn sublayer's
 * time at n[k]); c1 = mean of t_mlp[0 .. count_mlp - 1] (the MLP sublayer's
 * time, which does not depend on n).  The coefficients of the model are
 * non-negative: a negative intercept is refitted through the origin (c3 = 0),
 * a negative slope gives c2 = 0 and c3 = mean(t_attn).  Writes a kind-0 model
 * into *out.  Host arrays; no GPU work.  KS_ERR_INVALID_ARG on too few or
 * non-finite samples, equal context lengths, or a non-positive c1. */
ks_status ks_fit_latency(const double* n, const double* t_attn, int32_t count, const double* t_mlp,
                         int32_t count_mlp, ks_latency* out);

typedef struct ks_model ks_model;

/* ------------------------------------------------------------ model (a1-a3) */

/* Bytes of device workspace a model with this config needs (KV cache, RoPE
 * table, activations, split partials, history ring).  0 on an invalid config. */
size_t ks_workspace_bytes(const ks_config* cfg);

/* Validate cfg, borrow the weights and the workspace (dev, 256-byte aligned,
 * at least ks_workspace_bytes(cfg) bytes), build the RoPE table, zero the KV
 * cache region of the workspace (the attention streams whole 16-key tiles,
 * and keys past a row's position get an exact zero weight only if their
 * values are finite), and return a handle bound to `stream` (a cudaStream_t;
 * NULL = legacy default stream); the call waits for the stream.  bf16
 * configs need 2 n_layers n_kv_heads max_seq < 2^31 (32-bit cache-row
 * coordinates); ks_workspace_bytes returns 0 otherwise.  No decoding state
 * exists until ks_prefill. */
ks_status ks_model_create(const ks_config* cfg, const ks_weights* w, void* workspace,
                          size_t workspace_bytes, void* stream, ks_model** out);
ks_status ks_model_destroy(ks_model* m);

/* Run the prompt (host int32[n], 1 <= n, n + 1 <= max_seq) through the target
 * in chunks of max_rows rows, fill the KV cache, seed the history with the
 * last hist_init_rows prompt rows, and set the pending token to the greedy
 * next token, written to *next_token (host).  Resets any previous sequence. */
ks_status ks_prefill(ks_model* m, const int32_t* tokens, int32_t n, int32_t* next_token);

/* Return to the state right after the last ks_prefill without recomputing the
 * prompt: decoding writes K/V only at positions at or past the prompt length,
 * so the prompt's cache is still valid; the committed length, the pending
 * token (also written to *next_token, host) and the history are restored.
 * Serves several generations from one long prompt.  (An addition of this
 * library; the paper has no counterpart.)  KS_ERR_STATE before any prefill. */
ks_status ks_rewind(ks_model* m, int32_t* next_token);

/* a1 (Sec. 2, Sec. 2.2): gamma (1 <= gamma < max_rows) greedy draft tokens
 * from f^(S), S = { i : mask[i-1] != 0 } (host uint8[2L]; odd 1-based
 * sublayers are Attn, even are MLP), starting from the pending token at the
 * committed length p.  A skipped sublayer is the identity on the residual
 * stream.  Run Attn sublayers write K/V at positions p.. (overwritten by the
 * verify).  The drafts stay on the device; if draft_tokens (host int32[gamma])
 * is not NULL the call also waits for them and copies them out. */
ks_status ks_draft(ks_model* m, const uint8_t* mask, int32_t gamma, int32_t* draft_tokens);

/* a1 with the dynamic drafting exit of Sec. 3.5 ("Dynamic Drafting Exit"):
 * like ks_draft with gamma as the maximum draft length, but after each draft
 * token the device computes its confidence, the softmax probability of the
 * token over the draft's logits, 1 / sum_i exp(l_i - l_max), and once a token's
 * confidence is below tau_conf the step's remaining draft passes do nothing
 * (that token stays the step's last draft).  tau_conf: finite, >= 0 (0 never
 * stops; above 1 always stops after one token).  Everything stays on the
 * device with no host synchronisation unless an output is requested; the
 * following ks_verify (draft_tokens NULL, same gamma) still scores gamma + 1
 * rows but compares only the drafts produced.
 * Outputs (host, each optional; any of them makes the call wait): *n_drafted
 * (1 .. gamma), confidence[0 .. n_drafted) (float; room for gamma), and
 * draft_tokens[0 .. n_drafted) (room for gamma). */
ks_status ks_draft_dynamic(ks_model* m, const uint8_t* mask, int32_t gamma, float tau_conf, int32_t* n_drafted,
                           float* confidence, int32_t* draft_tokens);

/* Sampling mode (Sec. 2.1, sampling branch; the Sec. 4 experiments use
 * temperature 0.7, top_k 50, top_p 0.95).  A distribution is the row's logits
 * divided by the temperature, cut to the top_k largest (ties: lower id first;
 * top_k above 64 is taken as 64), softmaxed, cut to the shortest prefix in
 * descending probability whose cumulative probability reaches top_p, and
 * renormalised.  Uniform numbers are Philox4x64-10 (Salmon et al., SC 2011)
 * with key (seed, 0) and counter (step, row, purpose, 0): purpose 0 the draft
 * sample of position row, 1 the acceptance test of draft row, 2 the step's
 * residual or bonus sample; u = (first output word >> 40) / 2^24. */
typedef struct {
    float temperature;       /* > 0 (0 in ks_spec_params: greedy decoding)   */
    int32_t top_k;           /* >= 1                                          */
    float top_p;             /* (0, 1]                                        */
    uint64_t seed;
} ks_sampling;

/* a1, sampling: gamma draft tokens of f^(S), each drawn from its draft
 * distribution q_t with the uniform of (step, t, 0); the q_t stay on the
 * device for ks_verify_sample.  draft_tokens: host int32[gamma] or NULL (then
 * no synchronisation). */
ks_status ks_draft_sample(ks_model* m, const uint8_t* mask, int32_t gamma, const ks_sampling* s, uint64_t step,
                          int32_t* draft_tokens);

/* a2 + a3, sampling (Sec. 2.1): score [pending, drafts...] of the preceding
 * ks_draft_sample (same gamma, same step and sampling parameters) with the
 * full target, form the target distributions p_0..p_gamma, and accept draft t
 * while u(step, t, 1) <= min(1, p_t(x_t) / q_t(x_t)).  At the first rejection
 * the next token is drawn from norm(max(0, p_t - q_t)) (from p_t if that has
 * no mass), after gamma acceptances from p_gamma, with u(step, 0, 2).  The
 * tokens are distributed as samples of the target.  Outputs and commit as
 * ks_verify.  Waits for the stream. */
ks_status ks_verify_sample(ks_model* m, int32_t gamma, const ks_sampling* s, uint64_t step, int32_t* n_accepted,
                           int32_t* out_tokens, int32_t* n_out);

/* a2 + a3 (Sec. 2.1): score [pending, drafts...] (gamma + 1 rows at positions
 * p..p+gamma) with the full target in one pass, take the greedy argmax of
 * each row, accept the longest prefix of drafts equal to the target's
 * argmaxes (a of them) and append the target's own next token.  Commits the
 * a + 1 rows (p += a + 1), records their per-sublayer hidden states in the
 * history ring, and makes the appended token pending.
 * draft_tokens: host int32[gamma] to score, or NULL to score the drafts of the
 * preceding ks_draft call with the same gamma.
 * Outputs (host): *n_accepted = a; out_tokens[0..a] = the a + 1 new tokens
 * (room for gamma + 1); *n_out = a + 1.  Waits for the stream. */
ks_status ks_verify(ks_model* m, const int32_t* draft_tokens, int32_t gamma,
                    int32_t* n_accepted, int32_t* out_tokens, int32_t* n_out);

/* Plain greedy autoregressive decoding of n_tokens tokens with the full
 * target (the non-speculative baseline).  out (host int32[n_tokens]) receives
 * the pending token followed by the next n_tokens - 1 greedy tokens; the
 * last one is left pending.  One host synchronisation at the end. */
ks_status ks_decode_greedy(ks_model* m, int32_t n_tokens, int32_t* out);

/* Committed length p and the pending token. */
ks_status ks_model_position(const ks_model* m, int32_t* committed, int32_t* pending);

/* ------------------------------------------------------------ cosine (a4) */

/* Sec. 2 matrix cosine for n_pairs pairs of [rows, d] matrices:
 *   out[p] = (1/rows) sum_i <X_p[i], Y_p[i]> / (|X_p[i]| |Y_p[i]|)
 * X_p = X + p * pair_stride elements, Y_p likewise (row i at + i * d, or at
 * + row_index[i] * d when row_index (dev int32[rows]) is not NULL).
 * X, Y: dev, dtype KS_DTYPE_F32 or KS_DTYPE_BF16.  out: dev float[n_pairs].
 * Each pair's row terms are summed in row order (deterministic).  A zero row
 * gives a NaN term, as the definition does. */
ks_status ks_cosine(const void* X, const void* Y, int32_t dtype, int64_t n_pairs,
                    int32_t rows, int32_t d, int64_t pair_stride, const int32_t* row_index,
                    float* out, void* stream);

/* a4 for a model: sims (dev float[2L]) receive sigma_i = cos(X^(i-1), X^(i))
 * over the rows held in the history ring (Sec. 3.4: the tokens of the last m
 * speculation steps), i = 1..2L; *rows_used (host, optional) = r. */
ks_status ks_history_similarities(ks_model* m, float* sims, int32_t* rows_used);

/* ------------------------------------------------------------ select (a5) */

/* Integer weights of the 2L sublayers at context length context_len
 * (Sec. 3.4 / App. C, see ks_latency), then the exact 0/1 knapsack
 *   maximise sum_{i in S} q_i  subject to  sum_{i in S} w_i <= budget_units,
 * q_i = round((1 - sims[i-1]) * 2^30) as int64 (half away from zero, from the
 * fp32 similarity in double): the similarity lost by skipping sublayer i.
 * Among optimal masks the one with the smallest bitmask value (bit i-1 <->
 * sublayer i) is returned, so the result is exact and reproducible.
 * sims: dev float[n_sublayers].  Outputs (dev): mask_out uint8[n_sublayers]
 * (1 = run), objective_out double (sum q_i / 2^30, may be NULL), weights_out
 * int32[n_sublayers] (may be NULL).  n_sublayers even, 2..256;
 * 0 <= budget_units <= 65535.  scratch (dev, 16-byte aligned) must hold
 * ks_select_scratch_bytes(n_sublayers, budget_units) bytes; the call does not
 * allocate. */
size_t ks_select_scratch_bytes(int32_t n_sublayers, int32_t budget_units);
ks_status ks_select_mask(const ks_latency* lat, const float* sims, int64_t context_len,
                         int32_t n_sublayers, int32_t budget_units, uint8_t* mask_out,
                         double* objective_out, int32_t* weights_out, void* scratch,
                         size_t scratch_bytes, void* stream);

/* Allocation-free variant of ks_select_mask (the paper has no counterpart:
 * this is a deployment convenience).  Some callers cannot give this library
 * any device memory beyond their own inputs and outputs - for example a
 * plugin inside a host framework that owns every allocation, or a serving
 * loop that must not call cudaMalloc after start-up because cudaMalloc can
 * synchronise the device.  For them the knapsack's work tables live in one
 * array built into the library: a file-scope __device__ buffer of about
 * 1.1 MB on every GPU that loads the library, held until the process exits.
 * Same inputs, outputs and results as ks_select_mask, without the scratch
 * arguments; budget_units must be 0..KS_SELECT_STATIC_MAX_BUDGET (larger
 * budgets return KS_ERR_INVALID_ARG).  The call allocates nothing: no
 * cudaMalloc, cudaFree or allocating library routine.
 * Every call looks up the array's device address (cudaGetSymbolAddress)
 * on the current device, so a context created after cudaDeviceReset gets its
 * own copy.  With CUDA's lazy module loading, the first call on a device may
 * load this library's device code, and the driver then reserves memory for
 * the module and this array; make that first call during start-up, before
 * any stream capture.  All calls share the one array and the kernel
 * rewrites every table entry it reads, so no state leaks from one call to
 * the next; two calls whose kernels overlap on the GPU (different streams)
 * race on the array and must be ordered by the caller. */
#define KS_SELECT_STATIC_MAX_BUDGET 4095
ks_status ks_select_mask_static(const ks_latency* lat, const float* sims, int64_t context_len,
                                int32_t n_sublayers, int32_t budget_units, uint8_t* mask_out,
                                double* objective_out, int32_t* weights_out, void* stream);

/* The TPT stage of the layer selection (Sec. 3.5, Alg. 2, Eqs. 1, 3, 4), on
 * the model's history (the same rows as ks_history_similarities):
 *  1. candidate set A: with the values of a4 and the weights of `lat` (as in
 *     ks_select_mask), the knapsack optimum for each of n_candidates budgets
 *     floor(sum_i w_i (j + 1) / n_candidates), j = 0 .. n_candidates - 1;
 *  2. acceptance of each candidate on the r history rows (Eq. 4): the
 *     draft's final state on a row is taken to first order as the target's
 *     X^(2L) minus the recorded contribution X^(i) - X^(i-1) of every skipped
 *     sublayer i; its prediction (final RMSNorm, LM head, argmax, ties to the
 *     lowest id) is compared with the full layer set's on the same row;
 *  3. grid search of Eq. 3 over A x {1 .. max_gamma}: expected tokens (Eq. 1)
 *     over gamma t_Draft(S) + t_Target, with t_Attn(n) and t_MLP of the
 *     latency model (kind 0, n = the committed length) or the units as times
 *     (kind 1); candidates in order, gamma ascending, strictly larger wins.
 * n_candidates: 1 .. KS_TPT_MAX_CANDIDATES; max_gamma: 1 .. max_rows - 1.
 * Outputs (host): mask_out[2L] (the chosen candidate), *gamma_out, *tpt_out
 * (in tokens per unit of the latency's time), and, unless NULL,
 * alphas_out[n_candidates] and candidates_out[n_candidates][2L].  Uses the
 * model's pass buffers but no decoding state changes.  Waits for the stream.
 * KS_ERR_STATE before a prefill. */
#define KS_TPT_MAX_CANDIDATES 16
ks_status ks_select_tpt(ks_model* m, const ks_latency* lat, int32_t n_candidates, int32_t max_gamma,
                        uint8_t* mask_out, int32_t* gamma_out, double* tpt_out, double* alphas_out,
                        uint8_t* candidates_out);

/* NEXT row: the hidden-state dynamic program of Alg. 1 (Sec. 3.4) and the TPT
 * selection over its candidates (Sec. 3.5, Alg. 2).  On the r most recent
 * history rows (the last r committed positions, r <= max_rows), g[i, j] is the
 * best hidden state after sublayer i with skipped weight j (integer weights of
 * Sec. 3.4 from lat at the committed length): the execute candidate
 * f^(i)(g[i-1, j]) wins over the skip candidate g[i-1, j - w_i] when its
 * matrix cosine to the target's X^(i) is at least as high; states with cosine
 * below tau or j > K / 2 are dropped (Sec. 3.4, pruning; the paper uses tau
 * 0.5); g[i, 0] = X^(i).  Inside f^(i) a history row attends to the target's
 * K/V for earlier positions and to the state's own K/V (the target's cache is
 * restored afterwards).  Each surviving terminal state gives a layer set (by
 * its recorded choices) and an acceptance estimate (Eq. 4: the fraction of
 * rows whose LM-head argmax equals the target's); the Eq. 3 grid over the
 * candidates (executed weight ascending) and gamma = 1..max_gamma picks
 * (S*, gamma*).
 * scratch: device, 256-byte aligned, >= ks_dp_scratch_bytes(m, max_states,
 * max_rows) bytes; max_states (1..128) must cover K / 2 + 1.
 * Outputs (host): mask_out[2L], *gamma_out, *tpt_out; optional: *n_candidates,
 * js_out[] (the candidates' skipped weights), alphas_out[], candidates_out
 * [n][2L] (room for max_states each).  Uses the model's pass buffers; the
 * decoding state is unchanged.  Waits for the stream (twice). */
size_t ks_dp_scratch_bytes(const ks_model* m, int32_t max_states, int32_t max_rows);
ks_status ks_select_dp(ks_model* m, const ks_latency* lat, float tau, int32_t max_gamma, int32_t max_states,
                       int32_t max_rows, void* scratch, size_t scratch_bytes, uint8_t* mask_out, int32_t* gamma_out,
                       double* tpt_out, int32_t* n_candidates, int32_t* js_out, double* alphas_out,
                       uint8_t* candidates_out);

/* ------------------------------------------------- full speculative loop */

typedef struct {
    int32_t gamma;           /* draft length per step (1 <= gamma < max_rows); policy 2: until
                                the first selection                                         */
    int32_t policy;          /* 0 fixed mask; 1 knapsack re-solved every resolve_every steps;
                                2 TPT stage (ks_select_tpt) every resolve_every steps, which
                                also sets gamma; 3 the hidden-state DP (ks_select_dp) every
                                resolve_every steps, which also sets gamma                   */
    const uint8_t* mask;     /* host uint8[2L]: the mask for policy 0                      */
    ks_latency latency;      /* policies 1 and 2                                            */
    double budget_frac;      /* policy 1: budget = floor(budget_frac * sum_i w_i)          */
    int32_t resolve_every;   /* policies 1, 2: optimisation interval T in verify steps (>= 1) */
    int32_t max_steps;       /* stop after this many verify steps (0: no limit)             */
    int32_t tpt_candidates;  /* policy 2: n_candidates of ks_select_tpt                     */
    int32_t tpt_max_gamma;   /* policy 2: max_gamma of ks_select_tpt                        */
    double tau_conf;         /* > 0: dynamic drafting exit (ks_draft_dynamic) with this
                                tau_conf; 0: every step drafts gamma tokens               */
    ks_sampling sampling;    /* temperature > 0: sampling mode (ks_draft_sample /
                                ks_verify_sample, step = the verify step index from 0);
                                not combined with tau_conf                                 */
    void* dp_scratch;        /* policy 3: scratch of ks_select_dp (caller-owned, device)    */
    uint64_t dp_scratch_bytes;
    float dp_tau;            /* policy 3: tau of ks_select_dp                               */
    int32_t dp_max_states;   /* policy 3: max_states / max_rows of ks_select_dp; its
                                max_gamma is tpt_max_gamma                                 */
    int32_t dp_max_rows;
} ks_spec_params;

typedef struct {
    int64_t steps;           /* verify steps                                    */
    int64_t drafted;         /* draft tokens proposed                           */
    int64_t accepted;        /* draft tokens accepted                           */
    int64_t resolves;        /* knapsack solves                                 */
    int64_t attn_skipped;    /* sublayers skipped by the last mask: Attn / MLP  */
    int64_t mlp_skipped;
} ks_spec_stats;

/* Greedy self-speculative decoding of n_tokens tokens: repeat a1..a5 until
 * n_tokens tokens are known (the pending token counts as the first) or
 * max_steps verify steps have run.  Tokens produced = 1 + steps + accepted.
 * out: host int32[n_tokens].  The token stream equals ks_decode_greedy's.
 * accepted_per_step (host int32[], optional, room for n_tokens entries). */
ks_status ks_generate_speculative(ks_model* m, const ks_spec_params* params, int32_t n_tokens,
                                  int32_t* out, ks_spec_stats* stats, int32_t* accepted_per_step);

/* ------------------------------------------------------------ diagnostics */

/* Copy a window of device state to the caller (for tests):
 * what = 0: logits of the last pass, float[rows][vocab];
 *        1: the residual stream rows, float[rows][d];
 *        2: K cache of layer `layer`, [n_kv_heads][positions][head_dim] in the model dtype
 *           for positions [start, start + count), dst laid out [hk][count][hd];
 *        3: V cache, as 2;
 *        4: history ring states of the committed rows, float[2L+1][r][d], with
 *           count == r; count == 0 writes r itself (int32) to dst;
 *        5: sampling draft distributions of positions [start, start + count):
 *           per position int32 n, int32 ids[64], float probs[64] (first n used);
 *        6: sampling target distributions of the last ks_verify_sample rows, as 5;
 * dst is host memory of `bytes` bytes; the call waits for the stream. */
ks_status ks_debug_read(ks_model* m, int32_t what, int32_t layer, int32_t start, int32_t count,
                        void* dst, size_t bytes);

/* Host-side fault injection for tests of the error path: after the model's
 * stream is idle, write `code` into the device status word, as a kernel
 * whose bounded wait gave up writes 1 (a self-check failure writes 2..5);
 * 0 clears the word.  While the word is set, every synchronising call
 * reports it (1: KS_ERR_TIMEOUT, else KS_ERR_STATE) and the chained
 * projection kernels of later launches return at once.  Errors: null m,
 * code outside 0..5 -> KS_ERR_INVALID_ARG; a CUDA failure -> KS_ERR_CUDA. */
ks_status ks_debug_set_status(ks_model* m, int32_t code);

/* Per-kernel timing with CUDA events on the model's stream.  While enabled,
 * every launch of the kernel class `klass` (0 QKV, 1 attention, 2 merge,
 * 3 O-proj, 4 gate/up, 5 down, 6 LM head, 7 embed, 8 accept, 9 chained
 * projections, 10 bf16 attention query prep) is bracketed by events; ks_kernel_time returns the launches
 * and total milliseconds since enabling.  Enabling resets the counters.
 * bf16 models run the projections between two attention cores as one chained
 * launch (class 9); while any of classes 0, 3, 4, 5, 6 is enabled they run
 * one projection per launch instead, so that each can be timed alone.
 * ks_kernel_bytes: weight bytes the timed launches of the class had to read
 * (the algorithmic bytes of the projection classes; 0 for the others). */
ks_status ks_kernel_timing(ks_model* m, int32_t klass, int32_t enable);
ks_status ks_kernel_time(ks_model* m, int32_t klass, int64_t* launches, double* total_ms);
ks_status ks_kernel_bytes(const ks_model* m, int32_t klass, double* bytes);

/* Launch counter: kernels this handle has launched since creation. */
int64_t ks_launch_count(const ks_model* m);

/* Bytes this handle has copied host->device and device->host since creation
 * (prompt and draft uploads, history row lists, results, masks, tokens). */
ks_status ks_transfer_bytes(const ks_model* m, int64_t* h2d, int64_t* d2h);

const char* ks_status_str(ks_status s);
/* Last error message of the calling thread ("" if none). */
const char* ks_last_error(void);

#ifdef __cplusplus
}
#endif
#endif /* KNAPSPEC_H */
