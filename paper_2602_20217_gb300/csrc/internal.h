// Internal interfaces between the translation units of libknapspec.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/knapspec.h"

namespace ks {

// ------------------------------------------------------------------ GEMV
// Y[r][n] = sum_k W[n][k] * A[r][k] for r < R rows ("skinny GEMM"), with a
// fused prologue (optional RMSNorm of an fp32 residual input) and epilogue.
enum GemvEpi { EPI_STORE = 0, EPI_RESID = 1, EPI_SWIGLU = 2, EPI_LMHEAD = 3 };

struct GemvArgs {
    int dtype;              // KS_DTYPE_F32 / KS_DTYPE_BF16 (selects kernel and split plan)
    const void* W;          // [N (or 2N for SwiGLU)][K], row stride K, model dtype
    int N;                  // output features (SwiGLU: d_ff; rows n and N + n pair up)
    int K;
    int R;                  // activation rows, 1..16
    int ksplit;             // K slices (grid.y); set by gemv_plan
    int kc;                 // K per slice (multiple of 64)
    const void* in;         // fp32: the residual [R][in_ld] when norm_gain != null, else the input;
                            // bf16: the input in bf16 [R][in_ld] (x * gain when ss_in != null)
    int in_ld;
    const void* norm_gain;  // RMSNorm gain [K] (model dtype) or null
    float eps;
    const float* ss_in;     // with norm_gain: per-64-feature sums of squares [ss_groups][16]
    int ss_groups;
    float* ss_out;          // EPI_RESID: sums of squares of the new residual [groups][16]
    __nv_bfloat16* xg_out;  // EPI_RESID (bf16): new residual times next_gain, the next GEMV's input
    const void* next_gain;  // gain of the next RMSNorm (model dtype)
    int* err;               // device status word: set to 1 when a bounded wait gives up
    const int* stop;        // draft passes: the pass is skipped when *stop != 0 (null: always run)
    float* out; int out_ld;                    // EPI_STORE (fp32)
    float* resid; int resid_ld;                // EPI_RESID: resid[r][n] += y
    float* capture; long long capture_ld;      // EPI_RESID: optional copy of the new residual
    void* act; int act_ld;                     // EPI_SWIGLU: silu(gate) * up, model dtype
    float* logits; int logits_ld;              // EPI_LMHEAD
    float* amax_val; int* amax_idx;            // EPI_LMHEAD per-group candidates [groups][16]
    int* tokens;                               // EPI_LMHEAD argmax per row
    float* partial;                            // split-K partials [ksplit][R][N or 2N]
    int* counters;                             // [0] work queue, [1] finished CTAs, [2 + g] group tickets
};

void gemv_plan(GemvArgs& a, int epi);           // choose ksplit / kc from (N, K, dtype) only
size_t gemv_partial_floats(int N, int K, int R, int epi, int dtype);
int gemv_grid_x(int N);
cudaError_t launch_gemv(int dtype, int epi, const GemvArgs& a, cudaStream_t s);
// TMA map of a row-major bf16 matrix [rows][K] (K % 8 == 0, 16-byte aligned
// base), box 256 columns x box_rows rows, no swizzle, zero fill outside.
bool make_tma_map(CUtensorMap* map, const void* base, uint64_t rows, uint64_t K, uint32_t box_rows);
// Map for the chain kernel's stages: when K % 256 == 0 a 3-D view
// {256, rows, K / 256} whose box {256, box_rows, chunks} is a whole stage (one
// copy); otherwise the 2-D map above (one copy per 256-column chunk).
bool make_stage_map(CUtensorMap* map, const void* base, uint64_t rows, uint64_t K, uint32_t box_rows,
                    uint32_t chunks);
// Weight map for the chain kernel: 64-column chunks of 16 rows with the
// 128-byte swizzle (16-byte unit u of row r lands at unit u ^ (r & 7)).
// K % 64 == 0: 3-D view {64, rows, K / 64}, box of `chunks` chunks (one copy
// per stage); otherwise 2-D, box {64, 16} (one copy per chunk).
bool make_weight_map(CUtensorMap* map, const void* base, uint64_t rows, uint64_t K, uint32_t chunks);
int gemv_groups(int N, int dtype);              // output groups (argmax candidates) of a launch

// ----------------------------------------------------------------- chain
// bf16 models: a run of consecutive projections (phases) in one persistent
// launch.  Phase codes: 4 l + kind for layer l (kind: ChainKind 0..3), 4 L for
// the LM head.  Each phase reads the previous phase's complete output.  The
// tensor maps travel in the kernel parameters (TMA reads them from there
// without a descriptor fetch from global memory), which bounds a launch to
// kChainMaxPhases phases (about 24 KB of parameters).
constexpr int kChainMaxPhases = 160;
enum ChainKind { CH_QKV = 0, CH_O = 1, CH_GU = 2, CH_DOWN = 3, CH_LM = 4 };

constexpr int kChainSliceMaxItems = 640;   // residual phases with at most this many row groups are K-sliced
struct ChainArgs {
    CUtensorMap wmap[kChainMaxPhases];  // weights of each phase (make_weight_map)
    CUtensorMap amap[4];        // inputs for this R: xg (4-chunk stages), xg (2-chunk), attn_out, act
    int n_phases;
    int R;                      // rows, 1..16
    int stages;                 // ring stages (set by launch_chain)
    int n_layers, d, F, nqkv, hqd, vocab;
    float eps;
    float* x;                   // [R][d] fp32 residual (O / down add into it)
    float* ss;                  // [d / 16][16] per-16-feature sums of squares of x
    __nv_bfloat16* xg;          // [R][d] x * gain of the next RMSNorm (input of QKV / gate-up / LM head)
    float* qkv;                 // [R][nqkv] fp32
    __nv_bfloat16* act;         // [R][F] silu(gate) * up
    float* logits;              // [R][vocab]
    unsigned long long* best;   // [16] LM head argmax keys (zero between launches)
    int* tokens;                // [R] LM head argmax
    float* capture;             // history capture or null: sublayer i's rows at capture + i * capture_plane
    long long capture_plane;
    int* counters;              // chain_counter_ints() zeros; the launch leaves them zero
    int* err;                   // device status word
    const int* stop;            // draft passes: the launch does nothing when *stop != 0 (null: always)
    float* slice_part;          // K-sliced residual phases: [2][kChainSliceMaxItems][2][16][16] partial sums
    int* slice_ticket;          // [2][kChainSliceMaxItems] arrivals per item (zero between uses)
    uint16_t code[kChainMaxPhases];
    const __nv_bfloat16* gain[kChainMaxPhases];  // O / down phases: gain of the next RMSNorm
};
size_t chain_counter_ints();
cudaError_t launch_chain(const ChainArgs& a, cudaStream_t s);
int sm_count();

// ------------------------------------------------------------- attention
struct AttnArgs {
    // bf16: TMA map of the whole KV cache viewed as rows of hd elements
    // ([L][K, V][hk][max_seq] rows; 16-row boxes of hd / 64 swizzled 64-column
    // chunks, make_weight_map), and the first row of this layer's K and V
    CUtensorMap kvmap;
    int kv_row_k, kv_row_v;
    __nv_bfloat16* q;       // bf16: prepared queries [hk][G R][hd] (QK-norm, RoPE, log2(e)/sqrt(hd))
    int* err;               // device status word (bf16 kernels: a bounded wait gave up)
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
    float* part;            // [R][hq][n_chunks_max][hd + 4] (m, l, pad, pad, o[hd])
    int n_chunks_max;
    void* out;              // [R][hq hd] model dtype: merged attention output
    int out_ld;
    const int* stop;        // draft passes: skipped when *stop != 0 (null: always run)
};

// bf16: queries of the pass prepared once (q) and the new rows' K/V written
// to the cache; the attention kernel then only streams the cache.
cudaError_t launch_attn_prep(const AttnArgs& a, cudaStream_t s);
cudaError_t launch_attention(int dtype, const AttnArgs& a, cudaStream_t s);
cudaError_t launch_attn_merge(int dtype, const AttnArgs& a, cudaStream_t s);
// Fixed partition of the key axis for split-KV attention (absolute positions):
// chunks of 128 keys below 8192, 512 below 32768, 2048 beyond.
int attn_num_chunks(int n_keys);
constexpr int kSsGroup = 16;    // features per sum-of-squares partial (= rows of a bf16 GEMV work item)

// ---------------------------------------------------------------- select
size_t select_scratch_bytes(int n_items, int cap);
// Knapsack of a5 (optionally also the frontier of the TPT stage).
cudaError_t launch_select(const ks_latency* lat, const float* sims, int64_t n, int n_items, int budget,
                          double budget_frac, uint8_t* mask, double* objective, int32_t* weights,
                          int32_t* budget_out, void* scratch, int cap, cudaStream_t s, int n_frontier = 0,
                          uint8_t* frontier = nullptr);
// TPT stage after the frontier: Eq. 4 acceptance per candidate and Eq. 3 grid.
cudaError_t launch_tpt(const ks_latency* lat, int64_t n, int n_items, int n_layers, int K, int r, int D,
                       const uint8_t* frontier, const int32_t* tokens, uint8_t* mask_out, int32_t* info,
                       double* out, cudaStream_t s);
cudaError_t launch_cosine(const void* X, const void* Y, int dtype, int64_t n_pairs, int rows,
                          int d, int64_t pair_stride, const int32_t* row_index, float* out,
                          cudaStream_t s);

// Latency model checks shared by every entry point that takes one: kind 0
// needs c1 > 0, c2, c3 >= 0, t_Attn(context_len) = c2 n + c3 > 0 and the
// larger of t_Attn, t_MLP at most 65535 times the smaller; kind 1 needs
// units in 1..65535.
bool latency_valid(const ks_latency* lat, int32_t n_sublayers, int64_t context_len);

// Last error text for ks_last_error (thread-local).
void set_error(const char* fmt, ...);

// ---------------------------------------------------------- sampling mode
// Nucleus-filtered distributions (at most kSampleMaxK tokens per row) and the
// Sec. 2.1 acceptance of sampling-mode speculative decoding (sample.cu).
constexpr int kSampleMaxK = 64;
struct FilterArgs {
    const float* logits;    // [rows][ld] fp32
    int ld, vocab;
    float inv_t;            // 1 / temperature
    int top_k;              // 1 .. kSampleMaxK (larger values are clamped)
    float top_p;            // (0, 1]
    int* ids;               // [slots][kSampleMaxK] support in descending probability
    float* probs;           // [slots][kSampleMaxK] renormalised probabilities
    int* n;                 // [slots] support sizes
    int slot0;              // row r is stored at slot slot0 + r (a draft pass: its position t)
    int32_t* token_out;     // draft pass: the drawn token goes here (null: no draw)
    unsigned long long seed, step;
};
struct AcceptSampleArgs {
    int32_t* rows;          // [gamma + 1]: pending, drafts; rows[0] <- the new pending token
    int gamma;
    const int* p_ids; const float* p_probs; const int* p_n;   // target rows 0..gamma
    const int* q_ids; const float* q_probs; const int* q_n;   // draft positions 0..gamma-1
    int32_t* result;        // {a, gamma, tokens[0..a]}
    unsigned long long seed, step;
};
cudaError_t launch_filter(const FilterArgs& a, int rows, cudaStream_t s);
cudaError_t launch_spec_accept(const AcceptSampleArgs& a, cudaStream_t s);

// ------------------------------------------------ hidden-state DP (dp.cu)
constexpr int kDpMaxStates = 128;   // skipped weights 0 .. 127 (the TPT grid kernel's candidate limit)
cudaError_t launch_dp_cos(const float* A, long long stride, int n, const float* B, const int32_t* hidx, int r, int d,
                          float* sig, cudaStream_t s);
cudaError_t launch_dp_select(int J, int w, float tau, const int* valid_prev, const float* sig_e, const float* sig_s,
                             int* valid_cur, float* sig_cur, uint8_t* choice, int* src, cudaStream_t s);
cudaError_t launch_dp_gather(int J, const int* src, const int* valid_cur, const float* E, const float* G_prev,
                             long long stride, const float* X, const int32_t* hidx, int r, int d, float* G_cur,
                             cudaStream_t s);
cudaError_t launch_dp_backtrack(const int* js, int n_cand, int n_items, int J, const uint8_t* choices, const int* w,
                                uint8_t* masks, cudaStream_t s);
cudaError_t launch_dp_candidates(int J, const int* valid, int* js, int* n_cand, cudaStream_t s);

}  // namespace ks
