"""Oracle for KnapSpec's layer selection.  fp64 / exact integers.
TEST INFRASTRUCTURE ONLY.

Follows:
* Sec. 2: matrix cosine cos(X, Y) = (1/n) sum_i <X_i, Y_i> / (|X_i| |Y_i|).
* Eq. 1: expected tokens per step  sum_{i=0}^{gamma} alpha^i.
* Eq. 2: TPL(l, gamma);  Eq. 3: TPT(S, gamma) with
  t_Draft(S) = n_Attn(S) t_Attn + n_MLP(S) t_MLP and t_Target = L (t_Attn + t_MLP).
* App. C: t_MLP = c1, t_Attn(n) = c2 n + c3, fitted by least squares.
* Sec. 3.4 "Integer Weight Normalization": Delta = min(t_Attn(n), t_MLP),
  w = round(t / Delta).
* Sec. 3.3: each sublayer is a knapsack item; its latency is the weight and
  its similarity to the target's representation is the value.
* Sec. 3.5 / Alg. 2 / Eq. 4: the TPT stage - candidate layer sets, acceptance
  estimated on the history rows, grid search of Eq. 3 over candidates and
  draft lengths (readings at the end of this file).

Readings (listed in the design notes):
* Item value.  The value of running sublayer i is the similarity the draft
  would lose by skipping it, v_i = 1 - cos(X^(i-1), X^(i)) over the history
  rows; the knapsack maximises sum_{i in S} v_i.  (The paper's own objective
  cos(f(X), f^(S)(X)) is not additive; its hidden-state DP is separate.)
* Budget B is the largest total executed weight (units): sum_{i in S} w_i <= B.
* round(.) is round-half-away-from-zero; every weight is at least 1.
* Values are fixed-point integers q_i = round(v_i * 2^30), computed in double
  from the fp32 similarity.  Among optimal masks the one with the smallest
  integer value of the bitmask (bit i-1 <-> sublayer i) is chosen, which is
  what a DP over items 1..2L that takes an item only on a strict improvement,
  backtracked from item 2L down, returns.
* TPT at alpha = 1 uses the limit gamma + 1.
"""
from __future__ import annotations

import itertools

import numpy as np

Q_SCALE = 2.0 ** 30


# ------------------------------------------------------------- similarity
def row_cos(x: np.ndarray, y: np.ndarray) -> np.ndarray:
    """cos(x_i, y_i) for each row i (fp64)."""
    x = np.asarray(x, np.float64)
    y = np.asarray(y, np.float64)
    return np.sum(x * y, axis=-1) / (np.linalg.norm(x, axis=-1) * np.linalg.norm(y, axis=-1))


def matrix_cos(x: np.ndarray, y: np.ndarray) -> float:
    """Matrix cosine of Sec. 2: the mean over rows of the row cosines."""
    return float(np.mean(row_cos(x, y)))


def sublayer_similarities(hist: np.ndarray) -> np.ndarray:
    """sigma_i = cos(X^(i-1), X^(i)) for i = 1..2L; hist is [2L+1, r, d]."""
    return np.array([matrix_cos(hist[i - 1], hist[i]) for i in range(1, hist.shape[0])])


# ---------------------------------------------------------------- latency
def t_mlp(c1: float) -> float:
    return float(c1)


def t_attn(n: float, c2: float, c3: float) -> float:
    return float(c2) * float(n) + float(c3)


def fit_latency(ns, attn_times, mlp_times):
    """Least-squares fit of App. C's model: returns (c1, c2, c3)."""
    ns = np.asarray(ns, np.float64)
    A = np.stack([ns, np.ones_like(ns)], axis=1)
    (c2, c3), *_ = np.linalg.lstsq(A, np.asarray(attn_times, np.float64), rcond=None)
    c1 = float(np.mean(np.asarray(mlp_times, np.float64)))
    return c1, float(c2), float(c3)


def round_half_away(x: float) -> int:
    """Nearest integer, halves away from zero (exact for every double: the
    fractional part x - floor(x) is computed without rounding)."""
    a = abs(float(x))
    f = np.floor(a)
    r = int(f) + (1 if a - f >= 0.5 else 0)
    return r if x >= 0 else -r


def integer_weights(ta: float, tm: float) -> tuple:
    """(w_Attn, w_MLP) of Sec. 3.4: Delta = min(ta, tm), w = round(t / Delta) >= 1."""
    delta = min(ta, tm)
    return max(1, round_half_away(ta / delta)), max(1, round_half_away(tm / delta))


def sublayer_units(n_sublayers: int, c1=None, c2=None, c3=None, n=None, units=None) -> np.ndarray:
    """Per-sublayer integer weights: explicit units, or from the latency model at
    context length n (odd sublayers 1, 3, ... are Attn, even ones MLP)."""
    if units is not None:
        return np.asarray(units, np.int64)
    wa, wm = integer_weights(t_attn(n, c2, c3), t_mlp(c1))
    return np.array([wa if i % 2 == 1 else wm for i in range(1, n_sublayers + 1)], np.int64)


# --------------------------------------------------------------- knapsack
def quantize_values(sigma) -> np.ndarray:
    """q_i = round((1 - sigma_i) * 2^30), sigma given as fp32, arithmetic in double."""
    s = np.asarray(sigma, dtype=np.float32).astype(np.float64)
    return np.array([round_half_away((1.0 - v) * Q_SCALE) for v in s], dtype=np.int64)


def knapsack(weights, values, budget: int):
    """Exact 0/1 knapsack over items 1..N: maximise sum q_i s.t. sum w_i <= budget.

    best[c] is the best total with weight <= c using the items seen so far; an
    item is taken only when that strictly improves best[c].  Backtracking from
    item N down then yields the optimal mask with the smallest bitmask value.
    Returns (mask uint8[N], total value int)."""
    w = [int(v) for v in weights]
    q = [int(v) for v in values]
    N = len(w)
    if budget < 0:
        raise ValueError("budget must be >= 0")
    best = np.zeros(budget + 1, np.int64)
    take = np.zeros((N, budget + 1), bool)
    for i in range(N):
        # every capacity c >= w_i at once (Sec. 3.4: independent across the budget axis)
        wi = w[i]
        if wi > budget:
            continue
        cand = best[: budget + 1 - wi] + q[i]
        upd = cand > best[wi:]
        new = best.copy()
        new[wi:][upd] = cand[upd]
        take[i, wi:] = upd
        best = new
    mask = np.zeros(N, np.uint8)
    c = budget
    for i in range(N - 1, -1, -1):
        if take[i][c]:
            mask[i] = 1
            c -= w[i]
    return mask, int(best[budget])


def knapsack_brute(weights, values, budget: int):
    """Enumerate every mask; keep the best total, ties to the smaller bitmask."""
    w = np.asarray(weights, np.int64)
    q = np.asarray(values, np.int64)
    N = len(w)
    best_val, best_key = None, None
    for bits in itertools.product((0, 1), repeat=N):
        m = np.array(bits[::-1], np.int64)       # m[i] is bit i of the counter
        if int(m @ w) > budget:
            continue
        val = int(m @ q)
        key = int(sum(int(b) << i for i, b in enumerate(m)))
        if best_val is None or val > best_val or (val == best_val and key < best_key):
            best_val, best_key = val, key
    mask = np.array([(best_key >> i) & 1 for i in range(N)], np.uint8)
    return mask, best_val


def select_mask(sigma, budget: int, n_sublayers: int, c1=None, c2=None, c3=None,
                n=None, units=None):
    """The a5 step: latency -> integer weights -> values -> exact knapsack.

    Returns (mask uint8[2L], objective = sum_{i in S} q_i / 2^30, weights)."""
    w = sublayer_units(n_sublayers, c1, c2, c3, n, units)
    q = quantize_values(sigma)
    mask, total = knapsack(w, q, budget)
    return mask, total / Q_SCALE, w


# ------------------------------------------------------------ throughput
def expected_tokens(alpha: float, gamma: int) -> float:
    """Eq. 1: sum_{i=0}^{gamma} alpha^i."""
    return float(sum(alpha ** i for i in range(gamma + 1)))


def t_draft(mask, ta: float, tm: float) -> float:
    """n_Attn(S) t_Attn + n_MLP(S) t_MLP (odd 1-based sublayers are Attn)."""
    mask = np.asarray(mask)
    n_a = int(mask[0::2].sum())
    n_m = int(mask[1::2].sum())
    return n_a * ta + n_m * tm


def t_target(n_layers: int, ta: float, tm: float) -> float:
    return n_layers * (ta + tm)


def tpt(alpha: float, gamma: int, td: float, tt: float) -> float:
    """Eq. 3: expected tokens per step / (gamma t_Draft + t_Target)."""
    return expected_tokens(alpha, gamma) / (gamma * td + tt)


def tpl(alpha: float, gamma: int, exit_layer: int, n_layers: int) -> float:
    """Eq. 2 (DEL's tokens per layer)."""
    return expected_tokens(alpha, gamma) / (gamma * exit_layer + n_layers)


# ------------------------------------------------- TPT stage (NEXT row 1)
# Alg. 2 selects (S*, gamma*) from a candidate set A of layer sets: the
# knapsack optimum for each of several latency budgets (Sec. 3.3 / 3.5), an
# acceptance estimate alpha_S per candidate from the history (Eq. 4), and a
# grid search of Eq. 3 over A x [D].  Readings (listed in the design notes):
# * A: the optimal masks for the K budgets floor(sum_w * (j + 1) / K), j < K;
# * the draft's final hidden state on a history row is estimated to first
#   order from the recorded sublayer outputs: the target's X^(2L) minus the
#   contribution X^(i) - X^(i-1) of every skipped sublayer i (the paper's
#   propagated DP state of Alg. 1 is not built);
# * a prediction is the argmax of the LM head on the final-normalised state,
#   and the target tokens are those of the full layer set on the same rows;
# * Eq. 1 is summed term by term with alpha^i formed by repeated products.
def frontier_budgets(total_w: int, k: int) -> list:
    """Candidate budgets floor(total_w * (j + 1) / K) for j = 0..K-1."""
    return [(int(total_w) * (j + 1)) // int(k) for j in range(int(k))]


def frontier(weights, values, k: int):
    """The candidate set A: one optimal knapsack mask per candidate budget.
    Returns (list of uint8 masks, list of budgets)."""
    budgets = frontier_budgets(int(np.sum(weights)), k)
    return [knapsack(weights, values, c)[0] for c in budgets], budgets


def draft_states(hist: np.ndarray, mask) -> np.ndarray:
    """First-order final state of f^(S) on the history rows: X^(2L) minus the
    recorded contribution of each skipped sublayer.  hist is [2L+1, r, d]."""
    hist = np.asarray(hist, np.float64)
    h = hist[-1].copy()
    for i in range(1, hist.shape[0]):
        if not mask[i - 1]:
            h -= hist[i] - hist[i - 1]
    return h


def lm_argmax(states: np.ndarray, lm_head: np.ndarray, final_gain: np.ndarray, eps: float) -> np.ndarray:
    """Token predicted from each row: final RMSNorm, LM head, argmax (ties to
    the lowest id)."""
    x = np.asarray(states, np.float64)
    x = x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps) * np.asarray(final_gain, np.float64)
    return np.argmax(x @ np.asarray(lm_head, np.float64).T, axis=-1).astype(np.int64)


def alpha_hat(pred, target) -> float:
    """Eq. 4: the fraction of history rows on which the draft's prediction
    equals the target's token."""
    pred = np.asarray(pred)
    return float(np.count_nonzero(pred == np.asarray(target))) / float(len(pred))


def expected_tokens_iter(alpha: float, gamma: int) -> float:
    """Eq. 1 as a sum, alpha^i by repeated products (the order the device uses)."""
    e, p = 1.0, 1.0
    for _ in range(int(gamma)):
        p = p * alpha
        e = e + p
    return e


def select_tpt(masks, alphas, n_layers: int, max_gamma: int, ta: float = None, tm: float = None, units=None):
    """Alg. 2's grid search: candidates in order, gamma = 1..D ascending, a pair
    replaces the best only when its TPT (Eq. 3) is strictly larger.  Latencies
    are t_Attn / t_MLP, or explicit per-sublayer units.
    Returns (candidate index, gamma, tpt)."""
    best = (-1, 0, 0.0)
    if units is not None:
        units = [float(u) for u in units]
        tt = float(sum(units))
    else:
        tt = t_target(n_layers, ta, tm)
    for j, (m, a) in enumerate(zip(masks, alphas)):
        if units is not None:
            td = 0.0
            for i, u in enumerate(units):
                if m[i]:
                    td = td + u
        else:
            td = t_draft(m, ta, tm)
        for g in range(1, int(max_gamma) + 1):
            v = expected_tokens_iter(a, g) / (g * td + tt)
            if v > best[2]:
                best = (j, g, v)
    return best
