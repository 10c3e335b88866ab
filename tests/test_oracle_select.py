"""Pins for the selection oracle (CPU).

What pins what:
* matrix cosine: hand-worked example, cos(X, X) = 1, cos(X, -X) = -1, scale
  invariance, orthogonal rows -> 0.
* Lemma 1 (Sec. 4): equal-norm x' meeting the cosine bound keeps the argmax.
* latency model / integer weights: App. C Table 3 coefficients with hand
  arithmetic (tests/golden/latency_table3.json); least-squares fit recovers
  known coefficients.
* knapsack: brute force over all 2^N masks (N = 8, 12, 16), a textbook
  instance, and the special cases all-weights-one (top-B values), B >= sum w
  (every positive item), B = 0 (empty mask).
* Eq. 1: closed form (1 - a^(g+1)) / (1 - a), limits a -> 0 and a -> 1, and a
  Monte-Carlo truncated-geometric simulation.
* Eq. 3: TPT reduces to TPL (Eq. 2) when t_Attn = t_MLP (Sec. 3.2).
* TPT stage (Alg. 2): the estimated draft states telescope to X^(2L) (full
  set) and X^(0) (empty set) and equal the forward sum of kept
  contributions; each frontier mask is the brute-force optimum of its
  budget; Eq. 4 on the full set is 1; the LM-head argmax against a row-by-row
  loop; the grid search against brute force, alpha = 0 (gamma = 1) and
  alpha = 1 with a cheaper draft (gamma = D).
"""
import json
import os

import numpy as np
import pytest

from oracle import select as S

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ------------------------------------------------------------------ cosine
def test_matrix_cos_hand_example():
    X = np.array([[1.0, 0.0], [1.0, 1.0]])
    Y = np.array([[1.0, 0.0], [0.0, 1.0]])
    assert S.matrix_cos(X, Y) == pytest.approx((1.0 + 1.0 / np.sqrt(2.0)) / 2.0, abs=1e-15)


def test_matrix_cos_invariants():
    rng = np.random.default_rng(0)
    X = rng.standard_normal((7, 33))
    assert S.matrix_cos(X, X) == pytest.approx(1.0, abs=1e-14)
    assert S.matrix_cos(X, -X) == pytest.approx(-1.0, abs=1e-14)
    scales = rng.uniform(0.1, 10.0, size=(7, 1))
    Y = rng.standard_normal((7, 33))
    assert S.matrix_cos(X * scales, Y) == pytest.approx(S.matrix_cos(X, Y), abs=1e-14)
    E = np.eye(4)
    assert S.matrix_cos(E[:2], E[2:]) == 0.0


def test_sublayer_similarities_indexing():
    # X^(0) = X^(1) (a skipped sublayer), X^(2) = -X^(1)
    rng = np.random.default_rng(1)
    x = rng.standard_normal((3, 8))
    hist = np.stack([x, x, -x])
    sig = S.sublayer_similarities(hist)
    assert sig.shape == (2,)
    assert sig[0] == pytest.approx(1.0) and sig[1] == pytest.approx(-1.0)


def test_lemma1_cosine_bound_keeps_argmax():
    """Sec. 4, Lemma 1: |x'| = |x| and cos(x, x') >= 1 - xi^2 / (2 |x|^2 max |w_i* - w_j|^2)."""
    rng = np.random.default_rng(2)
    for trial in range(200):
        V, d = 50, 16
        W = rng.standard_normal((V, d))
        x = rng.standard_normal(d)
        s = W @ x
        i_star = int(np.argmax(s))
        xi = s[i_star] - np.max(np.delete(s, i_star))
        dmax = np.max(np.linalg.norm(W[i_star] - np.delete(W, i_star, axis=0), axis=1))
        bound = 1.0 - xi ** 2 / (2.0 * (x @ x) * dmax ** 2)
        # x' on the sphere |x'| = |x| at cosine exactly 'bound' in a random direction
        u = rng.standard_normal(d)
        u -= (u @ x) / (x @ x) * x
        u /= np.linalg.norm(u)
        c = max(bound, -1.0)
        xp = np.linalg.norm(x) * (c * x / np.linalg.norm(x) + np.sqrt(max(0.0, 1 - c * c)) * u)
        assert S.row_cos(x[None], xp[None])[0] >= bound - 1e-12
        assert int(np.argmax(W @ xp)) == i_star


# ----------------------------------------------------------------- latency
def test_integer_weights_table3_golden():
    with open(os.path.join(GOLDEN, "latency_table3.json")) as f:
        g = json.load(f)
    for c in g["cases"]:
        ta = S.t_attn(c["n"], c["c2"], c["c3"])
        assert ta == pytest.approx(c["t_attn"], rel=1e-12)
        assert S.integer_weights(ta, S.t_mlp(c["c1"])) == (c["w_attn"], c["w_mlp"])


def test_round_half_away():
    assert [S.round_half_away(v) for v in (0.5, 1.5, 2.5, -0.5, -1.5, 2.4999)] == [1, 2, 3, -1, -2, 2]
    # the largest double below 0.5 rounds to 0 (x + 0.5 would round up to 1.0)
    assert S.round_half_away(np.nextafter(0.5, 0.0)) == 0
    assert S.round_half_away(2.0 ** 52 + 1) == 2 ** 52 + 1


def test_sublayer_units_alternate_attn_mlp():
    w = S.sublayer_units(6, c1=1.0, c2=0.001, c3=0.0, n=3000)   # t_A = 3, t_M = 1
    assert list(w) == [3, 1, 3, 1, 3, 1]


def test_fit_latency_recovers_coefficients():
    ns = np.array([1024, 4096, 16384, 65536, 131072], np.float64)
    c1, c2, c3 = 0.3, 2.5e-5, 0.07
    fit = S.fit_latency(ns, c2 * ns + c3, np.full(len(ns), c1))
    assert fit == pytest.approx((c1, c2, c3), rel=1e-9)


# ---------------------------------------------------------------- knapsack
def test_knapsack_textbook_instance():
    mask, total = S.knapsack([1, 3, 4, 5], [1, 4, 5, 7], 7)
    assert total == 9 and list(mask) == [0, 1, 1, 0]


@pytest.mark.parametrize("N,budget_frac,seed", [(8, 0.5, 0), (8, 0.3, 1), (12, 0.6, 2), (16, 0.5, 3)])
def test_knapsack_matches_brute_force(N, budget_frac, seed):
    rng = np.random.default_rng(seed)
    for _ in range(3 if N < 16 else 1):
        w = rng.integers(1, 5, size=N)
        q = rng.integers(-5, 40, size=N) * 3          # coarse values -> many ties
        B = int(budget_frac * w.sum())
        m1, v1 = S.knapsack(w, q, B)
        m2, v2 = S.knapsack_brute(w, q, B)
        assert v1 == v2
        assert list(m1) == list(m2)
        assert int(m1 @ w) <= B


def test_knapsack_special_cases():
    rng = np.random.default_rng(4)
    q = rng.integers(0, 1000, size=10)
    q[3] = q[7]                                         # a tie
    # all weights 1 -> the B largest values (ties: lower index kept)
    m, v = S.knapsack(np.ones(10, int), q, 4)
    order = sorted(range(10), key=lambda i: (-q[i], i))[:4]
    assert v == sum(q[order]) and set(np.flatnonzero(m)) == set(order)
    # budget >= total weight -> every strictly positive item
    w = rng.integers(1, 4, size=10)
    m, v = S.knapsack(w, q - 500, int(w.sum()))
    assert list(m) == [int(x > 0) for x in q - 500]
    # zero budget -> empty mask
    m, v = S.knapsack(w, q, 0)
    assert m.sum() == 0 and v == 0
    with pytest.raises(ValueError):
        S.knapsack(w, q, -1)


def test_quantize_values():
    q = S.quantize_values(np.array([1.0, 0.5, 0.0, -1.0], np.float32))
    assert list(q) == [0, 2 ** 29, 2 ** 30, 2 ** 31]
    # fp32 input: 0.1f is not 0.1
    assert S.quantize_values([0.1])[0] == S.round_half_away((1.0 - float(np.float32(0.1))) * 2 ** 30)


def test_select_mask_tiny_config_vs_brute():
    from paper_2602_20217_gb300 import synth
    units = synth.unit_table(8, seed=2)
    assert set(units) <= {1, 2, 3, 4}
    rng = np.random.default_rng(5)
    sigma = rng.uniform(0.2, 1.0, size=8).astype(np.float32)
    mask, obj, w = S.select_mask(sigma, 5, 8, units=units)
    m2, v2 = S.knapsack_brute(units, S.quantize_values(sigma), 5)
    assert list(mask) == list(m2) and obj == v2 / 2 ** 30


# ------------------------------------------------------------- throughput
@pytest.mark.parametrize("alpha", [0.0, 0.3, 0.9, 0.97])
@pytest.mark.parametrize("gamma", [1, 4, 10])
def test_expected_tokens_closed_form(alpha, gamma):
    closed = (1 - alpha ** (gamma + 1)) / (1 - alpha)
    assert S.expected_tokens(alpha, gamma) == pytest.approx(closed, rel=1e-12)


def test_expected_tokens_limits_and_simulation():
    assert S.expected_tokens(1.0, 7) == 8.0
    assert S.expected_tokens(0.0, 7) == 1.0
    rng = np.random.default_rng(6)
    alpha, gamma, n = 0.8, 4, 200000
    acc = rng.random((n, gamma)) < alpha
    first_reject = np.where(acc.all(1), gamma, np.argmin(acc, axis=1))
    assert np.mean(first_reject + 1) == pytest.approx(S.expected_tokens(alpha, gamma), rel=5e-3)


def test_tpt_reduces_to_tpl_with_equal_latencies():
    L = 8
    mask = np.zeros(2 * L, np.uint8)
    mask[: 2 * 3] = 1                                   # early exit after 3 layers
    t = 0.37
    for alpha in (0.2, 0.7):
        for gamma in (1, 3, 6):
            # t_Draft = 6t, t_Target = 16t: TPT = TPL(exit = 6 sublayers, 2L = 16) / t
            got = S.tpt(alpha, gamma, S.t_draft(mask, t, t), S.t_target(L, t, t))
            assert got == pytest.approx(S.tpl(alpha, gamma, 6, 2 * L) / t, rel=1e-12)


def test_t_draft_counts_attn_and_mlp():
    mask = np.array([1, 0, 1, 1, 0, 1])   # sublayers 1,3 (Attn) and 4,6 (MLP) run
    assert S.t_draft(mask, 10.0, 1.0) == 2 * 10.0 + 2 * 1.0


# ------------------------------------------------------ TPT stage (NEXT-1)
def _history(seed=0, L=3, r=5, d=16):
    rng = np.random.default_rng(seed)
    return np.cumsum(rng.standard_normal((2 * L + 1, r, d)), axis=0)


def test_draft_states_telescope_to_the_endpoints():
    hist = _history()
    n = hist.shape[0] - 1
    assert np.allclose(S.draft_states(hist, np.ones(n, np.uint8)), hist[-1], atol=1e-12)
    assert np.allclose(S.draft_states(hist, np.zeros(n, np.uint8)), hist[0], atol=1e-12)
    mask = np.array([1, 0, 0, 1, 1, 0], np.uint8)
    # the same state built forwards: X^(0) plus the kept contributions
    fwd = hist[0] + sum(hist[i] - hist[i - 1] for i in range(1, n + 1) if mask[i - 1])
    assert np.allclose(S.draft_states(hist, mask), fwd, atol=1e-12)


def test_frontier_is_the_knapsack_optimum_per_budget():
    rng = np.random.default_rng(3)
    w = rng.integers(1, 5, 10)
    q = rng.integers(0, 1000, 10)
    masks, budgets = S.frontier(w, q, 6)
    assert budgets[-1] == int(w.sum()) and budgets == sorted(budgets)
    vals = []
    for m, b in zip(masks, budgets):
        bm, bv = S.knapsack_brute(w, q, b)
        assert np.array_equal(m, bm)
        vals.append(int(m.astype(np.int64) @ q))
    assert vals == sorted(vals)   # a larger budget never lowers the objective


def test_alpha_hat_full_set_is_one_and_lm_argmax_matches_definition():
    rng = np.random.default_rng(1)
    hist = _history(1, L=2, r=7, d=12)
    W = rng.standard_normal((30, 12))
    g = rng.uniform(0.5, 1.5, 12)
    target = S.lm_argmax(hist[-1], W, g, 1e-5)
    full = S.lm_argmax(S.draft_states(hist, np.ones(4, np.uint8)), W, g, 1e-5)
    assert S.alpha_hat(full, target) == 1.0
    # argmax written out row by row
    for i in range(7):
        x = hist[-1][i]
        y = x / np.sqrt(np.mean(x * x) + 1e-5) * g
        assert target[i] == int(np.argmax([W[v] @ y for v in range(30)]))
    assert S.alpha_hat([1, 2, 3, 4], [1, 0, 3, 0]) == 0.5


def test_expected_tokens_iter_matches_closed_form():
    for a in (0.0, 0.3, 0.9, 1.0):
        for g in range(1, 11):
            assert S.expected_tokens_iter(a, g) == pytest.approx(S.expected_tokens(a, g), rel=1e-14)


def test_select_tpt_grid_search_special_cases():
    masks = [np.array([0, 1, 0, 1], np.uint8), np.array([1, 1, 0, 1], np.uint8), np.ones(4, np.uint8)]
    ta, tm = 2.0, 3.0
    # brute force over the same grid
    alphas = [0.4, 0.7, 1.0]
    j, g, v = S.select_tpt(masks, alphas, 2, 10, ta=ta, tm=tm)
    grid = [(S.tpt(a, gg, S.t_draft(m, ta, tm), S.t_target(2, ta, tm)), jj, gg)
            for jj, (m, a) in enumerate(zip(masks, alphas)) for gg in range(1, 11)]
    best = max(grid, key=lambda x: x[0])
    assert (j, g) == (best[1], best[2]) and v == pytest.approx(best[0], rel=1e-12)
    # alpha = 0 everywhere: one draft token is the least waste
    assert S.select_tpt(masks, [0.0] * 3, 2, 10, ta=ta, tm=tm)[1] == 1
    # alpha = 1 with a draft cheaper than the target: TPT grows with gamma
    j1, g1, _ = S.select_tpt(masks[:1], [1.0], 2, 10, ta=ta, tm=tm)
    assert (j1, g1) == (0, 10)
    # explicit units act as latencies
    u = [1, 2, 1, 2]
    ju, gu, vu = S.select_tpt(masks, alphas, 2, 4, units=u)
    gridu = [(S.expected_tokens(a, gg) / (gg * float(np.dot(m, u)) + 6.0), jj, gg)
             for jj, (m, a) in enumerate(zip(masks, alphas)) for gg in range(1, 5)]
    bu = max(gridu, key=lambda x: x[0])
    assert (ju, gu) == (bu[1], bu[2])
