"""Pins of the Alg. 1 oracle (oracle/dp.py) to things other than itself: the
recorded target states, a replay of each backtracked layer set from scratch,
brute force over every layer set of the same skipped weight, and the pruning
limits."""
import itertools

import numpy as np
import pytest

from oracle import decoder as D
from oracle import dp as DP
from oracle import select as S

from test_oracle_decoder import rand_weights, tiny_cfg


def _session(L=2, seed=41, steps=3, std=0.5):
    cfg = tiny_cfg(L=L, qk_norm=True)
    w = rand_weights(cfg, seed=seed, std=std)
    prompt = np.random.default_rng(seed + 1).integers(0, cfg.vocab, 14)
    s = D.Session(cfg, w, 96, hist_steps=5, hist_init_rows=4)
    s.prefill(prompt)
    mask = np.array([0, 1] * L, np.uint8)
    for _ in range(steps):
        s.verify(s.draft(mask, 2))
    return cfg, w, s


def _replay(s, mask, hist):
    """f^(S) on X^(0) of the history rows, sublayer by sublayer, with the
    target's K/V for earlier positions and the rows' own K/V."""
    r = hist.shape[1]
    x = hist[0].copy()
    kv = {l: (s.k[l].copy(), s.v[l].copy()) for l in range(s.cfg.n_layers)}
    for i in range(1, hist.shape[0]):
        if mask[i - 1]:
            x = DP.sublayer(s, i, x, s.p - r, kv)
    return x


def test_sublayer_on_target_states_reproduces_the_next_state():
    cfg, w, s = _session()
    hist = s.history()
    r = hist.shape[1]
    for i in range(1, hist.shape[0]):
        kv = {(i - 1) // 2: (s.k[(i - 1) // 2].copy(), s.v[(i - 1) // 2].copy())}
        got = DP.sublayer(s, i, hist[i - 1], s.p - r, kv)
        assert np.max(np.abs(got - hist[i])) < 1e-10, i


@pytest.mark.parametrize("weights", [[1, 1, 1, 1], [2, 1, 2, 1], [1, 3, 2, 2]])
def test_backtracked_sets_replay_to_their_states(weights):
    cfg, w, s = _session()
    hist = s.history()
    states, sig, choices = DP.run_dp(s, hist, weights, tau=0.0)
    assert 0 in states and np.array_equal(states[0], hist[-1])
    for j, st in states.items():
        mask = DP.backtrack(choices, weights, j)
        assert sum(wi for wi, m in zip(weights, mask) if not m) == j          # skipped weight = j
        assert np.max(np.abs(_replay(s, mask, hist) - st)) < 1e-12
        assert abs(S.matrix_cos(st, hist[-1]) - sig[j]) < 1e-12
    assert max(states) <= sum(weights) // 2


@pytest.mark.parametrize("weights", [[1, 1, 1, 1], [2, 1, 1, 2]])
def test_dp_never_beats_brute_force(weights):
    cfg, w, s = _session(seed=47)
    hist = s.history()
    states, sig, choices = DP.run_dp(s, hist, weights, tau=-1.0)
    best = {}
    for bits in itertools.product([0, 1], repeat=len(weights)):
        mask = np.array(bits, np.uint8)
        j = sum(wi for wi, m in zip(weights, mask) if not m)
        if j > sum(weights) // 2:
            continue
        c = S.matrix_cos(_replay(s, mask, hist), hist[-1])
        best[j] = max(best.get(j, -2.0), c)
    for j, v in sig.items():
        assert v <= best[j] + 1e-12
    assert set(sig) == set(best)            # tau = -1 keeps every reachable skipped weight


def test_single_sublayer_choice_is_exact():
    # one executed sublayer with weight 1: the DP compares exactly the two
    # candidates, so it matches brute force
    cfg, w, s = _session(L=1, seed=53)
    hist = s.history()
    weights = [1, 1]
    states, sig, choices = DP.run_dp(s, hist, weights, tau=-1.0)
    for j in sig:
        cands = [m for m in ([1, 1], [0, 1], [1, 0], [0, 0]) if sum(1 - x for x in m) == j]
        best = max(S.matrix_cos(_replay(s, np.array(m, np.uint8), hist), hist[-1]) for m in cands)
        assert abs(sig[j] - best) < 1e-12


def test_pruning_limits():
    cfg, w, s = _session(seed=59)
    hist = s.history()
    states, sig, _ = DP.run_dp(s, hist, [1, 1, 1, 1], tau=1.0 - 1e-12)
    assert set(states) == {0}                # only the target's own states reach cos 1
    states, sig, _ = DP.run_dp(s, hist, [1, 1, 1, 1], tau=-1.0)
    assert max(states) <= 2                  # K / 2


def test_select_dp_picks_the_tpt_maximum():
    cfg, w, s = _session(seed=61)
    mask, g, v, masks, alphas, js = DP.select_dp(s, [1, 1, 1, 1], 6, tau=0.0, ta=1.0, tm=1.0)
    assert js == sorted(js, reverse=True)
    assert v == max(S.expected_tokens_iter(a, gg) / (gg * S.t_draft(m, 1.0, 1.0) + S.t_target(cfg.n_layers, 1.0, 1.0))
                    for m, a in zip(masks, alphas) for gg in range(1, 7))
    assert js[-1] == 0 and alphas[-1] == 1.0 and list(masks[-1]) == [1, 1, 1, 1]   # j = 0: the full model, last
