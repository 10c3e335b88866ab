"""GPU parity of the hidden-state DP of Alg. 1 and the TPT selection over its
candidates (Sec. 3.4, 3.5; a NEXT row) against the oracle (oracle/dp.py).

The oracle rebuilds the GPU's state from the committed tokens (a committed
row's target states depend only on the tokens up to it), runs Alg. 1 on the
same history rows, and records how far each of its decisions was from
flipping.  Checks:
* fp32 model (a prompt on which no oracle decision is within 1e-4 of
  flipping, asserted): the same candidates (the same skipped weights, the
  same layer sets);
* bf16 model (every oracle decision clear by more than 1e-2, asserted): the
  same candidates and layer sets as the oracle, acceptances equal up to rows
  whose top-2 logits lie within the bf16 logit tolerance;
* acceptances equal up to rows whose top-2 logits lie within 1e-3;
* the Eq. 3 grid on the GPU's acceptances picks the GPU's (S, gamma) with the
  same TPT bits;
* structural facts on a bf16 model (skipped weight of every layer set = its
  j, the full model last with acceptance 1);
* the target's K/V cache is unchanged by the DP."""
import numpy as np
import pytest

from helpers import need_gpu, oracle_model
from oracle import dp as DP
from oracle import decoder as D
from oracle import select as S

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    need_gpu()


def _setup(shape, prompt_len, n_gen, seed=0):
    from paper_2602_20217_gb300 import knapspec as ks
    from paper_2602_20217_gb300 import synth
    from paper_2602_20217_gb300.model import Model
    m = Model(shape, max_seq=512, seed=seed)
    prompt = synth.prompt_tokens(shape, prompt_len, seed=1)
    m.prefill(prompt)
    out, st, acc = m.generate(n_gen, 3, mask=np.array([0, 1] * shape.n_layers, np.uint8))
    p, pending = m.position()
    r_hist = int(ks.ks_debug_read(m.h, 4, 0, 0, 0, np.zeros(1, np.int32))[0])
    seq = list(prompt) + [int(t) for t in out[: p - len(prompt)]]
    return m, seq, p, r_hist


def _top2(logits):
    part = np.sort(logits, axis=-1)
    return part[:, -1] - part[:, -2]


def _logits(states, w, eps):
    x = np.asarray(states, np.float64)
    x = x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps) * w["final_norm"]
    return x @ w["lm_head"].T


@pytest.mark.parametrize("units_kind", ["ones", "two_one"])
def test_dp_candidates_match_the_oracle_fp32(units_kind):
    from paper_2602_20217_gb300 import knapspec as ks
    from paper_2602_20217_gb300.configs import TINY
    shape = TINY
    m, seq, p, r_hist = _setup(shape, 37, 26)
    n_sub = shape.n_sublayers
    units = np.array([1] * n_sub if units_kind == "ones" else [2, 1] * shape.n_layers, np.int32)
    lat = ks.latency(1, units=units)
    max_rows, tau, D_gamma = 16, 0.5, 6
    r = min(r_hist, max_rows)
    k_before = m.kv(0, p - r, r, "k").copy()
    v_before = m.kv(shape.n_layers - 1, p - r, r, "v").copy()
    mask, g, tpt, js, alphas, cands = m.select_dp(lat, D_gamma, tau=tau, max_states=64, max_rows=max_rows)
    assert np.array_equal(m.kv(0, p - r, r, "k"), k_before)
    assert np.array_equal(m.kv(shape.n_layers - 1, p - r, r, "v"), v_before)

    cfg, w = oracle_model(shape, seed=0)
    s = D.Session(cfg, w, p + 8, hist_steps=5, hist_init_rows=r)
    s.prefill(seq)
    assert s.p == p
    hist = s.history()
    margins = []
    states, sig, choices = DP.run_dp(s, hist, list(units), tau, margins)
    ref_js = sorted(states, reverse=True)
    ref_masks = [DP.backtrack(choices, list(units), j) for j in ref_js]
    # every oracle decision is clear of its threshold (this prompt and
    # generation length were chosen so), so the candidates must be equal
    assert min(margins) > 1e-4, min(margins)
    assert list(js) == ref_js
    assert np.array_equal(cands, np.array(ref_masks))
    # acceptances: rows with a near-tied prediction may go either way
    tgt_logits = _logits(hist[-1], w, cfg.rms_eps)
    for j, a_gpu in zip(js, alphas):
        if j not in states:
            continue
        sl = _logits(states[j], w, cfg.rms_eps)
        unsure = np.count_nonzero((_top2(sl) < 1e-3) | (_top2(tgt_logits) < 1e-3))
        a_ref = S.alpha_hat(np.argmax(sl, -1), np.argmax(tgt_logits, -1))
        assert abs(a_gpu - a_ref) <= unsure / r + 1e-12
    # the grid on the GPU's acceptances
    c, g_ref, v_ref = S.select_tpt(list(cands), list(alphas), shape.n_layers, D_gamma, units=units)
    assert g == g_ref and tpt == v_ref and np.array_equal(mask, cands[c])


def test_dp_candidates_match_the_oracle_bf16():
    from paper_2602_20217_gb300 import knapspec as ks
    from paper_2602_20217_gb300.configs import ModelShape
    shape = ModelShape("small-bf16", 2, 512, 8, 2, 128, 1368, 2000, qk_norm=True, dtype="bf16",
                       rope_theta=500000.0)
    m, seq, p, r_hist = _setup(shape, 45, 30)
    units = np.ones(shape.n_sublayers, np.int32)
    lat = ks.latency(1, units=units)
    max_rows, tau, D_gamma = 16, 0.5, 6
    r = min(r_hist, max_rows)
    mask, g, tpt, js, alphas, cands = m.select_dp(lat, D_gamma, tau=tau, max_states=32, max_rows=max_rows)
    cfg, w = oracle_model(shape, seed=0)
    s = D.Session(cfg, w, p + 8, hist_steps=5, hist_init_rows=r)
    s.prefill(seq)
    assert s.p == p
    hist = s.history()
    margins = []
    states, sig, choices = DP.run_dp(s, hist, list(units), tau, margins)
    # bf16 states differ from the fp64 oracle's by about 1e-3 in cosine; every
    # decision here is clear by more than ten times that
    assert min(margins) > 1e-2, min(margins)
    ref_js = sorted(states, reverse=True)
    assert list(js) == ref_js
    assert np.array_equal(cands, np.array([DP.backtrack(choices, list(units), j) for j in ref_js]))
    tgt_logits = _logits(hist[-1], w, cfg.rms_eps)
    tol = lambda lg: 2e-2 * np.max(np.abs(lg), axis=-1)
    for j, a_gpu in zip(js, alphas):
        sl = _logits(states[j], w, cfg.rms_eps)
        unsure = np.count_nonzero((_top2(sl) < tol(sl)) | (_top2(tgt_logits) < tol(tgt_logits)))
        a_ref = S.alpha_hat(np.argmax(sl, -1), np.argmax(tgt_logits, -1))
        assert abs(a_gpu - a_ref) <= unsure / r + 1e-12
    c, g_ref, v_ref = S.select_tpt(list(cands), list(alphas), shape.n_layers, D_gamma, units=units)
    assert g == g_ref and tpt == v_ref and np.array_equal(mask, cands[c])


def test_dp_structure_bf16():
    from paper_2602_20217_gb300 import knapspec as ks
    from paper_2602_20217_gb300.configs import ModelShape
    shape = ModelShape("small-bf16", 2, 512, 8, 2, 128, 1368, 2000, qk_norm=True, dtype="bf16",
                       rope_theta=500000.0)
    m, seq, p, r_hist = _setup(shape, 45, 30)
    lat = ks.latency(0, 0.08, 2e-5, 0.05)
    mask, g, tpt, js, alphas, cands = m.select_dp(lat, 8, tau=0.5, max_states=32, max_rows=24)
    # integer weights of this latency model at context p (Sec. 3.4)
    ta, tm = 2e-5 * p + 0.05, 0.08
    dl = min(ta, tm)
    wa, wm = max(1, S.round_half_away(ta / dl)), max(1, S.round_half_away(tm / dl))
    wts = [wa, wm] * shape.n_layers
    assert list(js) == sorted(js, reverse=True) and js[-1] == 0
    for j, mk in zip(js, cands):
        assert sum(wi for wi, x in zip(wts, mk) if not x) == j
    assert list(cands[-1]) == [1] * shape.n_sublayers and alphas[-1] == 1.0
    assert all(0.0 <= a <= 1.0 for a in alphas)
    c, g_ref, v_ref = S.select_tpt(list(cands), list(alphas), shape.n_layers, 8, ta, tm)
    assert g == g_ref and tpt == v_ref and np.array_equal(mask, cands[c])
    # decoding continues losslessly after the DP (the cache was restored)
    ar_model, _, _, _ = _setup(shape, 45, 30)
    a1 = ar_model.decode_greedy(12)
    a2 = m.decode_greedy(12)
    assert list(a1) == list(a2)


@pytest.mark.parametrize("kind", ["tiny", "bf16"])
def test_dp_policy_in_the_loop_is_lossless(kind):
    from paper_2602_20217_gb300 import knapspec as ks
    from paper_2602_20217_gb300.configs import ModelShape, TINY
    shape = TINY if kind == "tiny" else ModelShape("small-bf16", 2, 512, 8, 2, 128, 1368, 2000, qk_norm=True,
                                                   dtype="bf16", rope_theta=500000.0)
    m, seq, p, r_hist = _setup(shape, 31, 12)
    m2, _, _, _ = _setup(shape, 31, 12)
    ar = m2.decode_greedy(40)
    lat = ks.latency(1, units=np.array([2, 1] * shape.n_layers, np.int32))
    out, st, acc = m.generate(40, 3, latency=lat, resolve_every=5, dp=(6, 0.5, 64, 16))
    assert list(out) == list(ar)
    assert st.resolves >= 2
