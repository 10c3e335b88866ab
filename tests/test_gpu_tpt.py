"""GPU parity of the TPT stage (Sec. 3.5, Alg. 2; a NEXT row) against the
oracle, computed on the GPU's own history states:

* the candidate set (one knapsack optimum per frontier budget) bit for bit;
* Eq. 4's acceptance per candidate: the oracle's prediction on each history
  row from the same first-order draft state; rows where either the
  candidate's or the full set's top-2 logits lie within a tolerance may break
  either way and are allowed to differ;
* the Eq. 3 grid search: given the GPU's acceptances the oracle picks the same
  candidate and gamma, with the same TPT bits;
* the TPT policy in the full loop stays lossless (Sec. 2.1)."""
import numpy as np
import pytest

from helpers import need_gpu, oracle_model
from oracle import select as S

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    need_gpu()


def _top2_margin(logits):
    part = np.sort(logits, axis=-1)
    return part[:, -1] - part[:, -2]


def _logits(states, w, eps):
    x = np.asarray(states, np.float64)
    x = x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps) * w["final_norm"]
    return x @ w["lm_head"].T


def _check(shape, prompt_len, latency_kind, K, D, tol):
    from paper_2602_20217_gb300 import knapspec as ks
    from paper_2602_20217_gb300 import synth
    from paper_2602_20217_gb300.model import Model
    cfg, w = oracle_model(shape, seed=0)
    m = Model(shape, max_seq=512, seed=0)
    m.prefill(synth.prompt_tokens(shape, prompt_len, seed=1))
    n_sub = shape.n_sublayers
    m.generate(30, 3, mask=np.array([0, 1] * shape.n_layers, np.uint8))   # fills the history
    if latency_kind == 1:
        units = synth.unit_table(n_sub, seed=2)
        lat = ks.latency(1, units=units)
    else:
        lat = ks.latency(0, 0.08, 2e-5, 0.05)
    mask, g, tpt, alphas, cand = m.select_tpt(lat, K, D)

    hist = m.history()
    sims, r = m.history_similarities()
    pos = m.position()[0]
    if latency_kind == 1:
        wts = S.sublayer_units(n_sub, units=units)
    else:
        wts = S.sublayer_units(n_sub, 0.08, 2e-5, 0.05, n=pos)
    ref_masks, _ = S.frontier(wts, S.quantize_values(sims), K)
    for j in range(K):
        assert np.array_equal(cand[j], ref_masks[j]), j

    full_logits = _logits(hist[-1], w, cfg.rms_eps)
    full_tok = np.argmax(full_logits, axis=-1)
    full_m = _top2_margin(full_logits)
    for j in range(K):
        lg = _logits(S.draft_states(hist, cand[j]), w, cfg.rms_eps)
        pred = np.argmax(lg, axis=-1)
        a_ref = S.alpha_hat(pred, full_tok)
        unsure = int(np.count_nonzero((_top2_margin(lg) < tol) | (full_m < tol)))
        assert abs(alphas[j] * r - a_ref * r) <= unsure + 1e-9, (j, alphas[j], a_ref, unsure)

    if latency_kind == 1:
        ref = S.select_tpt(list(cand), list(alphas), shape.n_layers, D, units=units)
    else:
        ta = S.t_attn(pos, 2e-5, 0.05)
        ref = S.select_tpt(list(cand), list(alphas), shape.n_layers, D, ta=ta, tm=0.08)
    assert ref[1] == g and ref[2] == tpt   # the same double operations in the same order
    assert np.array_equal(mask, cand[ref[0]])
    m.close()


@pytest.mark.parametrize("latency_kind", [0, 1])
def test_tpt_stage_tiny_fp32(latency_kind):
    from paper_2602_20217_gb300.configs import TINY
    _check(TINY, 256, latency_kind, 6, 10, 1e-3)   # D = 10, the paper's (Sec. 3.5, Alg. 2)


def test_tpt_stage_small_bf16():
    from paper_2602_20217_gb300.configs import ModelShape
    shape = ModelShape("small-bf16", 2, 512, 8, 2, 128, 1368, 2000, qk_norm=True, dtype="bf16",
                       rope_theta=500000.0)
    _check(shape, 300, 0, 4, 10, 0.05)


def test_tpt_policy_is_lossless():
    from paper_2602_20217_gb300 import knapspec as ks
    from paper_2602_20217_gb300 import synth
    from paper_2602_20217_gb300.configs import TINY
    from paper_2602_20217_gb300.model import Model
    m = Model(TINY, max_seq=512, seed=0)
    prompt = synth.prompt_tokens(TINY, 256, seed=1)
    m.prefill(prompt)
    ar = m.decode_greedy(48)
    lat = ks.latency(1, units=synth.unit_table(TINY.n_sublayers, seed=2))
    for T in (1, 4):
        m.prefill(prompt)
        out, st, acc = m.generate(48, 4, latency=lat, resolve_every=T, tpt=(8, 10))
        assert list(out) == list(ar)
        assert st.resolves == (st.steps + T - 1) // T
        assert max(acc) <= 10
    m.close()


def test_tpt_policy_bf16_with_long_drafts_is_lossless():
    """The TPT policy with D = 10 on a bf16 model: verify passes of up to 11
    rows (two rounds of query rows in attention, one CTA per SM in the
    chained projections), speculative output equal to greedy output."""
    from paper_2602_20217_gb300 import knapspec as ks
    from paper_2602_20217_gb300 import synth
    from paper_2602_20217_gb300.configs import ModelShape
    from paper_2602_20217_gb300.model import Model
    shape = ModelShape("small-bf16", 2, 512, 8, 2, 128, 1368, 2000, qk_norm=True, dtype="bf16",
                       rope_theta=500000.0)
    m = Model(shape, max_seq=1024, seed=0)
    prompt = synth.prompt_tokens(shape, 300, seed=1)
    m.prefill(prompt)
    ar = m.decode_greedy(160)
    # fixed masks with long drafts: verify passes of 11 and 16 rows
    for gamma, mask in ((10, [0, 1, 0, 1]), (15, [1, 1, 0, 1])):
        m.rewind()
        out, st, acc = m.generate(160, gamma, mask=np.array(mask, np.uint8))
        assert list(out) == list(ar), gamma
        assert st.drafted == gamma * st.steps
    # the TPT policy choosing gamma up to D = 10
    lat = ks.latency(1, units=np.array([10, 1] * shape.n_layers, np.int32))
    m.rewind()
    out, st, acc = m.generate(160, 4, latency=lat, resolve_every=2, tpt=(4, 10))
    assert list(out) == list(ar)
    assert max(acc) <= 10
    m.close()
