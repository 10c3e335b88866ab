"""GPU parity of sampling-mode speculative decoding (Sec. 2.1, sampling
branch; a NEXT row) against the oracle (oracle/sampling.py):

* every draft and target distribution equals the oracle's filtering of the
  GPU's own logits (temperature, top-k, top-p): the same tokens in the same
  order and probabilities within fp32 rounding;
* every drawn token and every acceptance follows the oracle's rule on those
  distributions with the oracle's Philox uniforms (bit-identical draws);
  outcomes whose uniform lies within 1e-5 of a decision boundary may go
  either way;
* full-mask drafts (q == p bit for bit) are always accepted, a near-zero
  temperature reproduces greedy decoding, and the loop equals the step API."""
import numpy as np
import pytest

from helpers import need_gpu
from oracle import sampling as SP

pytestmark = pytest.mark.gpu

TOL = 1e-5


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    need_gpu()


def _small_bf16():
    from paper_2602_20217_gb300.configs import ModelShape
    return ModelShape("small-bf16", 2, 512, 8, 2, 128, 1368, 2000, qk_norm=True, dtype="bf16",
                      rope_theta=500000.0)


def _shape(kind):
    from paper_2602_20217_gb300.configs import TINY
    return TINY if kind == "tiny" else _small_bf16()


def _model(shape, prompt_len):
    from paper_2602_20217_gb300 import synth
    from paper_2602_20217_gb300.model import Model
    m = Model(shape, max_seq=512, seed=0)
    m.prefill(synth.prompt_tokens(shape, prompt_len, seed=1))
    return m


def _check_dist(gpu, logits_row, T, k, p):
    """The GPU's filtered distribution against the oracle's filtering of the
    same logits; a top-p cut whose cumulative sum lies within TOL of top_p may
    keep one token more or less."""
    ids, pr = gpu
    ref_ids, ref_pr = SP.filter_distribution(logits_row, T, k, p)
    n = min(len(ids), len(ref_ids))
    assert np.array_equal(ids[:n], ref_ids[:n])
    if len(ids) != len(ref_ids):
        full_ids, full_pr = SP.filter_distribution(logits_row, T, k, 1.0)
        c = np.cumsum(full_pr)
        assert abs(c[n - 1] - p) < TOL, (len(ids), len(ref_ids))
        return
    assert np.max(np.abs(pr.astype(np.float64) - ref_pr)) < TOL


def _near_cdf_boundary(probs, u):
    c = np.cumsum(np.asarray(probs, np.float64))
    return np.any(np.abs(c - u) < TOL)


@pytest.mark.parametrize("kind", ["tiny", "bf16"])
def test_draft_and_target_distributions_and_draws(kind):
    from paper_2602_20217_gb300 import knapspec as ks
    shape = _shape(kind)
    m = _model(shape, 33)
    T, K, P, seed = 0.7, 50, 0.95, 1234
    samp = ks.sampling(T, K, P, seed)
    mask = np.array([0, 1] * shape.n_layers, np.uint8)
    gamma = 3
    checked = 0
    for step in range(8):
        toks = m.draft_sample(mask, gamma, samp, step)
        q = ks.ks_sample_dists(m.h, "draft", 0, gamma)
        # the last draft pass's logits are still on the device: check q_{gamma-1}
        last = m.logits(1)[0].astype(np.float64)
        _check_dist(q[gamma - 1], last, T, K, P)
        for t in range(gamma):
            ids, pr = q[t]
            u = SP.uniform(seed, step, t, 0)
            if not _near_cdf_boundary(pr, u):
                assert int(toks[t]) == SP.sample(ids, pr.astype(np.float64), u)
        a, new = m.verify_sample(gamma, samp, step)
        p = ks.ks_sample_dists(m.h, "target", 0, gamma + 1)
        logits = m.logits(gamma + 1).astype(np.float64)
        for t in range(gamma + 1):
            _check_dist(p[t], logits[t], T, K, P)
        # the acceptance on the GPU's distributions with the oracle's uniforms
        pd = [(ids, pr.astype(np.float64)) for ids, pr in p]
        qd = [(ids, pr.astype(np.float64)) for ids, pr in q]
        a_ref, new_ref = SP.speculative_step(pd, qd, list(toks), seed, step)
        if (a, list(new)) != (a_ref, new_ref):
            # allowed only at a boundary: an acceptance test or the final draw
            amb = False
            for t in range(min(a, a_ref) + 1):
                if t < gamma:
                    x = int(toks[t])
                    px, qx = SP.prob_of(*pd[t], x), SP.prob_of(*qd[t], x)
                    if qx > 0 and abs(SP.uniform(seed, step, t, 1) - min(1.0, px / qx)) < TOL:
                        amb = True
            u2 = SP.uniform(seed, step, 0, 2)
            t_end = min(a, a_ref)
            res = SP.residual(*pd[t_end], *qd[t_end]) if t_end < gamma else None
            if _near_cdf_boundary(pd[t_end][1], u2) or (res is not None and _near_cdf_boundary(res[1], u2)):
                amb = True
            assert amb, (step, a, list(new), a_ref, new_ref)
            break
        checked += 1
    assert checked >= 4


def test_full_mask_drafts_are_always_accepted():
    from paper_2602_20217_gb300 import knapspec as ks
    shape = _small_bf16()
    m = _model(shape, 21)
    samp = ks.sampling(0.7, 50, 0.95, 99)
    full = np.ones(shape.n_sublayers, np.uint8)
    for step in range(6):
        m.draft_sample(full, 4, samp, step)
        a, new = m.verify_sample(4, samp, step)
        assert a == 4, step


@pytest.mark.parametrize("kind", ["tiny", "bf16"])
def test_near_zero_temperature_is_greedy(kind):
    from paper_2602_20217_gb300 import knapspec as ks
    shape = _shape(kind)
    m = _model(shape, 25)
    ar = m.decode_greedy(30)
    m2 = _model(shape, 25)
    mask = np.array([0, 1] * shape.n_layers, np.uint8)
    out, st, acc = m2.generate(30, 4, mask=mask, sampling=ks.sampling(1e-7, 50, 0.95, 5))
    assert list(out) == list(ar)


def test_loop_equals_step_api():
    from paper_2602_20217_gb300 import knapspec as ks
    shape = _small_bf16()
    mask = np.array([0, 1, 1, 1], np.uint8)
    samp = ks.sampling(0.7, 50, 0.95, 2024)
    m = _model(shape, 30)
    out, st, acc = m.generate(40, 3, mask=mask, sampling=samp)
    m2 = _model(shape, 30)
    toks = [int(out[0])]
    step = 0
    while len(toks) < 40:
        m2.draft_sample(mask, 3, samp, step)
        a, new = m2.verify_sample(3, samp, step)
        toks.extend(int(t) for t in new)
        step += 1
    assert toks[:40] == [int(t) for t in out]
    assert step == st.steps
