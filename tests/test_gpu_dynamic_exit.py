"""GPU parity of the dynamic drafting exit (Sec. 3.5, a NEXT row):

* a draft token's confidence (its softmax probability over the draft's
  logits) equals the fp64 value computed from the GPU's own logits, and the
  oracle's confidence from its own logits (fp32 model);
* the number of drafts follows the rule exactly on the GPU's confidences
  (stop after the first token below tau, keep it), and the drafts are the
  prefix of the undisturbed draft;
* the verify after an early exit compares only the drafts produced, and the
  full loop stays lossless (Sec. 2.1)."""
import numpy as np
import pytest

from helpers import need_gpu, oracle_model, token_ok
from oracle import decoder as D

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    need_gpu()


def _small_bf16():
    from paper_2602_20217_gb300.configs import ModelShape
    return ModelShape("small-bf16", 2, 512, 8, 2, 128, 1368, 2000, qk_norm=True, dtype="bf16",
                      rope_theta=500000.0)


def _model(shape, prompt_len, seed=0):
    from paper_2602_20217_gb300 import synth
    from paper_2602_20217_gb300.model import Model
    m = Model(shape, max_seq=512, seed=seed)
    prompt = synth.prompt_tokens(shape, prompt_len, seed=1)
    m.prefill(prompt)
    return m, prompt


def _rule(conf, tau, gamma):
    below = [i for i, c in enumerate(conf) if c < tau]
    return below[0] + 1 if below else gamma


@pytest.mark.parametrize("kind", ["tiny", "bf16"])
def test_confidence_is_softmax_max_of_the_draft_logits(kind):
    from paper_2602_20217_gb300.configs import TINY
    shape = TINY if kind == "tiny" else _small_bf16()
    m, prompt = _model(shape, 37)
    mask = np.array([1, 0] * (shape.n_layers // 2) + [0, 1] * (shape.n_layers - shape.n_layers // 2), np.uint8)
    if kind == "tiny":
        cfg, w = oracle_model(shape, seed=0)
        s = D.Session(cfg, w, 512)
        s.prefill(prompt)
    for step in range(6):
        n, conf, toks = m.draft_dynamic(mask, 1, 0.0)
        assert n == 1
        logits = m.logits(1)[0].astype(np.float64)
        # the GPU's confidence from its own logits (fp32 sums of a fixed order)
        assert abs(conf[0] - D.top1_prob(logits)) <= 2e-5 * D.top1_prob(logits)
        assert int(toks[0]) == int(np.argmax(logits))
        if kind == "tiny":
            # and the oracle's confidence from its own fp64 logits
            ref_logits, _ = s.forward([s.pending], s.p, mask=mask)
            ref = s.draft(mask, 1)
            assert abs(conf[0] - s.last_confidence[0]) <= 1e-3 * s.last_confidence[0]
            assert token_ok(toks[0], ref_logits[0], 1e-4)
            if int(toks[0]) != ref[0]:
                break                              # a near-tie broke differently: stop comparing
            a, new = s.verify(ref)
        a_gpu, new_gpu = m.verify(None, 1)
        if kind == "tiny" and list(new_gpu) != new:
            break


@pytest.mark.parametrize("kind", ["tiny", "bf16"])
def test_exit_rule_on_the_gpu_confidences(kind):
    from paper_2602_20217_gb300.configs import TINY
    shape = TINY if kind == "tiny" else _small_bf16()
    m, _ = _model(shape, 41)
    mask = np.array([0, 1] * shape.n_layers, np.uint8)
    gamma = 7
    for step in range(4):
        n_full, conf_full, toks_full = m.draft_dynamic(mask, gamma, 0.0)
        assert n_full == gamma and len(conf_full) == gamma
        # thresholds at, between and around the observed confidences
        taus = sorted(set([0.0, float(np.max(conf_full)) * 1.01, 2.0] + [float(c) for c in conf_full]
                          + [float(c) * 1.0000001 for c in conf_full]))
        for tau in taus:
            n, conf, toks = m.draft_dynamic(mask, gamma, tau)
            assert n == _rule(list(conf_full), np.float32(tau), gamma), (tau, n, conf_full)
            assert np.array_equal(toks, toks_full[:n])
            assert np.array_equal(conf, conf_full[:n])
        # verify after an exit compares only the produced drafts
        tau = float(np.median(conf_full))
        n, _, toks = m.draft_dynamic(mask, gamma, tau)
        a, new = m.verify(None, gamma)
        assert a <= n
        assert np.array_equal(np.asarray(new[:a]), toks[:a])


@pytest.mark.parametrize("kind", ["tiny", "bf16"])
def test_lossless_with_dynamic_exit(kind):
    from paper_2602_20217_gb300.configs import TINY
    shape = TINY if kind == "tiny" else _small_bf16()
    m, _ = _model(shape, 29)
    ar = m.decode_greedy(40)
    mask = np.array([0, 1] * shape.n_layers, np.uint8)
    # confidences of this model's drafts, to place thresholds inside their range
    m2, _ = _model(shape, 29)
    _, conf, _ = m2.draft_dynamic(mask, 8, 0.0)
    for tau in (0.0, float(np.quantile(conf, 0.3)), float(np.quantile(conf, 0.7)), 2.0):
        m3, _ = _model(shape, 29)
        out, st, acc = m3.generate(40, 5, mask=mask, tau_conf=tau)
        assert list(out) == list(ar), tau
        assert st.drafted <= 5 * st.steps
        if tau > 1.0:
            assert st.drafted == st.steps          # one draft per step
        if tau == 0.0:
            assert st.drafted == 5 * st.steps
