"""GPU parity against the plain fp32 C++ oracle (oracle/cpp/ksoracle.cpp), the
same passages as the fp64 numpy oracle's parity tests (Sec. 2, 2.1, 3.3, 3.4):

* tiny fp32 workload (4 layers, 256- and 200-token prompts whose greedy
  decisions are clear of near-ties): the pending token, the drafts of a skip
  mask, the acceptance count and new tokens of every verify pass equal the
  C++ oracle's; logits of the prefill's last rows and of a verify pass
  within 1e-4 per row; the history states' sublayer updates within 1e-4 per
  row;
* small bf16 model (2 layers, d 512, ragged d_ff and vocabulary, QK-norm):
  the C++ oracle fed the same bf16 weight values (as fp32) and the GPU's
  tokens: verify logits within 2e-2 per row;
* the knapsack (a5) on the GPU equal, bit for bit, to the C++ oracle's
  knapsack on the same integer weights and quantised values."""
import numpy as np
import pytest

from helpers import need_gpu, rel_err, token_ok
from oracle import cxx

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    need_gpu()
    cxx.build()


def _models(shape, max_seq, seed=0):
    from paper_2602_20217_gb300 import synth
    from paper_2602_20217_gb300.model import Model
    m = Model(shape, max_seq=max_seq, seed=seed)
    s = cxx.Session(cxx.Model(shape, synth.np_model_weights(shape, seed=seed)), max_seq)
    return m, s


def test_tiny_fp32_against_the_cxx_oracle():
    from paper_2602_20217_gb300 import synth
    from paper_2602_20217_gb300.configs import TINY
    prompt = synth.prompt_tokens(TINY, 256, seed=1)
    m, s = _models(TINY, 512)
    pend = m.prefill(prompt)
    ref_pend = s.prefill(prompt)
    assert pend == ref_pend
    lg = m.logits(16)
    # the prefill's last rows: the C++ oracle's logits of the same rows
    ref_lg, _ = cxx.Session(s.m, 512).forward(prompt, 0)
    assert rel_err(lg, ref_lg[-16:]) < 1e-4
    mask = np.array([0, 1, 1, 1, 0, 1, 1, 1], np.uint8)
    for step in range(4):
        drafts = m.draft(mask, 4)
        ref_drafts = s.draft(mask, 4)
        assert list(drafts) == list(ref_drafts), step
        a, new = m.verify(None, 4)
        ref_a, ref_new = s.verify(ref_drafts)
        assert (a, list(new)) == (ref_a, list(ref_new)), step
    # a verify pass's logits against the oracle's forward over the same rows
    p, pend = s.position()
    rows = [pend] + list(s.draft(mask, 4))
    g_rows = [m.position()[1]] + list(m.draft(mask, 4))
    assert rows == g_rows
    m.verify(None, 4)
    ref, states = s.forward(rows, p, capture=True)
    got = m.logits(5)
    assert rel_err(got, ref) < 1e-4
    for r in range(5):
        assert token_ok(int(np.argmax(got[r])), ref[r], 1e-3)
    m.close()
    s.close()


def test_history_states_against_the_cxx_oracle():
    from paper_2602_20217_gb300 import synth
    from paper_2602_20217_gb300.configs import TINY
    prompt = synth.prompt_tokens(TINY, 200, seed=3)
    m, s = _models(TINY, 512)
    assert m.prefill(prompt) == s.prefill(prompt)
    mask = np.array([0, 1] * TINY.n_layers, np.uint8)
    for _ in range(3):
        d = m.draft(mask, 3)
        assert list(d) == s.draft(mask, 3)
        a, new = m.verify(None, 3)
        assert (a, list(new)) == s.verify(d)
    got, ref = m.history().astype(np.float64), s.history().astype(np.float64)
    assert got.shape == ref.shape
    for i in range(1, got.shape[0]):          # each sublayer's update, per row
        assert rel_err(got[i] - got[i - 1], ref[i] - ref[i - 1]) < 1e-4, i
    m.close()
    s.close()


def test_small_bf16_verify_logits_against_the_cxx_oracle():
    from paper_2602_20217_gb300 import synth
    from paper_2602_20217_gb300.configs import ModelShape
    shape = ModelShape("small-bf16", 2, 512, 8, 2, 128, 1368, 2000, qk_norm=True, dtype="bf16",
                       rope_theta=500000.0)
    prompt = synth.prompt_tokens(shape, 300, seed=1)
    m, s = _models(shape, 512)
    pend = m.prefill(prompt)
    s.prefill(prompt)
    mask = np.array([0, 1, 1, 1], np.uint8)
    drafts = m.draft(mask, 4)
    m.verify(None, 4)
    got = m.logits(5)
    # the oracle runs the GPU's rows (its own greedy tokens may differ at near-ties)
    ref, _ = s.forward([pend] + list(drafts), 300)
    assert rel_err(got, ref) < 2e-2
    m.close()
    s.close()


def test_knapsack_against_the_cxx_oracle():
    import torch
    from oracle import select as S
    from paper_2602_20217_gb300 import knapspec as ks
    rng = np.random.default_rng(17)
    for n, budget in [(8, 5), (64, 40), (128, 300)]:
        units = rng.integers(1, 6, n).astype(np.int32)
        s32 = rng.uniform(0.3, 1.0, n).astype(np.float32)
        lat, keep = ks.latency(1, units=units)
        sims = torch.tensor(s32, device="cuda")
        mask = torch.zeros(n, dtype=torch.uint8, device="cuda")
        obj = torch.zeros(1, dtype=torch.float64, device="cuda")
        nbytes = ks.ks_select_scratch_bytes(n, budget)
        scratch = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
        ks.ks_select_mask(lat, sims, 0, n, budget, mask, obj, None, scratch, nbytes)
        torch.cuda.synchronize()
        ref_mask, ref_val = cxx.knapsack(units, S.quantize_values(s32), budget)
        assert np.array_equal(mask.cpu().numpy(), ref_mask)
        assert abs(float(obj.item()) - ref_val / S.Q_SCALE) <= 1e-6
