"""GPU parity of the Attn sublayer at long context (Sec. 2; the split-KV
attention kernel, its merge and the fused RoPE / QK-norm / K-V write) against
the oracle's attention sublayer (oracle/decoder.py).

A 40000-token prompt spans all three chunk regions of the key axis (128-key
chunks below 8192, 512-key chunks below 32768, 2048-key chunks beyond, and a
ragged last chunk).  The oracle cannot run the whole prompt, so each check is
local to one sublayer: for every committed row in the GPU's history ring and
every layer, the oracle applies f^(2l-1) to the GPU's own input state X^(2l-2)
of that row, attending to the GPU's K/V cache for the earlier positions (the
row's own K/V the oracle computes itself), and the result must match the
GPU's X^(2l-1) within the logits tolerance (2e-2 of the sublayer's update).
Rows come from the pass shapes the kernel specialises on: the prefill's last
16-row pass (three rounds of query tiles) and verify passes with R = 4 and
R = 5.  Greedy R = 1 passes leave no history rows, so the last one is checked
through its logits: the oracle runs that row through every layer on the GPU's
caches for the earlier positions."""
import numpy as np
import pytest

from helpers import need_gpu, oracle_model
from oracle import decoder as D

pytestmark = pytest.mark.gpu

N_PROMPT = 40000


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    need_gpu()


def _shape(hd):
    """hd 128 or 64 with four query heads per KV head; "g8": eight (two rounds
    of query tiles at R = 5)."""
    from paper_2602_20217_gb300.configs import ModelShape
    if hd == "g8":
        return ModelShape("g8-bf16", 2, 512, 16, 2, 128, 1368, 2000, qk_norm=True, dtype="bf16",
                          rope_theta=1000000.0)
    return ModelShape(f"small-bf16-hd{hd}", 2, 512, 8, 2, hd, 1368, 2000, qk_norm=True, dtype="bf16",
                      rope_theta=500000.0)


def _check_history(m, shape, cfg, w, tol=2e-2):
    """Every history row and layer: the oracle's Attn sublayer on the GPU's
    input state and cache vs the GPU's output state.  Returns the worst error."""
    hist = m.history().astype(np.float64)
    p, _ = m.position()
    r = hist.shape[1]
    worst = 0.0
    for l in range(shape.n_layers):
        K = m.kv(l, 0, p, "k").astype(np.float64)
        V = m.kv(l, 0, p, "v").astype(np.float64)
        for i in range(r):
            pos = p - r + i
            x = hist[2 * l][i:i + 1]
            k_keep, v_keep = K[:, pos].copy(), V[:, pos].copy()
            ref = D.attn_sublayer(cfg, w["layers"][l], x, np.array([pos]), K, V) - x
            K[:, pos], V[:, pos] = k_keep, v_keep
            got = hist[2 * l + 1][i:i + 1] - x
            err = float(np.max(np.abs(got - ref)) / np.max(np.abs(ref)))
            assert err < tol, (l, pos, err)
            worst = max(worst, err)
    return worst


def _check_last_greedy_row(m, shape, cfg, w, token, next_token):
    """The last R = 1 pass (position p - 1, input ``token``): its logits vs the
    oracle's forward of that one row over the GPU's K/V of the earlier
    positions; the emitted token must be the oracle's argmax up to a near-tie."""
    from helpers import rel_err, token_ok
    p, _ = m.position()
    pos = p - 1
    x = w["embed"][[token]].astype(np.float64)
    for l in range(shape.n_layers):
        K = m.kv(l, 0, p, "k").astype(np.float64)
        V = m.kv(l, 0, p, "v").astype(np.float64)
        x = D.attn_sublayer(cfg, w["layers"][l], x, np.array([pos]), K, V)
        x = D.mlp_sublayer(cfg, w["layers"][l], x)
    ref = D.final_logits(cfg, w, x)[0]
    assert rel_err(m.logits(1)[0], ref) < 2e-2
    assert token_ok(next_token, ref, 0.05 * np.max(np.abs(ref)))


@pytest.mark.parametrize("hd", [128, 64, "g8"])
def test_attention_sublayer_at_40k_context(hd):
    from paper_2602_20217_gb300 import synth
    from paper_2602_20217_gb300.model import Model
    shape = _shape(hd)
    cfg, w = oracle_model(shape, seed=0)
    m = Model(shape, max_seq=N_PROMPT + 128, seed=0)
    m.prefill(synth.prompt_tokens(shape, N_PROMPT, seed=5))
    assert m.position()[0] == N_PROMPT
    _check_history(m, shape, cfg, w)               # the prefill's last pass: R = 16
    out = m.decode_greedy(6)                       # R = 1 passes at positions N .. N + 4
    _check_last_greedy_row(m, shape, cfg, w, int(out[-2]), int(out[-1]))
    mask = np.array([0, 1] * shape.n_layers, np.uint8)
    for gamma in (3, 4):                           # verify passes: R = 4, R = 5
        out, st, acc = m.generate(12, gamma, mask=mask)
        assert st.steps >= 1
        _check_history(m, shape, cfg, w)
    m.close()


def test_speculative_equals_greedy_at_40k_context():
    """The lossless invariant across the long-chunk regions: greedy decoding
    and speculative decoding (Attn-skipping drafts, verify with R = 5) emit
    the same tokens bit for bit."""
    from paper_2602_20217_gb300 import synth
    from paper_2602_20217_gb300.model import Model
    shape = _shape(128)
    prompt = synth.prompt_tokens(shape, N_PROMPT, seed=7)
    m = Model(shape, max_seq=N_PROMPT + 128, seed=0)
    m.prefill(prompt)
    ar = m.decode_greedy(40)
    m.rewind()
    out, st, acc = m.generate(40, 4, mask=np.array([0, 1] * shape.n_layers, np.uint8))
    assert list(out) == list(ar)
    m.close()
