"""GPU parity at full size: the Llama-3-8B-shaped decoder of the 4096-token
workload and the Qwen3-8B-shaped decoder (per-head QK-RMSNorm) of the
32768-token workload, in the launch configuration the bench times (bf16,
gamma 4, knapsack mask re-solved every step), against the oracle on sampled
outputs it can compute one by one.

* Lossless (Sec. 2.1): speculative output equals greedy output bit for bit.
* LM head (final RMSNorm + lm_head): the GPU's logits of the prefill's last
  rows (those in the history ring) on every 64th vocabulary row, from the
  GPU's final states X^(2L).
* Sublayers f^(i) of the first and last layers (Attn: RMSNorm, QKV, RoPE,
  causal GQA over the GPU's K/V cache, W_o, residual; MLP: RMSNorm, SwiGLU,
  W_down, residual) applied by the oracle to the GPU's input state of every
  history row, for the prefill's rows (R = 16) and for the rows committed by
  verify passes (R = 5).  Tolerance: 2e-2 of the sublayer's update (the
  logits tolerance).

Weights are regenerated on the host, one layer at a time, by the seeded input
generator (synth) that also fills the GPU's weights."""
import numpy as np
import pytest

from helpers import need_gpu, rel_err
from oracle import decoder as D

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    need_gpu()


def _host_layer(shape, seed, layer):
    """One layer's weights as fp64 host arrays, same values as the GPU's."""
    import torch
    from paper_2602_20217_gb300 import synth
    out = {}
    for kind, s in synth.weight_shapes(shape)["layer"].items():
        if kind in synth.NORM_KINDS:
            out[kind] = np.ones(s, np.float64)
            continue
        t = torch.empty(s, dtype=torch.bfloat16 if shape.dtype == "bf16" else torch.float32)
        synth.torch_normal_(t, synth.stream_key(seed, layer, kind), 0.02)
        out[kind] = t.double().numpy()
    return out


def _check_rows(m, cfg, lw, layer, hist, p, tol=2e-2):
    """Attn and MLP sublayers of ``layer`` on every history row."""
    r = hist.shape[1]
    K = m.kv(layer, 0, p, "k").astype(np.float64)
    V = m.kv(layer, 0, p, "v").astype(np.float64)
    worst = 0.0
    for i in range(r):
        pos = p - r + i
        x = hist[2 * layer][i:i + 1]
        kk, vv = K[:, pos].copy(), V[:, pos].copy()
        ref = D.attn_sublayer(cfg, lw, x, np.array([pos]), K, V) - x
        K[:, pos], V[:, pos] = kk, vv
        err = rel_err(hist[2 * layer + 1][i:i + 1] - x, ref)
        assert err < tol, ("attn", layer, pos, err)
        worst = max(worst, err)
    x = hist[2 * layer + 1]
    ref = D.mlp_sublayer(cfg, lw, x) - x
    err = rel_err(hist[2 * layer + 2] - x, ref)
    assert err < tol, ("mlp", layer, err)
    return max(worst, err)


@pytest.mark.parametrize("workload", ["llama8b-4k", "qwen8b-32k"])
def test_bench_configuration(workload):
    from paper_2602_20217_gb300 import knapspec as ks, synth
    from paper_2602_20217_gb300.configs import WORKLOADS
    from paper_2602_20217_gb300.model import Model
    wl = WORKLOADS[workload]
    shape = wl.shape
    cfg = D.OracleConfig.like(shape)
    prompt = synth.prompt_tokens(shape, wl.prompt_len, seed=wl.prompt_seed)
    m = Model(shape, max_seq=wl.prompt_len + 256, seed=wl.weight_seed)
    m.prefill(prompt)

    # prefill rows (R = 16): LM head on sampled vocabulary rows, first and last layer
    hist = m.history().astype(np.float64)
    p, _ = m.position()
    r = hist.shape[1]                 # the history ring keeps the pass's last r rows
    assert p == wl.prompt_len and 1 <= r <= 16
    vocab_rows = np.arange(0, shape.vocab, 64)
    lm = synth.np_weight_rows(shape, wl.weight_seed, 0, "lm_head", vocab_rows).astype(np.float64)
    h = D.rms_norm(hist[-1], np.ones(shape.d_model), cfg.rms_eps)   # final-norm gain: ones
    assert rel_err(m.logits(16)[16 - r:, vocab_rows], h @ lm.T) < 2e-2
    layers = {l: _host_layer(shape, wl.weight_seed, l) for l in (0, shape.n_layers - 1)}
    for l, lw in layers.items():
        _check_rows(m, cfg, lw, l, hist, p)

    # the bench's loop: gamma 4, knapsack re-solved every step, budget 0.8
    ar = m.decode_greedy(48)
    m.rewind()
    lat = ks.latency(0, 0.084, 3.0e-6, 0.055)   # (struct, keep-alive) as generate takes it
    out, st, acc = m.generate(48, 4, latency=lat, budget_frac=0.8, resolve_every=1)
    assert list(out) == list(ar)
    assert st.steps >= 1

    # rows committed by verify passes (R = 5)
    hist = m.history().astype(np.float64)
    p, _ = m.position()
    for l, lw in layers.items():
        _check_rows(m, cfg, lw, l, hist, p)
    m.close()
