"""GPU parity at full size for every bf16 workload: the Llama-3-8B shape at
4096 and 131072 tokens of context, the Qwen3-8B shape (per-head QK-RMSNorm)
at 32768 and the Qwen3-32B shape (d 5120, d_ff 25600, vocabulary 151936,
8 query heads per KV head, 64 layers) at 65536, in the launch configuration
the bench times (bf16, gamma 4, knapsack mask re-solved every step), against
the oracle on sampled outputs it can compute one by one.

* Lossless (Sec. 2.1): speculative output equals greedy output bit for bit.
* LM head (final RMSNorm + lm_head) over the FULL vocabulary for the last
  four prefill rows and for the rows committed by the last verify pass, from
  the GPU's final states X^(2L): logits within 2e-2 per row, and the GPU's
  greedy token is the oracle's argmax or within that tolerance of it.
* Sublayers f^(i) of the first, a middle and the last layer (Attn: RMSNorm,
  QKV, QK-norm, RoPE, causal GQA over the GPU's K/V cache, W_o, residual;
  MLP: RMSNorm, SwiGLU, W_down, residual) applied by the oracle to the GPU's
  input state of every history row, for the prefill's rows (R = 16) and for
  the rows committed by verify passes (R = 5).  Tolerance: 2e-2 of the
  sublayer's update, per row (the logits tolerance).

Weights are regenerated on the host by the seeded input generator (synth)
that also fills the GPU's weights: one layer at a time, and the LM head in
row blocks."""
import numpy as np
import pytest

from helpers import need_gpu, rel_err, token_within_tolerance
from oracle import decoder as D

pytestmark = pytest.mark.gpu

TOL = 2e-2


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


def _oracle_logits(shape, seed, eps, final_states, block=16384):
    """Full-vocabulary logits of the final RMSNorm (gain 1) + LM head, fp64 on
    the host, with the LM head regenerated in blocks of rows."""
    import torch
    from paper_2602_20217_gb300 import synth
    h = D.rms_norm(np.asarray(final_states, np.float64), np.ones(shape.d_model), eps)
    key = synth.stream_key(seed, synth.GLOBAL_LAYER, "lm_head")
    out = np.empty((h.shape[0], shape.vocab), np.float64)
    dt = torch.bfloat16 if shape.dtype == "bf16" else torch.float32
    for r0 in range(0, shape.vocab, block):
        n = min(block, shape.vocab - r0)
        t = torch.empty((n, shape.d_model), dtype=dt)
        synth.torch_normal_(t, key, 0.02, start=r0 * shape.d_model)
        out[:, r0:r0 + n] = h @ t.double().numpy().T
    return out


def _check_lm_head(shape, seed, eps, gpu_logits, final_states, gpu_tokens):
    ref = _oracle_logits(shape, seed, eps, final_states)
    err = rel_err(gpu_logits, ref)
    assert err < TOL, ("lm head", err)
    for row, tok in zip(ref, gpu_tokens):
        assert token_within_tolerance(tok, row, TOL), (int(tok), int(np.argmax(row)))
    return err


def _check_rows(m, cfg, lw, layer, hist, p):
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
        assert err < TOL, ("attn", layer, pos, err)
        worst = max(worst, err)
    x = hist[2 * layer + 1]
    ref = D.mlp_sublayer(cfg, lw, x) - x
    err = rel_err(hist[2 * layer + 2] - x, ref)
    assert err < TOL, ("mlp", layer, err)
    return max(worst, err)


@pytest.mark.parametrize("workload", ["llama8b-4k", "qwen8b-32k", "llama8b-128k", "qwen32b-64k"])
def test_bench_configuration(workload):
    from paper_2602_20217_gb300 import knapspec as ks, synth
    from paper_2602_20217_gb300.configs import WORKLOADS
    from paper_2602_20217_gb300.model import Model
    wl = WORKLOADS[workload]
    shape = wl.shape
    cfg = D.OracleConfig.like(shape)
    prompt = synth.prompt_tokens(shape, wl.prompt_len, seed=wl.prompt_seed)
    m = Model(shape, max_seq=wl.prompt_len + 256, seed=wl.weight_seed)
    pending = m.prefill(prompt)

    # prefill rows (R = 16): the LM head over the full vocabulary on the
    # last four rows (the last row's greedy token is the pending token)
    hist = m.history().astype(np.float64)
    p, _ = m.position()
    r = hist.shape[1]                 # the history ring keeps the pass's last r rows
    assert p == wl.prompt_len and 4 <= r <= 16
    lg = m.logits(16)[-4:]
    toks = list(np.argmax(lg[:-1], axis=1)) + [pending]
    assert int(np.argmax(lg[-1])) == pending
    _check_lm_head(shape, wl.weight_seed, cfg.rms_eps, lg, hist[-1][-4:], toks)

    layers = {l: _host_layer(shape, wl.weight_seed, l) for l in (0, shape.n_layers // 2, shape.n_layers - 1)}
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
    # the last verify pass: its committed rows a + 1 are the newest history
    # rows; their greedy tokens are the argmaxes of the pass's logits
    a_last = int(acc[int(st.steps) - 1])
    n = min(4, a_last + 1)
    lg = m.logits(5)[a_last + 1 - n:a_last + 1]
    _check_lm_head(shape, wl.weight_seed, cfg.rms_eps, lg, hist[-1][-n:],
                   list(np.argmax(lg, axis=1)))
    m.close()
