"""Pins of the plain fp32 C++ oracle (oracle/cpp/ksoracle.cpp) on the host.

It is checked against things other than itself:
* sublayers (Sec. 2): an independent fp64 torch composition of the Llama /
  Qwen3 block (F.rms_norm, F.linear, complex-number RoPE, SDPA), within fp32
  round-off; a layer with one visible key returns that key's value through
  W_o; zeroed output projections make every sublayer the identity;
* RoPE: the textbook golden values (tests/golden/rope_rotate_half.json)
  through a 1-head attention sublayer whose projections are identities;
* decoding (Sec. 2.1): the fp64 numpy oracle end to end on the tiny
  workload's model (logits within 1e-5 per row, the same greedy tokens where
  the fp64 top-2 margin is clear, the same history states); full-mask drafts
  equal the target and are all accepted; greedy speculative output is
  token-identical to greedy decoding for several masks and gammas (exact in
  fp32: every row's arithmetic is independent of the rows beside it);
* selection (Sec. 2, 3.3, 3.4, App. C): matrix-cosine identities; the App. C
  Table 3 integer weights (tests/golden/latency_table3.json); the knapsack
  against brute force over all 2^N masks and the textbook special cases."""
import json
import os

import numpy as np
import pytest
import torch

from oracle import cxx
from oracle import decoder as D
from oracle import select as S

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


@pytest.fixture(scope="module", autouse=True)
def _built():
    cxx.build()


def _shape(qk_norm=False, **kw):
    from paper_2602_20217_gb300.configs import ModelShape
    base = dict(name="cxx-test", n_layers=2, d_model=64, n_q_heads=4, n_kv_heads=2, head_dim=16, d_ff=96,
                vocab=50, qk_norm=qk_norm, dtype="f32", rope_theta=10000.0)
    base.update(kw)
    return ModelShape(**base)


def _rand_weights(shape, seed):
    from paper_2602_20217_gb300 import synth
    rng = np.random.default_rng(seed)
    shapes = synth.weight_shapes(shape)
    mk = lambda s, k: (np.ones(s) + 0.1 * rng.standard_normal(s) if k in synth.NORM_KINDS
                       else 0.2 * rng.standard_normal(s)).astype(np.float32)
    w = {k: mk(s, k) for k, s in shapes["global"].items()}
    w["layers"] = [{k: mk(s, k) for k, s in shapes["layer"].items()} for _ in range(shape.n_layers)]
    return w


def _torch_block(cfg, lw, x, pos, K, V, kind):
    """Independent fp64 torch composition of one sublayer (as in the numpy oracle's pins)."""
    import torch.nn.functional as F
    t = lambda a: torch.tensor(np.asarray(a, np.float64))
    hq, hk, hd = cfg.n_q_heads, cfg.n_kv_heads, cfg.head_dim
    X = t(x)
    if kind == "mlp":
        h = F.rms_norm(X, (cfg.d_model,), t(lw["mlp_norm"]), eps=cfg.rms_eps)
        g, u = F.linear(h, t(lw["w_gate_up"])).chunk(2, dim=-1)
        return (X + F.linear(F.silu(g) * u, t(lw["w_down"]))).numpy()
    h = F.rms_norm(X, (cfg.d_model,), t(lw["attn_norm"]), eps=cfg.rms_eps)
    q, k, v = F.linear(h, t(lw["w_qkv"])).split([hq * hd, hk * hd, hk * hd], dim=-1)
    q, k, v = q.view(-1, hq, hd), k.view(-1, hk, hd), v.view(-1, hk, hd)
    if cfg.qk_norm:
        q = F.rms_norm(q, (hd,), t(lw["q_norm"]), eps=cfg.rms_eps)
        k = F.rms_norm(k, (hd,), t(lw["k_norm"]), eps=cfg.rms_eps)

    def rope_complex(a):
        a = a.numpy()
        hh = hd // 2
        z = a[..., :hh] + 1j * a[..., hh:]
        f = np.array([cfg.rope_theta ** (-(2.0 * j) / hd) for j in range(hh)])
        z = z * np.exp(1j * np.asarray(pos, np.float64)[:, None, None] * f[None, None, :])
        return t(np.concatenate([z.real, z.imag], axis=-1))
    q, k = rope_complex(q), rope_complex(k)
    Kc, Vc = t(K).clone(), t(V).clone()
    Kc[:, pos] = k.transpose(0, 1)
    Vc[:, pos] = v.transpose(0, 1)
    n = int(pos[-1]) + 1
    mask = torch.tensor(np.arange(n)[None, :] <= np.asarray(pos)[:, None])
    o = F.scaled_dot_product_attention(q.transpose(0, 1)[None], Kc[None, :, :n], Vc[None, :, :n],
                                       attn_mask=mask, enable_gqa=True)[0].transpose(0, 1)
    return (X + F.linear(o.reshape(len(pos), hq * hd), t(lw["w_o"]))).numpy()


@pytest.mark.parametrize("qk_norm", [False, True])
def test_sublayers_vs_torch_composition(qk_norm):
    sh = _shape(qk_norm)
    w = _rand_weights(sh, 4)
    m = cxx.Model(sh, w)
    cfg = D.OracleConfig.like(sh)
    rng = np.random.default_rng(5)
    n_max, n_prev, R = 32, 9, 4
    K = rng.standard_normal((sh.n_kv_heads, n_max, sh.head_dim)).astype(np.float32)
    V = rng.standard_normal((sh.n_kv_heads, n_max, sh.head_dim)).astype(np.float32)
    x = rng.standard_normal((R, sh.d_model)).astype(np.float32)
    pos = np.arange(n_prev, n_prev + R)
    ref = _torch_block(cfg, w["layers"][0], x, pos, K, V, "attn")
    got = m.attn_sublayer(0, x, pos, K.copy(), V.copy())
    assert np.max(np.abs(got - ref)) / np.max(np.abs(ref)) < 1e-5
    ref = _torch_block(cfg, w["layers"][1], x, pos, K, V, "mlp")
    got = m.mlp_sublayer(1, x)
    assert np.max(np.abs(got - ref)) / np.max(np.abs(ref)) < 1e-5


def test_rope_golden_through_identity_attention():
    """hd = 2 * len(x) heads with identity projections: the K written to the
    cache is RoPE(x) at the row's position, checked against the golden values."""
    with open(os.path.join(GOLDEN, "rope_rotate_half.json")) as f:
        g = json.load(f)
    for c in g["cases"]:
        x = np.array(c["x"], np.float64)
        hd = len(x)
        if hd % 2 or hd < 2:
            continue
        sh = _shape(n_layers=1, d_model=hd, n_q_heads=1, n_kv_heads=1, head_dim=hd, rope_theta=g["theta"],
                    rms_eps=1e-30)
        w = _rand_weights(sh, 1)
        lw = w["layers"][0]
        lw["attn_norm"][:] = 1.0
        lw["w_qkv"][:] = np.vstack([np.eye(hd)] * 3)
        m = cxx.Model(sh, w)
        # the normalised input is x / rms(x), and RoPE is linear
        rms = np.sqrt(np.mean(x * x))
        pos = int(c["pos"])
        K = np.zeros((1, pos + 1, hd), np.float32)
        V = np.zeros((1, pos + 1, hd), np.float32)
        m.attn_sublayer(0, x[None].astype(np.float32), [pos], K, V)
        assert np.allclose(K[0, pos] * rms, c["y"], rtol=0, atol=2e-6), c


def test_single_key_attention_and_zeroed_outputs():
    sh = _shape(n_layers=1)
    w = _rand_weights(sh, 2)
    m = cxx.Model(sh, w)
    rng = np.random.default_rng(3)
    x = rng.standard_normal((1, sh.d_model)).astype(np.float32)
    K = np.zeros((sh.n_kv_heads, 4, sh.head_dim), np.float32)
    V = np.zeros_like(K)
    y = m.attn_sublayer(0, x, [0], K, V)           # one visible key: its own value
    lw = w["layers"][0]
    h = D.rms_norm(x.astype(np.float64), lw["attn_norm"], sh.rms_eps)
    qkv = h @ lw["w_qkv"].T
    hq, hk, hd = sh.n_q_heads, sh.n_kv_heads, sh.head_dim
    v = qkv[0, (hq + hk) * hd:].reshape(hk, hd)
    o = np.concatenate([v[j // (hq // hk)] for j in range(hq)])
    assert np.allclose(y, x + o @ lw["w_o"].T, rtol=1e-5, atol=1e-5)
    for lw in w["layers"]:
        lw["w_o"][:] = 0.0
        lw["w_down"][:] = 0.0
    m = cxx.Model(sh, w)
    assert np.array_equal(m.attn_sublayer(0, x, [0], K, V), x)
    assert np.array_equal(m.mlp_sublayer(0, x), x)


def test_tiny_workload_against_the_numpy_oracle():
    from paper_2602_20217_gb300 import synth
    from paper_2602_20217_gb300.configs import TINY
    w32 = synth.np_model_weights(TINY, 0)
    prompt = synth.prompt_tokens(TINY, 256, seed=1)
    s = cxx.Session(cxx.Model(TINY, w32), 512)
    so = D.Session(D.OracleConfig.like(TINY), D.as_f64(w32), 512)
    assert s.prefill(prompt) == so.prefill(prompt)
    assert np.allclose(s.history(), so.history(), rtol=0, atol=1e-5)
    mask = np.array([0, 1, 1, 1, 0, 1, 1, 1], np.uint8)
    for _ in range(4):
        d, do = s.draft(mask, 4), so.draft(mask, 4)
        assert d == do
        (a, new), (ao, newo) = s.verify(d), so.verify(do)
        assert (a, new) == (ao, newo)
    p, pend = s.position()
    lg, st = s.forward([pend, 5, 6], p, capture=True)
    lo, sto = so.forward([pend, 5, 6], p, capture=True)
    err = np.max(np.abs(lg - lo), axis=1) / np.max(np.abs(lo), axis=1)
    assert np.max(err) < 1e-5
    assert np.allclose(st, sto, rtol=0, atol=1e-5)
    assert np.allclose(s.history(), so.history(), rtol=0, atol=1e-5)


def _spec(session, mask, gamma, n_new):
    out = [session.position()[1]]
    while len(out) < n_new:
        a, new = session.verify(session.draft(mask, gamma))
        out.extend(new)
    return out[:n_new]


def test_full_mask_drafts_and_lossless_decoding():
    from paper_2602_20217_gb300 import synth
    from paper_2602_20217_gb300.configs import TINY
    w32 = synth.np_model_weights(TINY, 0)
    m = cxx.Model(TINY, w32)
    prompt = synth.prompt_tokens(TINY, 48, seed=1)
    g = cxx.Session(m, 256)
    ar = [g.prefill(prompt)] + [g.ar_step() for _ in range(39)]
    full = np.ones(TINY.n_sublayers, np.uint8)
    s = cxx.Session(m, 256)
    s.prefill(prompt)
    a, new = s.verify(s.draft(full, 5))
    assert a == 5 and new == ar[1:7]
    rng = np.random.default_rng(0)
    for mask, gamma in [(np.zeros(8, np.uint8), 3), (full, 4), (rng.integers(0, 2, 8).astype(np.uint8), 2),
                        (np.array([0, 1] * 4, np.uint8), 6)]:
        s = cxx.Session(m, 256)
        s.prefill(prompt)
        assert _spec(s, mask, gamma, 40) == ar, (mask, gamma)


def test_matrix_cosine_identities():
    rng = np.random.default_rng(8)
    X = rng.standard_normal((7, 33)).astype(np.float32)
    assert cxx.matrix_cos(X, X) == pytest.approx(1.0, abs=1e-6)
    assert cxx.matrix_cos(X, -X) == pytest.approx(-1.0, abs=1e-6)
    assert cxx.matrix_cos(X, 3.0 * X) == pytest.approx(1.0, abs=1e-6)
    Y = rng.standard_normal((7, 33)).astype(np.float32)
    ref = float(np.sum(X.astype(np.float64) * Y) / (np.linalg.norm(X.astype(np.float64)) * np.linalg.norm(Y)))
    assert cxx.matrix_cos(X, Y) == pytest.approx(ref, abs=1e-5)


def test_integer_weights_table3_golden():
    with open(os.path.join(GOLDEN, "latency_table3.json")) as f:
        g = json.load(f)
    for c in g["cases"]:
        ta = c["c2"] * c["n"] + c["c3"]
        assert cxx.integer_weights(ta, c["c1"]) == (c["w_attn"], c["w_mlp"]), c


def test_knapsack_against_brute_force_and_special_cases():
    rng = np.random.default_rng(9)
    for trial in range(40):
        n = int(rng.integers(2, 15))
        w = rng.integers(1, 6, n)
        q = rng.integers(0, 1 << 30, n)
        if trial % 5 == 0:
            q[: n // 2] = q[0]          # ties
        B = int(rng.integers(0, w.sum() + 2))
        m, v = cxx.knapsack(w, q, B)
        mb, vb = cxx.knapsack(w, q, B, brute=True)
        assert v == vb and np.array_equal(m, mb)
        assert int(np.sum(w[m == 1])) <= B and int(np.sum(q[m == 1])) == v
        mo, vo = S.knapsack(w, q, B)
        assert v == vo and np.array_equal(m, mo)
    q = np.array([5, 9, 1, 7, 3], np.int64)
    m, _ = cxx.knapsack(np.ones(5), q, 2)          # all weights 1: the top-B values
    assert list(m) == [0, 1, 0, 1, 0]
    m, _ = cxx.knapsack([2, 3, 1, 4, 2], q, 100)   # budget above the weight sum: everything
    assert list(m) == [1] * 5
    m, v = cxx.knapsack([2, 3, 1, 4, 2], q, 0)     # no budget: nothing
    assert list(m) == [0] * 5 and v == 0
