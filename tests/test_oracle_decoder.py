"""Pins for the decoder oracle (CPU).

What pins what (none re-types the oracle's formulas):
* RMSNorm: hand values and unit RMS; torch.nn.functional.rms_norm.
* RoPE: textbook cos/sin values (tests/golden/rope_rotate_half.json), identity
  at position 0, norm preservation, relative-position property, and an
  independent complex-number formulation.
* silu: silu(x) - silu(-x) = x, silu(0) = 0; torch.nn.functional.silu.
* GQA attention: torch scaled_dot_product_attention (causal, enable_gqa);
  one visible key returns its value; equal scores return the mean value.
* Attn / MLP sublayers: an independent torch composition (F.linear, F.rms_norm,
  SDPA, complex RoPE) of the Llama / Qwen3 block.
* Residual structure (Sec. 2 footnote, reading R1): with W_o = W_down = 0 every
  mask gives lm_head . RMSNorm(embed[token]).
* Causality: prefill in chunks == prefill at once == one token at a time.
* Full mask (S = [2L]) drafts are the target's greedy tokens and verification
  accepts all of them (Sec. 2.2).
* Lossless greedy SD (Sec. 2.1): speculative output == greedy output for empty,
  random, adversarial and full masks.
"""
import json
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle import decoder as D

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def tiny_cfg(qk_norm=False, L=2, hq=4, hk=2, hd=16, d=48, ff=40, V=97):
    return D.OracleConfig(L, d, hq, hk, hd, ff, V, qk_norm, 1e-5, 10000.0)


def rand_weights(cfg, seed=0, std=0.2):
    rng = np.random.default_rng(seed)
    hd = cfg.head_dim
    nq = (cfg.n_q_heads + 2 * cfg.n_kv_heads) * hd

    def lw():
        w = {
            "attn_norm": rng.uniform(0.5, 1.5, cfg.d_model),
            "w_qkv": rng.standard_normal((nq, cfg.d_model)) * std,
            "w_o": rng.standard_normal((cfg.d_model, cfg.n_q_heads * hd)) * std,
            "mlp_norm": rng.uniform(0.5, 1.5, cfg.d_model),
            "w_gate_up": rng.standard_normal((2 * cfg.d_ff, cfg.d_model)) * std,
            "w_down": rng.standard_normal((cfg.d_model, cfg.d_ff)) * std,
        }
        if cfg.qk_norm:
            w["q_norm"] = rng.uniform(0.5, 1.5, hd)
            w["k_norm"] = rng.uniform(0.5, 1.5, hd)
        return w

    return {
        "layers": [lw() for _ in range(cfg.n_layers)],
        "embed": rng.standard_normal((cfg.vocab, cfg.d_model)),
        "lm_head": rng.standard_normal((cfg.vocab, cfg.d_model)) * std,
        "final_norm": rng.uniform(0.5, 1.5, cfg.d_model),
    }


# ------------------------------------------------------------------ pieces
def test_rms_norm_hand_and_torch():
    y = D.rms_norm(np.array([[3.0, 4.0]]), np.ones(2), 0.0)
    assert np.allclose(y, [[3 / np.sqrt(12.5), 4 / np.sqrt(12.5)]], rtol=0, atol=1e-15)
    rng = np.random.default_rng(0)
    x = rng.standard_normal((5, 32))
    g = rng.uniform(0.5, 2, 32)
    ref = F.rms_norm(torch.tensor(x), (32,), torch.tensor(g), eps=1e-5).numpy()
    assert np.allclose(D.rms_norm(x, g, 1e-5), ref, rtol=1e-12, atol=1e-13)
    assert np.allclose(np.sqrt(np.mean(D.rms_norm(x, np.ones(32), 0.0) ** 2, axis=1)), 1.0)


def test_rope_golden_values():
    with open(os.path.join(GOLDEN, "rope_rotate_half.json")) as f:
        g = json.load(f)
    for c in g["cases"]:
        y = D.rope(np.array(c["x"], np.float64)[None, None, :], np.array([c["pos"]]), g["theta"])
        assert np.allclose(y[0, 0], c["y"], rtol=0, atol=1e-15), c


def _rope_complex(x, pos, theta):
    """Independent formulation: z_j = x_j + i x_{j+h} times exp(i pos theta^(-2j/hd))."""
    hd = x.shape[-1]
    h = hd // 2
    z = x[..., :h] + 1j * x[..., h:]
    freqs = np.array([theta ** (-(2.0 * j) / hd) for j in range(h)])
    rot = np.exp(1j * np.outer(pos, freqs))[:, None, :]
    w = z * rot
    return np.concatenate([w.real, w.imag], axis=-1)


def test_rope_properties():
    rng = np.random.default_rng(1)
    x = rng.standard_normal((6, 3, 16))
    pos = np.array([0, 1, 7, 100, 4095, 131071])
    y = D.rope(x, pos, 500000.0)
    assert np.allclose(y, _rope_complex(x, pos, 500000.0), rtol=0, atol=1e-12)
    assert np.allclose(y[0], x[0], atol=0)                         # identity at 0
    assert np.allclose(np.linalg.norm(y, axis=-1), np.linalg.norm(x, axis=-1))
    # <R(p) q, R(p') k> depends only on p - p'
    q, k = rng.standard_normal((2, 1, 1, 16))
    a = (D.rope(q, np.array([10]), 1e4) * D.rope(k, np.array([3]), 1e4)).sum()
    b = (D.rope(q, np.array([1007]), 1e4) * D.rope(k, np.array([1000]), 1e4)).sum()
    assert a == pytest.approx(b, rel=1e-10)


def test_silu_identities():
    x = np.linspace(-20, 20, 101)
    assert np.allclose(D.silu(x) - D.silu(-x), x, atol=1e-12)
    assert D.silu(np.array([0.0]))[0] == 0.0
    assert np.allclose(D.silu(x), F.silu(torch.tensor(x)).numpy(), rtol=1e-13, atol=1e-15)


def test_gqa_attention_vs_sdpa():
    rng = np.random.default_rng(2)
    hq, hk, hd, n = 8, 2, 16, 23
    K = rng.standard_normal((hk, n, hd))
    V = rng.standard_normal((hk, n, hd))
    R = 5
    pos = np.arange(n - R, n)
    q = rng.standard_normal((R, hq, hd))
    got = D.gqa_attention(q, K, V, pos)
    # SDPA with a boolean mask: query r sees keys 0..pos[r]
    mask = torch.tensor(np.arange(n)[None, :] <= pos[:, None])
    ref = F.scaled_dot_product_attention(
        torch.tensor(q).transpose(0, 1)[None], torch.tensor(K)[None], torch.tensor(V)[None],
        attn_mask=mask, enable_gqa=True)[0].transpose(0, 1).numpy()
    assert np.allclose(got, ref, rtol=1e-11, atol=1e-12)


def test_attention_special_cases():
    rng = np.random.default_rng(3)
    K = rng.standard_normal((1, 4, 8))
    V = rng.standard_normal((1, 4, 8))
    q = rng.standard_normal((1, 2, 8))
    out = D.gqa_attention(q, K, V, np.array([0]))                  # one visible key
    assert np.allclose(out[0, 0], V[0, 0]) and np.allclose(out[0, 1], V[0, 0])
    out = D.gqa_attention(np.zeros((1, 1, 8)), K, V, np.array([3]))  # equal scores
    assert np.allclose(out[0, 0], V[0].mean(0))


# ----------------------------------------------------------------- sublayers
def _torch_block(cfg, lw, x, pos, K, V, kind):
    """Independent torch composition of one Llama/Qwen3 sublayer (fp64)."""
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
    q = t(_rope_complex(q.numpy(), pos, cfg.rope_theta))
    k = t(_rope_complex(k.numpy(), pos, cfg.rope_theta))
    Kc, Vc = t(K).clone(), t(V).clone()
    Kc[:, pos] = k.transpose(0, 1)
    Vc[:, pos] = v.transpose(0, 1)
    n = int(pos[-1]) + 1
    mask = torch.tensor(np.arange(n)[None, :] <= pos[:, None])
    o = F.scaled_dot_product_attention(q.transpose(0, 1)[None], Kc[None, :, :n], Vc[None, :, :n],
                                       attn_mask=mask, enable_gqa=True)[0].transpose(0, 1)
    return (X + F.linear(o.reshape(len(pos), hq * hd), t(lw["w_o"]))).numpy()


@pytest.mark.parametrize("qk_norm", [False, True])
def test_sublayers_vs_torch_composition(qk_norm):
    cfg = tiny_cfg(qk_norm=qk_norm)
    w = rand_weights(cfg, seed=4)
    rng = np.random.default_rng(5)
    n_prev, R = 9, 4
    K = rng.standard_normal((cfg.n_kv_heads, 32, cfg.head_dim))
    V = rng.standard_normal((cfg.n_kv_heads, 32, cfg.head_dim))
    x = rng.standard_normal((R, cfg.d_model))
    pos = np.arange(n_prev, n_prev + R)
    ref = _torch_block(cfg, w["layers"][0], x, pos, K, V, "attn")
    got = D.attn_sublayer(cfg, w["layers"][0], x, pos, K.copy(), V.copy())
    assert np.allclose(got, ref, rtol=1e-10, atol=1e-11)
    ref = _torch_block(cfg, w["layers"][1], x, pos, K, V, "mlp")
    assert np.allclose(D.mlp_sublayer(cfg, w["layers"][1], x), ref, rtol=1e-12, atol=1e-12)


def test_residual_structure_zero_outputs():
    cfg = tiny_cfg()
    w = rand_weights(cfg, seed=6)
    for lw in w["layers"]:
        lw["w_o"][:] = 0.0
        lw["w_down"][:] = 0.0
    toks = [3, 14, 15, 92]
    expect = D.rms_norm(w["embed"][toks], w["final_norm"], cfg.rms_eps) @ w["lm_head"].T
    rng = np.random.default_rng(7)
    for mask in [None, np.zeros(4, np.uint8), rng.integers(0, 2, 4)]:
        s = D.Session(cfg, w, 16)
        logits, _ = s.forward(toks, 0, mask=mask)
        assert np.allclose(logits, expect, rtol=1e-12, atol=1e-12)


# ------------------------------------------------------------- generation
def test_prefill_chunking_and_token_by_token_agree():
    cfg = tiny_cfg(qk_norm=True)
    w = rand_weights(cfg, seed=8)
    toks = np.random.default_rng(9).integers(0, cfg.vocab, 21)
    a = D.Session(cfg, w, 32)
    la, _ = a.forward(toks, 0)
    b = D.Session(cfg, w, 32)
    lb = np.concatenate([b.forward(toks[s:s + 5], s)[0] for s in range(0, 21, 5)])
    c = D.Session(cfg, w, 32)
    lc = np.concatenate([c.forward([t], i)[0] for i, t in enumerate(toks)])
    assert np.allclose(la, lb, rtol=1e-11, atol=1e-12) and np.allclose(la, lc, rtol=1e-11, atol=1e-12)
    for l in range(cfg.n_layers):
        assert np.allclose(a.k[l][:, :21], c.k[l][:, :21], atol=1e-12)


def test_full_mask_draft_is_target_and_is_fully_accepted():
    cfg = tiny_cfg()
    w = rand_weights(cfg, seed=10)
    prompt = np.random.default_rng(11).integers(0, cfg.vocab, 12)
    ar = D.greedy_generate(cfg, w, prompt, 9)
    s = D.Session(cfg, w, 64)
    s.prefill(prompt)
    drafts = s.draft(np.ones(2 * cfg.n_layers, np.uint8), 4)
    assert drafts == ar[1:5]
    a, new = s.verify(drafts)
    assert a == 4 and new == ar[1:6]
    assert s.p == 12 + 5 and s.pending == ar[5]


def test_adversarial_drafts_rejected_and_bonus_is_ar_token():
    cfg = tiny_cfg()
    w = rand_weights(cfg, seed=12)
    prompt = np.random.default_rng(13).integers(0, cfg.vocab, 10)
    ar = D.greedy_generate(cfg, w, prompt, 6)
    s = D.Session(cfg, w, 64)
    s.prefill(prompt)
    wrong = [(ar[1] + 1) % cfg.vocab, ar[2], ar[3]]
    a, new = s.verify(wrong)
    assert a == 0 and new == [ar[1]]
    a, new = s.verify([ar[2], ar[3], (ar[4] + 5) % cfg.vocab])
    assert a == 2 and new == ar[2:5]


@pytest.mark.parametrize("mask_kind", ["empty", "random", "attn_only", "full"])
def test_lossless_greedy_speculative_decoding(mask_kind):
    cfg = tiny_cfg(qk_norm=True, L=3)
    w = rand_weights(cfg, seed=14)
    prompt = np.random.default_rng(15).integers(0, cfg.vocab, 16)
    n = 2 * cfg.n_layers
    masks = {"empty": np.zeros(n, np.uint8), "full": np.ones(n, np.uint8),
             "attn_only": np.array([1, 0] * cfg.n_layers, np.uint8),
             "random": np.random.default_rng(16).integers(0, 2, n).astype(np.uint8)}
    ar = D.greedy_generate(cfg, w, prompt, 24)
    for gamma in (1, 3, 5):
        toks, acc, _ = D.spec_generate(cfg, w, prompt, 24, gamma, lambda s: masks[mask_kind])
        assert toks == ar
        if mask_kind == "full":
            assert all(a == gamma for a in acc[:-1])


def test_history_ring_holds_committed_rows():
    cfg = tiny_cfg()
    w = rand_weights(cfg, seed=17)
    prompt = np.random.default_rng(18).integers(0, cfg.vocab, 12)
    s = D.Session(cfg, w, 128, hist_steps=3, hist_init_rows=4)
    s.prefill(prompt)
    assert s.history().shape == (2 * cfg.n_layers + 1, 4, cfg.d_model)
    rows = []
    for _ in range(5):
        before = s.pending
        drafts = s.draft(np.ones(2 * cfg.n_layers, np.uint8), 2)
        a, _ = s.verify(drafts)
        rows.append(a + 1)
    assert s.history().shape[1] == sum(rows[-3:])
    # X^(0) of the newest entry = embeddings of that step's committed tokens
    committed = [before] + drafts[:a]
    assert np.array_equal(s.history()[0, -(a + 1):], w["embed"][committed])


def test_top1_prob_closed_forms():
    # Sec. 3.5 confidence = softmax probability of the argmax token
    assert abs(D.top1_prob(np.full(1000, 3.7)) - 1e-3) < 1e-15          # uniform: 1 / V
    assert abs(D.top1_prob(np.array([np.log(3.0), 0.0])) - 0.75) < 1e-15  # 3 / (3 + 1)
    assert D.top1_prob(np.array([5.0, 5.0, -800.0, -800.0])) == 0.5      # two tied maxima
    assert D.top1_prob(np.array([0.0, 0.0, 0.0, 800.0])) == 1.0           # one dominant logit
    l = np.random.default_rng(0).normal(size=257)
    p = D.top1_prob(l)
    assert abs(D.top1_prob(l + 1234.5) - p) < 1e-12                      # shift invariance
    l2 = l.copy()
    l2[np.argmax(l)] += 0.5
    assert D.top1_prob(l2) > p                                            # a larger max is more confident
    # brute force in exact rationals: logits log(k) give probabilities k / sum(k)
    ks = np.arange(1, 9, dtype=np.float64)
    assert abs(D.top1_prob(np.log(ks)) - 8.0 / 36.0) < 1e-15


def test_dynamic_exit_stops_after_first_unconfident_token():
    cfg = tiny_cfg(L=3)
    w = rand_weights(cfg, seed=21, std=0.6)
    prompt = np.random.default_rng(22).integers(0, cfg.vocab, 14)
    mask = np.array([1, 0, 1, 1, 0, 1], np.uint8)
    s = D.Session(cfg, w, 64)
    s.prefill(prompt)
    full = s.draft(mask, 6)                       # no exit: gamma tokens
    conf = list(s.last_confidence)
    assert len(full) == 6 and len(conf) == 6
    # the recorded confidence is top1_prob of the draft's own logits
    s2 = D.Session(cfg, w, 64)
    s2.prefill(prompt)
    logits, _ = s2.forward([s2.pending], s2.p, mask=mask)
    assert abs(conf[0] - D.top1_prob(logits[0])) < 1e-15
    for tau in (0.0, 1.01, *sorted(conf)):
        s3 = D.Session(cfg, w, 64)
        s3.prefill(prompt)
        got = s3.draft(mask, 6, tau)
        below = [i for i, c in enumerate(conf) if c < tau]
        n = below[0] + 1 if below else 6          # the unconfident token is kept, then drafting stops
        assert got == full[:n], (tau, got, full)


@pytest.mark.parametrize("tau", [0.0, 0.2, 0.5, 1.01])
def test_lossless_with_dynamic_exit(tau):
    cfg = tiny_cfg(qk_norm=True, L=3)
    w = rand_weights(cfg, seed=23, std=0.6)
    prompt = np.random.default_rng(24).integers(0, cfg.vocab, 16)
    mask = np.array([0, 1, 1, 1, 0, 1], np.uint8)
    ar = D.greedy_generate(cfg, w, prompt, 24)
    toks, acc, _ = D.spec_generate(cfg, w, prompt, 24, 5, lambda s: mask, tau_conf=tau)
    assert toks == ar
    if tau > 1.0:
        assert all(a <= 1 for a in acc)           # one draft per step
