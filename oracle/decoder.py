"""Oracle decoder: the target model f as 2L sublayers, the draft f^(S), greedy
speculative verification.  fp64 numpy.  TEST INFRASTRUCTURE ONLY.

Follows:
* Sec. 2 (Preliminaries): f = f_MLP^(L) o f_Attn^(L) o ... o f_MLP^(1) o f_Attn^(1),
  flattened to f^(2i-1) = Attn_i, f^(2i) = MLP_i; each sublayer includes its
  normalisation (footnote 1); f^(S) composes the sublayers in S in order.
* Sec. 2.1: a draft proposes gamma tokens, the target scores them in one
  parallel pass, and in greedy decoding a draft token is accepted while it
  equals the target's argmax; the target's own next token follows the
  accepted prefix (so a step yields a + 1 tokens, Eq. 1).
* Sec. 3.4 (Eq. 6 context): the history X holds the per-sublayer hidden states
  of the r tokens generated in the last m = 5 speculation steps.

Readings where the paper is silent (each listed in the design notes):
* Each sublayer is residual: f^(i)(x) = x + Sub_i(Norm_i(x)); skipping it is the
  identity on the residual stream.
* Llama/Qwen3 blocks: pre-RMSNorm, fused [Wq; Wk; Wv], optional per-head QK
  RMSNorm (Qwen3), rotate-half RoPE with inv_freq_j = theta^(-2j/hd), causal GQA
  with scale 1/sqrt(hd), output projection; MLP = W_down(silu(W_gate h) * W_up h).
* A draft step writes K/V only in the Attn sublayers it runs; verification
  rewrites positions p..p+gamma in every layer; the committed length advances
  by a + 1 and rows past it are ignored.
* Greedy argmax breaks ties towards the lowest token id.
* History: the committed rows of each verify step form one entry; the prompt's
  last ``hist_init_rows`` rows form the first entry; the last m entries are kept.
* Dynamic drafting exit (Sec. 3.5, "Dynamic Drafting Exit"): the confidence of
  a draft token is the softmax probability of its argmax over the draft's
  logits; drafting stops after the first token whose confidence is below
  tau_conf, and that token stays the step's last draft (its verification costs
  nothing extra).  The confidence is exp(l_max) / sum_i exp(l_i), computed as
  1 / sum_i exp(l_i - l_max).
"""
from __future__ import annotations

from collections import deque
from dataclasses import dataclass

import numpy as np


@dataclass(frozen=True)
class OracleConfig:
    n_layers: int
    d_model: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    d_ff: int
    vocab: int
    qk_norm: bool = False
    rms_eps: float = 1e-5
    rope_theta: float = 10000.0

    @staticmethod
    def like(shape) -> "OracleConfig":
        return OracleConfig(shape.n_layers, shape.d_model, shape.n_q_heads, shape.n_kv_heads,
                            shape.head_dim, shape.d_ff, shape.vocab, bool(shape.qk_norm),
                            float(shape.rms_eps), float(shape.rope_theta))


# ------------------------------------------------------------------ pieces
def rms_norm(x: np.ndarray, gain: np.ndarray, eps: float) -> np.ndarray:
    """RMSNorm over the last axis: x / sqrt(mean(x^2) + eps) * gain."""
    ms = np.mean(x * x, axis=-1, keepdims=True)
    return x / np.sqrt(ms + eps) * gain


def rope(x: np.ndarray, pos: np.ndarray, theta: float) -> np.ndarray:
    """Rotate-half rotary embedding of x [R, H, hd] at positions pos [R].

    Pair (j, j + hd/2) is rotated by the angle pos * theta^(-2j/hd)."""
    hd = x.shape[-1]
    half = hd // 2
    inv_freq = theta ** (-2.0 * np.arange(half, dtype=np.float64) / hd)
    ang = np.asarray(pos, dtype=np.float64)[:, None] * inv_freq[None, :]
    c = np.cos(ang)[:, None, :]
    s = np.sin(ang)[:, None, :]
    a, b = x[..., :half], x[..., half:]
    return np.concatenate([a * c - b * s, b * c + a * s], axis=-1)


def silu(z: np.ndarray) -> np.ndarray:
    return z / (1.0 + np.exp(-z))


def gqa_attention(q: np.ndarray, k_cache: np.ndarray, v_cache: np.ndarray,
                  pos: np.ndarray) -> np.ndarray:
    """Causal grouped-query attention for R query rows.

    q [R, hq, hd]; k_cache, v_cache [hk, n, hd]; row r sees keys 0..pos[r].
    Query head h uses KV head h // (hq / hk).  Returns [R, hq, hd]."""
    R, hq, hd = q.shape
    hk = k_cache.shape[0]
    group = hq // hk
    out = np.empty_like(q)
    for r in range(R):
        n = int(pos[r]) + 1
        for h in range(hq):
            keys = k_cache[h // group, :n]
            vals = v_cache[h // group, :n]
            s = keys @ q[r, h] / np.sqrt(hd)
            p = np.exp(s - s.max())
            out[r, h] = (p / p.sum()) @ vals
    return out


# --------------------------------------------------------------- sublayers
def attn_sublayer(cfg: OracleConfig, lw: dict, x: np.ndarray, pos: np.ndarray,
                  k_cache: np.ndarray, v_cache: np.ndarray) -> np.ndarray:
    """f^(2l-1): x + W_o GQA(RoPE(QKN(q)), RoPE(QKN(k)), v) with h = RMSNorm(x).

    Writes this call's K/V rows into the caches (positions ``pos``) first, so
    the rows of one call see each other causally."""
    hq, hk, hd = cfg.n_q_heads, cfg.n_kv_heads, cfg.head_dim
    R = x.shape[0]
    h = rms_norm(x, lw["attn_norm"], cfg.rms_eps)
    qkv = h @ lw["w_qkv"].T
    q = qkv[:, : hq * hd].reshape(R, hq, hd)
    k = qkv[:, hq * hd: (hq + hk) * hd].reshape(R, hk, hd)
    v = qkv[:, (hq + hk) * hd:].reshape(R, hk, hd)
    if cfg.qk_norm:
        q = rms_norm(q, lw["q_norm"], cfg.rms_eps)
        k = rms_norm(k, lw["k_norm"], cfg.rms_eps)
    q = rope(q, pos, cfg.rope_theta)
    k = rope(k, pos, cfg.rope_theta)
    for r in range(R):
        k_cache[:, pos[r]] = k[r]
        v_cache[:, pos[r]] = v[r]
    o = gqa_attention(q, k_cache, v_cache, pos)
    return x + o.reshape(R, hq * hd) @ lw["w_o"].T


def mlp_sublayer(cfg: OracleConfig, lw: dict, x: np.ndarray) -> np.ndarray:
    """f^(2l): x + W_down(silu(W_gate h) * W_up h) with h = RMSNorm(x)."""
    F = cfg.d_ff
    h = rms_norm(x, lw["mlp_norm"], cfg.rms_eps)
    gu = h @ lw["w_gate_up"].T
    return x + (silu(gu[:, :F]) * gu[:, F:]) @ lw["w_down"].T


def final_logits(cfg: OracleConfig, w: dict, x: np.ndarray) -> np.ndarray:
    """LM head on the final-normalised residual stream."""
    return rms_norm(x, w["final_norm"], cfg.rms_eps) @ w["lm_head"].T


def greedy(logits: np.ndarray) -> np.ndarray:
    """Per-row argmax; ties go to the lowest token id."""
    return np.argmax(logits, axis=-1).astype(np.int64)


def top1_prob(logits_row: np.ndarray) -> float:
    """Softmax probability of the argmax token of one row of logits (the
    draft confidence of Sec. 3.5): 1 / sum_i exp(l_i - max_j l_j)."""
    l = np.asarray(logits_row, dtype=np.float64)
    return float(1.0 / np.sum(np.exp(l - np.max(l))))


def as_f64(weights: dict) -> dict:
    """Widen a weight dict (fp32 / bf16 values held as fp32) to fp64."""
    out = {k: np.asarray(v, np.float64) for k, v in weights.items() if k != "layers"}
    out["layers"] = [{k: np.asarray(v, np.float64) for k, v in lw.items()} for lw in weights["layers"]]
    return out


# ----------------------------------------------------------------- session
class Session:
    """One sequence: KV cache, committed length p, pending token, history.

    ``pending`` is the newest known token; its K/V are not in the cache yet.
    """

    def __init__(self, cfg: OracleConfig, weights: dict, n_max: int,
                 hist_steps: int = 5, hist_init_rows: int = 8):
        self.cfg = cfg
        self.w = weights
        self.n_max = n_max
        L, hk, hd = cfg.n_layers, cfg.n_kv_heads, cfg.head_dim
        self.k = [np.zeros((hk, n_max, hd)) for _ in range(L)]
        self.v = [np.zeros((hk, n_max, hd)) for _ in range(L)]
        self.p = 0
        self.pending = None
        self.hist = deque(maxlen=hist_steps)
        self.hist_init_rows = hist_init_rows

    # f^(S) on consecutive rows starting at position pos0 (Sec. 2)
    def forward(self, tokens, pos0: int, mask=None, capture: bool = False):
        """Run the sublayers kept by ``mask`` (None = all 2L) on ``tokens`` at
        positions pos0.. ; returns (logits [R, V], states [2L+1, R, d] or None).

        states[i] is X^(i), the residual stream after sublayer i (a skipped
        sublayer leaves it unchanged); states[0] is the embedding."""
        cfg, w = self.cfg, self.w
        tokens = np.asarray(tokens, dtype=np.int64)
        pos = pos0 + np.arange(len(tokens))
        if pos[-1] >= self.n_max:
            raise ValueError("KV capacity exceeded")
        x = w["embed"][tokens].astype(np.float64)
        states = [x] if capture else None
        for i in range(1, 2 * cfg.n_layers + 1):
            if mask is None or mask[i - 1]:
                l = (i - 1) // 2
                if i % 2 == 1:
                    x = attn_sublayer(cfg, w["layers"][l], x, pos, self.k[l], self.v[l])
                else:
                    x = mlp_sublayer(cfg, w["layers"][l], x)
            if capture:
                states.append(x)
        logits = final_logits(cfg, w, x)
        return logits, (np.stack(states) if capture else None)

    def prefill(self, prompt, chunk: int = 256) -> int:
        """Run the prompt through the target; the greedy next token becomes pending."""
        prompt = np.asarray(prompt, dtype=np.int64)
        P = len(prompt)
        last = None
        for s in range(0, P, chunk):
            part = prompt[s: s + chunk]
            logits, states = self.forward(part, s, capture=True)
            last = (logits, states)
        logits, states = last
        self.p = P
        self.pending = int(greedy(logits[-1:])[0])
        r0 = min(self.hist_init_rows, states.shape[1])
        self.hist.clear()
        self.hist.append(states[:, -r0:, :])
        return self.pending

    def ar_step(self) -> int:
        """One greedy autoregressive step: commit ``pending``, return the new token."""
        logits, _ = self.forward([self.pending], self.p)
        self.p += 1
        self.pending = int(greedy(logits)[0])
        return self.pending

    def draft(self, mask, gamma: int, tau_conf: float | None = None) -> list:
        """Up to gamma greedy tokens from f^(S) starting at the pending token
        (Sec. 2.2).  With tau_conf, drafting stops after the first token whose
        top-1 probability is below tau_conf (Sec. 3.5, dynamic drafting exit).
        The confidence of every drafted token is left in ``last_confidence``."""
        tok = self.pending
        out = []
        self.last_confidence = []
        for t in range(gamma):
            logits, _ = self.forward([tok], self.p + t, mask=mask)
            tok = int(greedy(logits)[0])
            out.append(tok)
            c = top1_prob(logits[0])
            self.last_confidence.append(c)
            if tau_conf is not None and c < tau_conf:
                break
        return out

    def verify(self, drafts) -> tuple:
        """Score [pending] + drafts with the target in one pass (Sec. 2.1).

        Returns (a, new_tokens): a accepted drafts followed by the target's own
        token, a + 1 tokens in all.  Commits them and records the history."""
        rows = [self.pending] + list(drafts)
        logits, states = self.forward(rows, self.p, capture=True)
        z = greedy(logits)
        a = 0
        while a < len(drafts) and int(drafts[a]) == int(z[a]):
            a += 1
        new = [int(t) for t in drafts[:a]] + [int(z[a])]
        self.hist.append(states[:, : a + 1, :])
        self.p += a + 1
        self.pending = int(z[a])
        return a, new

    def history(self) -> np.ndarray:
        """X^(0..2L) of the rows in the history ring, stacked as [2L+1, r, d]."""
        return np.concatenate(list(self.hist), axis=1)


def greedy_generate(cfg, weights, prompt, n_new: int, n_max: int | None = None) -> list:
    """Plain greedy decoding: the first token comes from the prompt's last row."""
    n_max = n_max or (len(prompt) + n_new + 1)
    s = Session(cfg, weights, n_max)
    out = [s.prefill(prompt)]
    while len(out) < n_new:
        out.append(s.ar_step())
    return out


def spec_generate(cfg, weights, prompt, n_new: int, gamma: int, choose_mask,
                  n_max: int | None = None, resolve_every: int = 1, tau_conf: float | None = None):
    """Greedy self-speculative decoding.

    ``choose_mask(session)`` returns the draft mask; it is called before the
    first step and again every ``resolve_every`` verify steps.  ``tau_conf``
    enables the dynamic drafting exit (Sec. 3.5).  Returns (tokens, per-step
    accepted counts, masks used)."""
    n_max = n_max or (len(prompt) + n_new + gamma + 2)
    s = Session(cfg, weights, n_max)
    out = [s.prefill(prompt)]
    accepted, masks = [], []
    mask = None
    step = 0
    while len(out) < n_new:
        if step % resolve_every == 0:
            mask = choose_mask(s)
        g = min(gamma, n_max - s.p - 1)
        drafts = s.draft(mask, g, tau_conf)
        a, new = s.verify(drafts)
        out.extend(new)
        accepted.append(a)
        masks.append(np.array(mask, dtype=np.uint8))
        step += 1
    return out[:n_new], accepted, masks
