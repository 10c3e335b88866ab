"""Oracle of sampling-mode speculative decoding.  Plain Python / fp64 numpy.
TEST INFRASTRUCTURE ONLY.

Follows:
* Sec. 2.1: in sampling, a draft token s~ proposed by the draft model q is
  accepted when u <= min(1, p(s~) / q(s~)) for u ~ U(0, 1), p being the
  target model's distribution at the same position.  At the first rejection
  the standard speculative-sampling rule of the works Sec. 2.1 cites replaces
  the token by a sample of norm(max(0, p - q)); when every draft is accepted
  the target's distribution after the last draft gives one more token.  The
  output tokens are then distributed exactly as samples of p.
* Sec. 4 (sampling experiments): nucleus sampling with temperature T = 0.7,
  top-k = 50 and top-p = 0.95.

Readings where the paper is silent (listed in the design notes):
* Filtering order: logits / T, then the k largest (ties: lower token id
  first), then softmax over those k, then the shortest prefix of them in
  descending probability (ties: lower id first) whose cumulative probability
  reaches top_p (at least one token), renormalised.  Draft and target
  distributions are filtered the same way.
* A sample with uniform u takes the first token of that ordered support whose
  cumulative probability exceeds u (cumulative sums in the support's order).
  The residual distribution norm(max(0, p - q)) is sampled the same way, over
  p's support in p's order; if it has no mass (p <= q everywhere) the token is
  drawn from p.
* Random numbers: Philox4x64 with 10 rounds (Salmon et al., SC 2011), key
  (seed, 0), counter (step, row, purpose, 0) with purpose 0 = the draft sample
  of row t, 1 = the acceptance test of draft t, 2 = the residual or bonus
  sample of the step.  u = (top 24 bits of the first output word) / 2^24, a
  float that both sides represent exactly.
"""
from __future__ import annotations

import numpy as np

MASK64 = (1 << 64) - 1
PHILOX_M0 = 0xD2E7470EE14C6C93
PHILOX_M1 = 0xCA5A826395121157
PHILOX_W0 = 0x9E3779B97F4A7C15
PHILOX_W1 = 0xBB67AE8584CAA73B


def _mulhilo(a: int, b: int):
    p = a * b
    return (p >> 64) & MASK64, p & MASK64


def philox4x64_10(counter, key):
    """Philox4x64-10 block function: four 64-bit counter words and two 64-bit
    key words to four 64-bit outputs (Python integers)."""
    x0, x1, x2, x3 = (int(c) & MASK64 for c in counter)
    k0, k1 = (int(k) & MASK64 for k in key)
    for r in range(10):
        if r:
            k0 = (k0 + PHILOX_W0) & MASK64
            k1 = (k1 + PHILOX_W1) & MASK64
        hi0, lo0 = _mulhilo(PHILOX_M0, x0)
        hi1, lo1 = _mulhilo(PHILOX_M1, x2)
        x0, x1, x2, x3 = hi1 ^ x1 ^ k0, lo1, hi0 ^ x3 ^ k1, lo0
    return x0, x1, x2, x3


def uniform(seed: int, step: int, row: int, purpose: int) -> float:
    """The uniform number of (step, row, purpose): the top 24 bits of the first
    Philox output word over 2^24, in [0, 1)."""
    x0 = philox4x64_10((step, row, purpose, 0), (seed, 0))[0]
    return (x0 >> 40) / float(1 << 24)


def filter_distribution(logits_row, temperature: float, top_k: int, top_p: float):
    """Temperature, top-k and top-p (nucleus) filtering of one row of logits.
    Returns (ids, probs): the kept tokens in descending probability (ties:
    lower id first) and their renormalised probabilities (fp64)."""
    l = np.asarray(logits_row, dtype=np.float64) / float(temperature)
    order = sorted(range(len(l)), key=lambda i: (-l[i], i))   # descending, ties by id
    ids = order[: min(int(top_k), len(l))]
    z = np.array([l[i] for i in ids])
    pr = np.exp(z - z.max())
    pr /= pr.sum()
    keep, c = 0, 0.0
    for j in range(len(ids)):
        c += pr[j]
        keep = j + 1
        if c >= top_p:
            break
    ids = np.array(ids[:keep], dtype=np.int64)
    pr = pr[:keep] / pr[:keep].sum()
    return ids, pr


def sample(ids, probs, u: float) -> int:
    """Inverse-CDF sample over an ordered support: the first token whose
    cumulative probability exceeds u (the last one if rounding leaves u above
    the total)."""
    c = 0.0
    for t, p in zip(ids, probs):
        c += p
        if u < c:
            return int(t)
    return int(ids[-1])


def prob_of(ids, probs, token: int) -> float:
    """Probability of ``token`` under an ordered support (0 outside it)."""
    for t, p in zip(ids, probs):
        if int(t) == int(token):
            return float(p)
    return 0.0


def residual(p_ids, p_probs, q_ids, q_probs):
    """norm(max(0, p - q)) over p's support in p's order; None when p <= q
    everywhere."""
    r = np.array([max(0.0, p - prob_of(q_ids, q_probs, t)) for t, p in zip(p_ids, p_probs)])
    s = r.sum()
    if s <= 0.0:
        return None
    return np.asarray(p_ids), r / s


def verify_one(p_dist, q_dist, x: int, u_accept: float, u_resample: float):
    """Sec. 2.1 test of one draft token x sampled from q: accepted when
    u_accept <= min(1, p(x) / q(x)); otherwise the replacement is sampled from
    norm(max(0, p - q)) with u_resample.  Returns (accepted, replacement)."""
    p_ids, p_pr = p_dist
    q_ids, q_pr = q_dist
    px, qx = prob_of(p_ids, p_pr, x), prob_of(q_ids, q_pr, x)
    if qx > 0.0 and u_accept <= min(1.0, px / qx):
        return True, None
    res = residual(p_ids, p_pr, q_ids, q_pr)
    ids, pr = res if res is not None else (p_ids, p_pr)
    return False, sample(ids, pr, u_resample)


def speculative_step(p_dists, q_dists, drafts, seed: int, step: int):
    """One sampling-mode verification (Sec. 2.1).  p_dists: gamma + 1 target
    distributions (ids, probs) for rows 0..gamma; q_dists: the gamma draft
    distributions the drafts were sampled from.  Returns (a, new tokens)."""
    gamma = len(drafts)
    u_last = uniform(seed, step, 0, 2)
    for t in range(gamma):
        ok, rep = verify_one(p_dists[t], q_dists[t], int(drafts[t]), uniform(seed, step, t, 1), u_last)
        if not ok:
            return t, [int(d) for d in drafts[:t]] + [rep]
    p_ids, p_pr = p_dists[gamma]
    return gamma, [int(d) for d in drafts] + [sample(p_ids, p_pr, u_last)]


def draft_sample(session, mask, gamma: int, seed: int, step: int, temperature: float, top_k: int, top_p: float):
    """gamma draft tokens of f^(S) (Sec. 2.2), each sampled from its filtered
    distribution with the uniform of (step, t, 0).  Returns (drafts, q_dists)."""
    tok = session.pending
    drafts, q = [], []
    for t in range(gamma):
        logits, _ = session.forward([tok], session.p + t, mask=mask)
        dist = filter_distribution(logits[0], temperature, top_k, top_p)
        tok = sample(dist[0], dist[1], uniform(seed, step, t, 0))
        drafts.append(tok)
        q.append(dist)
    return drafts, q


def verify_sample(session, drafts, q_dists, seed: int, step: int, temperature: float, top_k: int,
                  top_p: float):
    """Score [pending] + drafts with the target (Sec. 2.1, sampling): commits
    the a + 1 new tokens and records the history like the greedy verify."""
    rows = [session.pending] + list(drafts)
    logits, states = session.forward(rows, session.p, capture=True)
    p = [filter_distribution(logits[t], temperature, top_k, top_p) for t in range(len(rows))]
    a, new = speculative_step(p, q_dists, drafts, seed, step)
    session.hist.append(states[:, : a + 1, :])
    session.p += a + 1
    session.pending = int(new[-1])
    return a, new


def spec_sample_generate(cfg, weights, prompt, n_new: int, gamma: int, mask, seed: int,
                         temperature: float = 0.7, top_k: int = 50, top_p: float = 0.95):
    """Sampling-mode self-speculative decoding with a fixed mask; step s uses
    the uniforms of counter step s.  The first token is the prompt's greedy
    token (as in greedy decoding).  Returns (tokens, per-step accepted)."""
    from oracle.decoder import Session
    s = Session(cfg, weights, len(prompt) + n_new + gamma + 2)
    out = [s.prefill(prompt)]
    acc = []
    step = 0
    while len(out) < n_new:
        drafts, q = draft_sample(s, mask, gamma, seed, step, temperature, top_k, top_p)
        a, new = verify_sample(s, drafts, q, seed, step, temperature, top_k, top_p)
        out.extend(new)
        acc.append(a)
        step += 1
    return out[:n_new], acc
