"""Oracle of the hidden-state dynamic program of Alg. 1 (Sec. 3.4) and the
TPT selection over its candidates (Sec. 3.5, Alg. 2).  fp64 numpy.
TEST INFRASTRUCTURE ONLY.

Follows:
* Alg. 1 and the recurrence of Sec. 3.4: g[i, j] is the best hidden state of
  the r history rows after sublayer i with skipped weight j; the execute
  candidate is f^(i)(g[i-1, j]), the skip candidate g[i-1, j - w_i]; the one
  with the higher cosine to X^(i) wins.  One pass yields a candidate layer set
  for every skipped weight j.
* Sec. 3.4, "Efficiency via Pruning": states whose cosine to X^(i) is below
  tau = 0.5 and skipped weights above K / 2 are dropped.
* Sec. 3.5 / Eq. 4 / Alg. 2: each terminal state's acceptance estimate is the
  fraction of history rows whose LM-head argmax equals the target's; the grid
  search of Eq. 3 over candidates and gamma picks (S*, gamma*).

Readings where the paper is silent or at odds with itself (listed in the
design notes):
* Pull form of the recurrence: g[i, j] takes the execute candidate when its
  cosine is >= the skip candidate's (ties execute, as the recurrence says);
  a state is valid when its source is valid, its cosine is >= tau and
  j <= K // 2 (explicit flags instead of the all-zero sentinel).
* Column 0 holds the target's states: g[i, 0] = X^(i).
* Attention inside f^(i) for the history rows (positions p - r .. p - 1, the
  last r committed positions): a row attends to the target's K/V for earlier
  positions and to the state's own K/V for the history positions (causal).
* Backtracking follows stored choices; at j = 0 every remaining sublayer is
  executed.  Candidates are ordered by executed weight K - j ascending.
* Prediction = argmax of the LM head after the final RMSNorm (ties: lowest id).
"""
from __future__ import annotations

import numpy as np

from oracle import decoder as D
from oracle import select as S


def sublayer(session, i: int, x: np.ndarray, pos0: int, kv: dict) -> np.ndarray:
    """f^(i) on the rows x at positions pos0.. (1-based sublayer i).  Attn
    sublayers attend to ``kv[l]``: a copy of the target's cache of layer l in
    which the rows write their own K/V."""
    cfg, w = session.cfg, session.w
    l = (i - 1) // 2
    if i % 2 == 1:
        K, V = kv[l]
        return D.attn_sublayer(cfg, w["layers"][l], x, pos0 + np.arange(x.shape[0]), K, V)
    return D.mlp_sublayer(cfg, w["layers"][l], x)


def _state_kv(session, layer: int):
    return session.k[layer].copy(), session.v[layer].copy()


def run_dp(session, hist: np.ndarray, weights, tau: float = 0.5, margins: list | None = None):
    """Alg. 1 over the history rows.  hist: [2L+1, r, d] = X^(0..2L) of the
    last r committed positions; weights: integer w_i of sublayers 1..2L.
    Returns (states, sigma, choices): states[j] = g[2L, j] for the valid
    terminal j, sigma[j] its cosine to X^(2L), choices[i-1][j] in {"e", "s"}.
    ``margins``, if given, collects how far each decision was from flipping."""
    hist = np.asarray(hist, np.float64)
    n_sub = hist.shape[0] - 1
    r = hist.shape[1]
    pos0 = session.p - r
    w = [int(x) for x in weights]
    Jmax = sum(w) // 2
    g = {0: hist[0]}
    sig = {0: 1.0}
    choices = []
    for i in range(1, n_sub + 1):
        wi = w[i - 1]
        X = hist[i]
        execd = {}
        for j, st in g.items():
            if j == 0:
                execd[0] = X                                  # column 0: the target's states
            else:
                kv = {(i - 1) // 2: _state_kv(session, (i - 1) // 2)} if i % 2 == 1 else {}
                execd[j] = sublayer(session, i, st, pos0, kv)
        new, nsig, ch = {}, {}, {}
        for j in range(Jmax + 1):
            ce = execd.get(j)
            cs = g.get(j - wi) if j >= wi else None
            if ce is None and cs is None:
                continue
            se = S.matrix_cos(ce, X) if ce is not None else -np.inf
            ss = S.matrix_cos(cs, X) if cs is not None else -np.inf
            if margins is not None:      # distance of every decision from its threshold (for tests)
                if ce is not None and cs is not None:
                    margins.append(abs(se - ss))
                margins.append(abs(max(se, ss) - tau))
            if se >= ss:
                st, s, c = ce, se, "e"
            else:
                st, s, c = cs, ss, "s"
            if s < tau:
                continue
            new[j], nsig[j], ch[j] = st, s, c
        g, sig = new, nsig
        choices.append(ch)
    return g, sig, choices


def backtrack(choices, weights, j: int) -> np.ndarray:
    """The layer set of terminal state j: 1 = executed, from the stored choices."""
    n_sub = len(choices)
    mask = np.zeros(n_sub, np.uint8)
    for i in range(n_sub, 0, -1):
        if j == 0 or choices[i - 1][j] == "e":
            mask[i - 1] = 1
        else:
            j -= int(weights[i - 1])
    return mask


def select_dp(session, weights, max_gamma: int, tau: float = 0.5, ta=None, tm=None, units=None):
    """Alg. 1 + Alg. 2 on the session's history: candidates from the DP
    (executed weight ascending), Eq. 4 acceptances, Eq. 3 grid.  Returns
    (mask, gamma, tpt, masks, alphas, js)."""
    cfg, w = session.cfg, session.w
    hist = session.history()
    r = hist.shape[1]
    states, sig, choices = run_dp(session, hist, weights, tau)
    js = sorted(states.keys(), reverse=True)                   # executed weight K - j ascending
    target = S.lm_argmax(hist[-1], w["lm_head"], w["final_norm"], cfg.rms_eps)
    masks, alphas = [], []
    for j in js:
        masks.append(backtrack(choices, weights, j))
        pred = S.lm_argmax(states[j], w["lm_head"], w["final_norm"], cfg.rms_eps)
        alphas.append(S.alpha_hat(pred, target))
    c, g, v = S.select_tpt(masks, alphas, cfg.n_layers, max_gamma, ta, tm, units)
    return masks[c], g, v, masks, alphas, js
