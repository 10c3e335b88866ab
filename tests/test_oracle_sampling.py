"""Pins of the sampling-mode oracle (oracle/sampling.py) to things other than
itself: numpy's Philox bit generator, closed forms of the filters and of
inverse-CDF sampling, the exact output distribution of the Sec. 2.1
acceptance rule, and the greedy limit T -> 0."""
import numpy as np
import pytest

from oracle import decoder as D
from oracle import sampling as SP

from test_oracle_decoder import rand_weights, tiny_cfg


@pytest.mark.parametrize("key,counter", [([0x1234, 0x5678], [0, 0, 0, 0]),
                                         ([2**64 - 1, 2**63 + 5], [7, 11, 13, 17]),
                                         ([0, 1], [2**64 - 1, 0, 0, 0]),       # carry into the second word
                                         ([987654321, 0], [2**64 - 2, 2**64 - 1, 3, 0])])
def test_philox_matches_numpy(key, counter):
    # numpy's Philox (4x64, 10 rounds) produces block(counter + 1) first
    c = sum(int(w) << (64 * i) for i, w in enumerate(counter))
    bg = np.random.Philox(key=int(key[0]) + (int(key[1]) << 64), counter=c)
    raw = [int(x) for x in bg.random_raw(8)]
    for b in range(2):
        n = c + 1 + b
        words = [(n >> (64 * i)) & SP.MASK64 for i in range(4)]
        assert list(SP.philox4x64_10(words, key)) == raw[4 * b: 4 * b + 4]


def test_uniforms_lie_on_the_24_bit_grid():
    us = [SP.uniform(42, s, r, p) for s in range(20) for r in range(4) for p in range(3)]
    assert all(0.0 <= u < 1.0 for u in us)
    assert all(float(u * (1 << 24)).is_integer() for u in us)
    assert len(set(us)) == len(us)                     # distinct counters, distinct draws
    assert abs(np.mean(us) - 0.5) < 0.1


def test_filter_closed_forms():
    ids, pr = SP.filter_distribution(np.zeros(100), 0.7, 50, 0.95)
    assert list(ids) == list(range(48)) and np.allclose(pr, 1 / 48)   # 48/50 = 0.96 >= 0.95 > 47/50
    ids, pr = SP.filter_distribution(np.array([0.3, 2.0, -1.0]), 0.7, 1, 0.95)
    assert list(ids) == [1] and pr[0] == 1.0                            # top-1 = argmax
    ids, pr = SP.filter_distribution(np.array([np.log(3.0), 0.0]), 1.0, 2, 0.7)
    assert list(ids) == [0] and pr[0] == 1.0                            # 0.75 >= 0.7 keeps one token
    ids, pr = SP.filter_distribution(np.array([np.log(3.0), 0.0]), 1.0, 2, 0.8)
    assert list(ids) == [0, 1] and np.allclose(pr, [0.75, 0.25])
    i2, p2 = SP.filter_distribution(np.array([2 * np.log(3.0), 0.0]), 2.0, 2, 0.8)
    assert list(i2) == [0, 1] and np.allclose(p2, [0.75, 0.25])         # logits / T
    ids, _ = SP.filter_distribution(np.array([1.0, 5.0, 5.0, 1.0]), 1.0, 3, 1.0)
    assert list(ids) == [1, 2, 0]                                       # ties: lower id first


def test_inverse_cdf_sampling_boundaries():
    ids, pr = [5, 2, 9], [0.5, 0.3, 0.2]
    assert [SP.sample(ids, pr, u) for u in (0.0, 0.4999, 0.5, 0.7999, 0.8, 0.9999)] == [5, 5, 2, 2, 9, 9]


def test_acceptance_rule_reproduces_the_target_distribution():
    # draft x ~ q, accept with min(1, p/q), else resample from norm(max(0, p - q)):
    # the output is distributed as p (Sec. 2.1).  Exact up to the grid's 1/N.
    p = (np.array([0, 1, 2, 3]), np.array([0.4, 0.3, 0.2, 0.1]))
    q = (np.array([2, 0, 3, 1]), np.array([0.4, 0.25, 0.2, 0.15]))
    N = 60
    grid = (np.arange(N) + 0.5) / N
    counts = np.zeros(4)
    accepted = 0
    for u0 in grid:
        x = SP.sample(q[0], q[1], u0)
        for u1 in grid:
            for u2 in grid:
                ok, rep = SP.verify_one(p, q, x, u1, u2)
                counts[x if ok else rep] += 1
                accepted += ok
    dist = counts / counts.sum()
    assert np.max(np.abs(dist - p[1])) < 3.0 / N
    # acceptance probability = sum_x min(p(x), q(x))
    p_of = dict(zip(p[0], p[1]))
    q_of = dict(zip(q[0], q[1]))
    alpha = sum(min(p_of[t], q_of[t]) for t in range(4))
    assert abs(accepted / N**3 - alpha) < 3.0 / N


def test_identical_draft_and_target_always_accept():
    p = SP.filter_distribution(np.random.default_rng(0).normal(size=64), 0.7, 50, 0.95)
    for u0 in np.linspace(0, 0.999, 30):
        x = SP.sample(p[0], p[1], u0)
        for u1 in np.linspace(0, 0.999999, 30):
            assert SP.verify_one(p, p, x, u1, 0.5) == (True, None)


def test_zero_temperature_limit_is_greedy_and_full_mask_accepts_all():
    cfg = tiny_cfg(L=2)
    w = rand_weights(cfg, seed=31, std=0.6)
    prompt = np.random.default_rng(32).integers(0, cfg.vocab, 12)
    ar = D.greedy_generate(cfg, w, prompt, 16)
    mask = np.array([1, 0, 0, 1], np.uint8)
    toks, acc = SP.spec_sample_generate(cfg, w, prompt, 16, 3, mask, seed=5, temperature=1e-6)
    assert toks == ar
    full = np.ones(2 * cfg.n_layers, np.uint8)
    toks, acc = SP.spec_sample_generate(cfg, w, prompt, 16, 3, full, seed=6)
    assert all(a == 3 for a in acc)                   # q == p: every draft accepted
