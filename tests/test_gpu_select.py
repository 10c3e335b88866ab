"""GPU parity of a4 (ks_cosine) and a5 (ks_select_mask) against the oracle.

Masks and weights must be bit-exact and the objective equal to the oracle's
fixed-point total / 2^30 (the stated tolerance is 1e-6; integer quantisation
makes it exact).  Cosines within 1e-3 absolute (observed ~1e-6)."""
import numpy as np
import pytest

from helpers import need_gpu
from oracle import select as S

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    need_gpu()
    import torch
    return torch.device("cuda:0")


def run_select(dev, sigma, n, budget, lat_kind, c=(0.3, 1e-5, 0.1), units=None):
    import torch
    from paper_2602_20217_gb300 import knapspec as ks
    N = len(sigma)
    sims = torch.tensor(np.asarray(sigma, np.float32), device=dev)
    mask = torch.zeros(N, dtype=torch.uint8, device=dev)
    obj = torch.zeros(1, dtype=torch.float64, device=dev)
    wts = torch.zeros(N, dtype=torch.int32, device=dev)
    nbytes = ks.ks_select_scratch_bytes(N, budget)
    scratch = torch.empty(nbytes, dtype=torch.uint8, device=dev)
    lat, keep = ks.latency(lat_kind, *c, units=units)
    ks.ks_select_mask(lat, sims, n, N, budget, mask, obj, wts, scratch, nbytes)
    torch.cuda.synchronize()
    return mask.cpu().numpy(), float(obj.item()), wts.cpu().numpy()


def check_against_oracle(dev, sigma, n, budget, kind, c=(0.3, 1e-5, 0.1), units=None):
    mask, obj, w = run_select(dev, sigma, n, budget, kind, c, units)
    if kind == 0:
        rm, robj, rw = S.select_mask(sigma, budget, len(sigma), *c, n=n)
    else:
        rm, robj, rw = S.select_mask(sigma, budget, len(sigma), units=units)
    assert list(w) == list(rw)
    assert list(mask) == list(rm), (mask, rm)
    assert obj == robj
    assert abs(obj - robj) <= 1e-6
    assert int(np.asarray(mask) @ np.asarray(rw)) <= budget
    return mask


def test_tiny_workload_knapsack(dev):
    from paper_2602_20217_gb300 import synth
    units = synth.unit_table(8, seed=2)
    rng = np.random.default_rng(0)
    for _ in range(5):
        sigma = rng.uniform(0.0, 1.0, 8).astype(np.float32)
        m = check_against_oracle(dev, sigma, 0, 5, 1, units=units)
        m2, v2 = S.knapsack_brute(units, S.quantize_values(sigma), 5)
        assert list(m) == list(m2)


@pytest.mark.parametrize("N", [8, 16, 64, 72, 128, 256])
def test_latency_model_knapsack(dev, N):
    rng = np.random.default_rng(N)
    for n, c in [(0, (0.279, 0.735e-4, 0.279)), (4096, (0.279, 0.735e-4, 0.279)),
                 (131072, (0.279, 0.735e-4, 0.279)), (32768, (0.52, 0.942e-4, 0.216))]:
        sigma = rng.uniform(0.3, 1.0, N).astype(np.float32)
        wsum = int(S.sublayer_units(N, *c, n=n).sum())
        for frac in (0.0, 0.4, 0.5, 0.7, 1.0):
            check_against_oracle(dev, sigma, n, int(frac * wsum), 0, c)


def test_explicit_units_with_ties(dev):
    rng = np.random.default_rng(7)
    for N in (16, 64, 128):
        units = rng.integers(1, 6, N).astype(np.int32)
        # only four distinct similarities: many equal-value items and masks
        sigma = rng.choice(np.array([0.25, 0.5, 0.75, 0.875], np.float32), N)
        for B in (0, 1, 7, int(units.sum()) // 2, int(units.sum()), int(units.sum()) + 9):
            check_against_oracle(dev, sigma, 0, B, 1, units=units)


def test_brute_force_small(dev):
    rng = np.random.default_rng(11)
    for N in (10, 12, 14):
        units = rng.integers(1, 5, N).astype(np.int32)
        sigma = rng.uniform(-0.2, 1.05, N).astype(np.float32)   # includes q < 0 items
        B = int(units.sum() * 0.45)
        mask, obj, _ = run_select(dev, sigma, 0, B, 1, units=units)
        bm, bv = S.knapsack_brute(units, S.quantize_values(sigma), B)
        assert list(mask) == list(bm) and obj == bv / 2 ** 30


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_cosine_matches_oracle(dev, dtype):
    import torch
    from paper_2602_20217_gb300 import knapspec as ks
    rng = np.random.default_rng(3)
    P, r, d = 65, 35, 4096
    X = rng.standard_normal((P, r, d)).astype(np.float32)
    Y = (X + 0.3 * rng.standard_normal((P, r, d))).astype(np.float32)
    tdt = torch.float32 if dtype == "f32" else torch.bfloat16
    Xt = torch.tensor(X, device=dev).to(tdt)
    Yt = torch.tensor(Y, device=dev).to(tdt)
    out = torch.zeros(P, dtype=torch.float32, device=dev)
    ks.ks_cosine(Xt, Yt, ks.KS_DTYPE_F32 if dtype == "f32" else ks.KS_DTYPE_BF16, P, r, d, r * d, None, out)
    torch.cuda.synchronize()
    Xr, Yr = Xt.float().cpu().numpy(), Yt.float().cpu().numpy()
    ref = np.array([S.matrix_cos(Xr[p], Yr[p]) for p in range(P)])
    assert np.max(np.abs(out.cpu().numpy() - ref)) < 1e-5
    # row subset via row_index, and one row
    idx = torch.tensor([34, 0, 17, 5], dtype=torch.int32, device=dev)
    ks.ks_cosine(Xt, Yt, ks.KS_DTYPE_F32 if dtype == "f32" else ks.KS_DTYPE_BF16, P, 4, d, r * d, idx, out)
    torch.cuda.synchronize()
    ref = np.array([S.matrix_cos(Xr[p][[34, 0, 17, 5]], Yr[p][[34, 0, 17, 5]]) for p in range(P)])
    assert np.max(np.abs(out.cpu().numpy() - ref)) < 1e-5
    ks.ks_cosine(Xt, Yt, ks.KS_DTYPE_F32 if dtype == "f32" else ks.KS_DTYPE_BF16, 1, 1, d, 0, None, out)
    torch.cuda.synchronize()
    assert abs(out[0].item() - S.matrix_cos(Xr[0][:1], Yr[0][:1])) < 1e-5


def test_cosine_invariants_on_device(dev):
    import torch
    from paper_2602_20217_gb300 import knapspec as ks
    rng = np.random.default_rng(4)
    X = torch.tensor(rng.standard_normal((2, 7, 333)).astype(np.float32), device=dev)
    out = torch.zeros(2, dtype=torch.float32, device=dev)
    ks.ks_cosine(X, X, 0, 2, 7, 333, 7 * 333, None, out)
    torch.cuda.synchronize()
    assert np.allclose(out.cpu().numpy(), 1.0, atol=1e-6)
    Xn = -X
    ks.ks_cosine(X, Xn, 0, 2, 7, 333, 7 * 333, None, out)
    torch.cuda.synchronize()
    assert np.allclose(out.cpu().numpy(), -1.0, atol=1e-6)
