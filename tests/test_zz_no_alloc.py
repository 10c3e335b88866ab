"""The allocation-free knapsack selection, ks_select_mask_static.

Callers that cannot allocate device memory (a plugin whose host framework
owns every buffer, a serving loop that must not call cudaMalloc once it is
running) use this variant: its work tables are an array built into the
library.  Through the C ABI it must give exactly what ks_select_mask gives
with a caller-supplied scratch buffer, on two calls in a row (the array keeps
the previous call's contents, which must not leak into the next result), and
refuse budgets larger than the built-in tables with a clear error.

This file is named to run last, so a failure here leaves every other test's
result in place; it also passes when run alone."""
import numpy as np
import pytest

from helpers import need_gpu

pytestmark = pytest.mark.gpu


def _select(ks, fn, lat, sims, n, budget, ctx):
    import torch
    mask = torch.zeros(n, dtype=torch.uint8, device="cuda")
    obj = torch.zeros(1, dtype=torch.float64, device="cuda")
    wts = torch.zeros(n, dtype=torch.int32, device="cuda")
    if fn == "static":
        ks.ks_select_mask_static(lat, sims, ctx, n, budget, mask, obj, wts)
    else:
        nbytes = ks.ks_select_scratch_bytes(n, budget)
        scratch = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
        ks.ks_select_mask(lat, sims, ctx, n, budget, mask, obj, wts, scratch, nbytes)
    torch.cuda.synchronize()
    return mask.cpu().numpy(), float(obj.item()), wts.cpu().numpy()


def test_static_tables_match_scratch_version_on_consecutive_calls():
    need_gpu()
    import torch
    from paper_2602_20217_gb300 import knapspec as ks
    rng = np.random.default_rng(123)
    cases = [
        # (kind, n_sublayers, budget, context): a large budget first, then a
        # small one, so stale entries from the first call would show
        (1, 128, 3000, 0),
        (0, 64, 40, 131072),
    ]
    for kind, n, budget, ctx in cases:
        sims = torch.tensor(rng.uniform(0.2, 1.0, n).astype(np.float32), device="cuda")
        if kind == 1:
            units = rng.integers(1, 60, n).astype(np.int32)
            lat, keep = ks.latency(1, units=units)
        else:
            lat, keep = ks.latency(0, 0.279, 0.735e-4, 0.279)
        got = _select(ks, "static", lat, sims, n, budget, ctx)
        ref = _select(ks, "scratch", lat, sims, n, budget, ctx)
        assert np.array_equal(got[0], ref[0])
        assert got[1] == ref[1]
        assert np.array_equal(got[2], ref[2])


def test_static_tables_full_extent_against_oracle():
    """The largest problem the built-in tables hold (256 sublayers at the
    largest budget): equal to ks_select_mask and to the oracle's knapsack."""
    need_gpu()
    import torch
    from oracle import select as O
    from paper_2602_20217_gb300 import knapspec as ks
    rng = np.random.default_rng(7)
    n, budget = 256, ks.KS_SELECT_STATIC_MAX_BUDGET
    units = rng.integers(1, 40, n).astype(np.int32)
    lat, keep = ks.latency(1, units=units)
    s32 = rng.uniform(0.2, 1.0, n).astype(np.float32)
    sims = torch.tensor(s32, device="cuda")
    got = _select(ks, "static", lat, sims, n, budget, 0)
    ref = _select(ks, "scratch", lat, sims, n, budget, 0)
    assert np.array_equal(got[0], ref[0]) and got[1] == ref[1] and np.array_equal(got[2], ref[2])
    omask, oval = O.knapsack(units, O.quantize_values(s32), budget)
    assert np.array_equal(got[0], omask)
    assert abs(got[1] - oval / O.Q_SCALE) <= 1e-6
    assert np.array_equal(got[2], units)


def test_static_calls_allocate_no_device_memory():
    """After a first call (which may load the library's device code), further
    calls leave the device's free memory and torch's allocations unchanged."""
    need_gpu()
    import torch
    from paper_2602_20217_gb300 import knapspec as ks
    n, budget = 64, 1000
    rng = np.random.default_rng(11)
    sims = torch.tensor(rng.uniform(0.2, 1.0, n).astype(np.float32), device="cuda")
    lat, keep = ks.latency(0, 0.279, 0.735e-4, 0.279)
    mask = torch.zeros(n, dtype=torch.uint8, device="cuda")
    obj = torch.zeros(1, dtype=torch.float64, device="cuda")
    wts = torch.zeros(n, dtype=torch.int32, device="cuda")
    ks.ks_select_mask_static(lat, sims, 65536, n, budget, mask, obj, wts)
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    alloc0 = torch.cuda.memory_allocated()
    for ctx in (4096, 131072, 65536):
        ks.ks_select_mask_static(lat, sims, ctx, n, budget, mask, obj, wts)
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert torch.cuda.memory_allocated() == alloc0
    assert free1 == free0


def test_static_tables_reject_oversized_budget():
    need_gpu()
    import torch
    from paper_2602_20217_gb300 import knapspec as ks
    sims = torch.full((8,), 0.5, dtype=torch.float32, device="cuda")
    lat, keep = ks.latency(1, units=np.ones(8, np.int32))
    with pytest.raises(ks.KsError) as e:
        _select(ks, "static", lat, sims, 8, ks.KS_SELECT_STATIC_MAX_BUDGET + 1, 0)
    assert e.value.status == ks.KS_ERR_INVALID_ARG
