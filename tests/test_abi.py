"""C ABI on the host (no GPU): the library builds and loads, exports every
function include/knapspec.h declares, and rejects bad arguments before any
device work."""
import ctypes as C
import os
import re
import shutil

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "knapspec.h")


@pytest.fixture(scope="module")
def lib():
    if shutil.which("nvcc") is None and not os.path.exists("/usr/local/cuda/bin/nvcc"):
        pytest.skip("nvcc not available")
    from paper_2602_20217_gb300 import build, knapspec
    build.build()
    return knapspec.load()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(ks_\w+)\s*\(", text)))


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert len(names) >= 15
    for n in names:
        assert hasattr(lib, n), n


def test_status_strings(lib):
    from paper_2602_20217_gb300 import knapspec as ks
    for s in range(8):
        assert lib.ks_status_str(s).decode().startswith("KS_")
    assert lib.ks_status_str(99).decode() == "KS_ERR_UNKNOWN"


def test_workspace_bytes_validation(lib):
    from paper_2602_20217_gb300 import knapspec as ks
    from paper_2602_20217_gb300.configs import LLAMA3_8B, QWEN3_32B, TINY
    small = ks.ks_workspace_bytes(ks.make_config(TINY, 512))
    big = ks.ks_workspace_bytes(ks.make_config(LLAMA3_8B, 4096 + 300))
    assert 0 < small < big
    # KV cache alone for 8B at 4396 positions: 2 * 32 * 8 * 4396 * 128 * 2 bytes
    assert big > 2 * 32 * 8 * 4396 * 128 * 2
    assert ks.ks_workspace_bytes(ks.make_config(QWEN3_32B, 65536 + 300)) > 0
    for field, bad in [("head_dim", 96), ("max_rows", 17), ("n_kv_heads", 3), ("d_model", 100),
                       ("dtype", 7), ("max_seq", 1), ("hist_init_rows", 0)]:
        cfg = ks.make_config(TINY, 512)
        setattr(cfg, field, bad)
        assert ks.ks_workspace_bytes(cfg) == 0, field


def test_select_scratch_bytes(lib):
    from paper_2602_20217_gb300 import knapspec as ks
    n = ks.ks_select_scratch_bytes(64, 100)
    assert n >= 64 * 101 + 16 * 101 and n % 256 == 0
    assert ks.ks_select_scratch_bytes(1, 10) == 0
    assert ks.ks_select_scratch_bytes(300, 10) == 0
    assert ks.ks_select_scratch_bytes(64, -1) == 0
    assert ks.ks_select_scratch_bytes(64, 70000) == 0


def test_error_paths_touch_no_device(lib):
    from paper_2602_20217_gb300 import knapspec as ks
    from paper_2602_20217_gb300.configs import TINY
    cfg = ks.make_config(TINY, 512)
    h = C.c_void_p()
    # null weights / workspace / out
    assert lib.ks_model_create(C.byref(cfg), None, None, 0, None, C.byref(h)) == ks.KS_ERR_INVALID_ARG
    assert lib.ks_model_create(C.byref(cfg), None, None, 0, None, None) == ks.KS_ERR_INVALID_ARG
    assert b"null" in lib.ks_last_error()
    # invalid config is rejected before the weights are looked at
    bad = ks.make_config(TINY, 512)
    bad.head_dim = 80
    assert lib.ks_model_create(C.byref(bad), None, None, 0, None, C.byref(h)) == ks.KS_ERR_INVALID_ARG
    # misaligned workspace
    w = ks.KsWeights()
    assert lib.ks_model_create(C.byref(cfg), C.byref(w), 0x1001, 1 << 20, None, C.byref(h)) == ks.KS_ERR_INVALID_ARG
    # model calls on a null handle
    out = np.zeros(8, np.int32)
    a, n = C.c_int32(), C.c_int32()
    assert lib.ks_prefill(None, out.ctypes.data, 4, C.byref(a)) == ks.KS_ERR_INVALID_ARG
    assert lib.ks_draft(None, out.ctypes.data, 4, None) == ks.KS_ERR_INVALID_ARG
    assert lib.ks_draft_dynamic(None, out.ctypes.data, 4, 0.7, None, None, None) == ks.KS_ERR_INVALID_ARG
    assert lib.ks_verify(None, None, 4, C.byref(a), out.ctypes.data, C.byref(n)) == ks.KS_ERR_INVALID_ARG
    assert lib.ks_decode_greedy(None, 4, out.ctypes.data) == ks.KS_ERR_INVALID_ARG
    assert lib.ks_model_destroy(None) == ks.KS_ERR_INVALID_ARG
    assert lib.ks_launch_count(None) == -1
    lat, _ = ks.latency(0, 1.0, 0.0, 1.0)
    g, t = C.c_int32(), C.c_double()
    assert lib.ks_select_tpt(None, C.byref(lat), 4, 4, out.ctypes.data, C.byref(g), C.byref(t), None,
                             None) == ks.KS_ERR_INVALID_ARG
    samp = ks.sampling(0.7, 50, 0.95, 1)
    assert lib.ks_draft_sample(None, out.ctypes.data, 4, C.byref(samp), 0, None) == ks.KS_ERR_INVALID_ARG
    assert lib.ks_verify_sample(None, 4, C.byref(samp), 0, C.byref(a), out.ctypes.data,
                                C.byref(n)) == ks.KS_ERR_INVALID_ARG
    assert lib.ks_select_dp(None, C.byref(lat), 0.5, 4, 8, 8, None, 0, out.ctypes.data, C.byref(g), C.byref(t),
                            None, None, None, None) == ks.KS_ERR_INVALID_ARG
    assert lib.ks_dp_scratch_bytes(None, 8, 8) == 0


def test_select_mask_argument_checks(lib):
    from paper_2602_20217_gb300 import knapspec as ks
    lat, _ = ks.latency(0, 0.3, 1e-5, 0.1)
    fake = 0x10000  # never dereferenced: every call below fails validation first
    args = dict(context_len=4096, n_sublayers=8, budget_units=5)

    def call(lat_, sims=fake, n=8, budget=5, mask=fake, scratch=fake, nbytes=1 << 20, ctx=4096):
        return lib.ks_select_mask(C.byref(lat_), sims, ctx, n, budget, mask, None, None, scratch, nbytes, None)

    assert call(lat, sims=None) == ks.KS_ERR_INVALID_ARG
    assert call(lat, mask=None) == ks.KS_ERR_INVALID_ARG
    assert call(lat, n=7) == ks.KS_ERR_INVALID_ARG
    assert call(lat, n=258) == ks.KS_ERR_INVALID_ARG
    assert call(lat, budget=-1) == ks.KS_ERR_INVALID_ARG
    assert call(lat, ctx=-5) == ks.KS_ERR_INVALID_ARG
    assert call(lat, scratch=fake + 4) == ks.KS_ERR_INVALID_ARG
    assert call(lat, nbytes=16) == ks.KS_ERR_WORKSPACE
    bad, _ = ks.latency(0, 0.0, 1e-5, 0.1)                 # c1 must be > 0
    assert call(bad) == ks.KS_ERR_INVALID_ARG
    units = np.array([1, 2, 3, 0, 1, 1, 1, 1], np.int32)  # a unit < 1
    bad, keep = ks.latency(1, units=units)
    assert call(bad) == ks.KS_ERR_INVALID_ARG
    bad, _ = ks.latency(5)
    assert call(bad) == ks.KS_ERR_INVALID_ARG
    # t_Attn(n) = c2 n + c3 must be positive at the context length used
    zero_attn, _ = ks.latency(0, 0.3, 0.0, 0.0)
    assert call(zero_attn, ctx=0) == ks.KS_ERR_INVALID_ARG
    assert call(zero_attn, ctx=4096) == ks.KS_ERR_INVALID_ARG
    # the ratio of the two times must fit the integer weights (at most 65535)
    lopsided, _ = ks.latency(0, 1.0, 0.0, 1.0 / 70000.0)
    assert call(lopsided) == ks.KS_ERR_INVALID_ARG
    ok_ratio, _ = ks.latency(0, 1.0, 0.0, 1.0 / 60000.0)
    assert call(ok_ratio, nbytes=16) == ks.KS_ERR_WORKSPACE   # passes the model check, fails the next one
    growing, _ = ks.latency(0, 1e-9, 1e-9, 0.0)            # t_Attn / t_MLP = n: valid at 4096, not at 1e6
    assert call(growing, nbytes=16) == ks.KS_ERR_WORKSPACE
    assert call(growing, ctx=1000000) == ks.KS_ERR_INVALID_ARG
    # the allocation-free variant applies the same checks before any device work
    for bad_lat, ctx in [(zero_attn, 0), (lopsided, 4096), (growing, 1000000)]:
        assert lib.ks_select_mask_static(C.byref(bad_lat), fake, ctx, 8, 5, fake, None, None,
                                         None) == ks.KS_ERR_INVALID_ARG
    assert args


def test_cosine_argument_checks(lib):
    from paper_2602_20217_gb300 import knapspec as ks
    f = 0x10000
    assert lib.ks_cosine(None, f, 0, 1, 1, 8, 0, None, f, None) == ks.KS_ERR_INVALID_ARG
    assert lib.ks_cosine(f, f, 0, 0, 1, 8, 0, None, f, None) == ks.KS_ERR_INVALID_ARG
    assert lib.ks_cosine(f, f, 0, 1, 0, 8, 0, None, f, None) == ks.KS_ERR_INVALID_ARG
    assert lib.ks_cosine(f, f, 3, 1, 1, 8, 0, None, f, None) == ks.KS_ERR_INVALID_ARG


def test_product_path_fails_loudly_without_library(tmp_path):
    from paper_2602_20217_gb300 import knapspec as ks
    saved = ks._lib
    ks._lib = None
    try:
        with pytest.raises(RuntimeError, match="not found"):
            ks.load(str(tmp_path / "missing.so"))
    finally:
        ks._lib = saved


def test_fit_latency_matches_the_oracle_fit(lib):
    """App. C's least-squares fit in the library equals the oracle's
    (np.linalg.lstsq) fit, and the non-negativity rules apply."""
    from oracle import select as S
    from paper_2602_20217_gb300 import knapspec as ks
    rng = np.random.default_rng(4)
    ns = np.array([4096, 8192, 16384, 32768, 65536], np.float64)
    t_attn = 0.01 + 6.9e-7 * ns + rng.normal(0, 1e-4, len(ns))
    t_mlp = 0.16 + rng.normal(0, 1e-3, 3)
    got = ks.ks_fit_latency(ns, t_attn, t_mlp)
    c1, c2, c3 = S.fit_latency(ns, t_attn, t_mlp)
    assert got.kind == 0
    assert got.c1 == pytest.approx(c1, rel=1e-12)
    assert got.c2 == pytest.approx(c2, rel=1e-9)
    assert got.c3 == pytest.approx(c3, rel=1e-9)
    # a negative intercept: refitted through the origin
    got = ks.ks_fit_latency([1000.0, 2000.0, 3000.0], [0.9, 2.0, 3.1], [0.5])
    assert got.c3 == 0.0
    assert got.c2 == pytest.approx((1000 * 0.9 + 2000 * 2.0 + 3000 * 3.1) / (1000 ** 2 + 2000 ** 2 + 3000 ** 2))
    # a negative slope: the mean time as the intercept
    got = ks.ks_fit_latency([1000.0, 2000.0], [0.3, 0.2], [0.5])
    assert got.c2 == 0.0 and got.c3 == pytest.approx(0.25)
    # too few points, equal lengths, non-positive MLP time
    for args in [([1.0], [1.0], [1.0]), ([5.0, 5.0], [1.0, 2.0], [1.0]), ([1.0, 2.0], [1.0, 2.0], [0.0])]:
        with pytest.raises(ks.KsError):
            ks.ks_fit_latency(*args)

