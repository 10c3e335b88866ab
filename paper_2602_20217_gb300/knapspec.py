"""Thin ctypes binding of libknapspec (include/knapspec.h).

Argument marshalling only: every step of the hot path runs in the library's
CUDA kernels.  Functions keep the C names; pointers are passed as integers
(``tensor.data_ptr()``) or numpy arrays for host buffers.  A missing library
is an error - there is no fallback.
"""
from __future__ import annotations

import ctypes as C
import os

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libknapspec.so")

KS_OK, KS_ERR_INVALID_ARG, KS_ERR_CUDA, KS_ERR_WORKSPACE, KS_ERR_CAPACITY, KS_ERR_TIMEOUT, \
    KS_ERR_UNSUPPORTED, KS_ERR_STATE = range(8)
KS_DTYPE_F32, KS_DTYPE_BF16 = 0, 1
KLASS = {"qkv": 0, "attn": 1, "merge": 2, "oproj": 3, "gateup": 4, "down": 5, "lmhead": 6,
         "embed": 7, "accept": 8, "chain": 9, "prep": 10}


class KsConfig(C.Structure):
    _fields_ = [("n_layers", C.c_int32), ("d_model", C.c_int32), ("n_q_heads", C.c_int32),
                ("n_kv_heads", C.c_int32), ("head_dim", C.c_int32), ("d_ff", C.c_int32),
                ("vocab", C.c_int32), ("qk_norm", C.c_int32), ("dtype", C.c_int32),
                ("max_seq", C.c_int32), ("max_rows", C.c_int32), ("hist_steps", C.c_int32),
                ("hist_init_rows", C.c_int32), ("rms_eps", C.c_float), ("rope_theta", C.c_double)]


PP = C.POINTER(C.c_void_p)


class KsWeights(C.Structure):
    _fields_ = [("embed", C.c_void_p), ("lm_head", C.c_void_p), ("final_norm", C.c_void_p),
                ("attn_norm", PP), ("w_qkv", PP), ("w_o", PP), ("q_norm", PP), ("k_norm", PP),
                ("mlp_norm", PP), ("w_gate_up", PP), ("w_down", PP)]


class KsLatency(C.Structure):
    _fields_ = [("kind", C.c_int32), ("c1", C.c_double), ("c2", C.c_double), ("c3", C.c_double),
                ("units", C.POINTER(C.c_int32))]


class KsSampling(C.Structure):
    _fields_ = [("temperature", C.c_float), ("top_k", C.c_int32), ("top_p", C.c_float), ("seed", C.c_uint64)]


class KsSpecParams(C.Structure):
    _fields_ = [("gamma", C.c_int32), ("policy", C.c_int32), ("mask", C.POINTER(C.c_uint8)),
                ("latency", KsLatency), ("budget_frac", C.c_double), ("resolve_every", C.c_int32),
                ("max_steps", C.c_int32), ("tpt_candidates", C.c_int32), ("tpt_max_gamma", C.c_int32),
                ("tau_conf", C.c_double), ("sampling", KsSampling), ("dp_scratch", C.c_void_p),
                ("dp_scratch_bytes", C.c_uint64), ("dp_tau", C.c_float), ("dp_max_states", C.c_int32),
                ("dp_max_rows", C.c_int32)]


class KsSpecStats(C.Structure):
    _fields_ = [("steps", C.c_int64), ("drafted", C.c_int64), ("accepted", C.c_int64),
                ("resolves", C.c_int64), ("attn_skipped", C.c_int64), ("mlp_skipped", C.c_int64)]


class KsError(RuntimeError):
    def __init__(self, status: int, where: str, msg: str):
        super().__init__(f"{where}: {_status_name(status)}: {msg}")
        self.status = status


_lib = None

_SIGS = {
    "ks_workspace_bytes": (C.c_size_t, [C.POINTER(KsConfig)]),
    "ks_model_create": (C.c_int, [C.POINTER(KsConfig), C.POINTER(KsWeights), C.c_void_p, C.c_size_t,
                                  C.c_void_p, C.POINTER(C.c_void_p)]),
    "ks_model_destroy": (C.c_int, [C.c_void_p]),
    "ks_prefill": (C.c_int, [C.c_void_p, C.c_void_p, C.c_int32, C.POINTER(C.c_int32)]),
    "ks_rewind": (C.c_int, [C.c_void_p, C.POINTER(C.c_int32)]),
    "ks_draft": (C.c_int, [C.c_void_p, C.c_void_p, C.c_int32, C.c_void_p]),
    "ks_draft_dynamic": (C.c_int, [C.c_void_p, C.c_void_p, C.c_int32, C.c_float, C.c_void_p, C.c_void_p,
                                   C.c_void_p]),
    "ks_dp_scratch_bytes": (C.c_size_t, [C.c_void_p, C.c_int32, C.c_int32]),
    "ks_select_dp": (C.c_int, [C.c_void_p, C.POINTER(KsLatency), C.c_float, C.c_int32, C.c_int32, C.c_int32,
                               C.c_void_p, C.c_size_t, C.c_void_p, C.POINTER(C.c_int32), C.POINTER(C.c_double),
                               C.POINTER(C.c_int32), C.c_void_p, C.c_void_p, C.c_void_p]),
    "ks_draft_sample": (C.c_int, [C.c_void_p, C.c_void_p, C.c_int32, C.POINTER(KsSampling), C.c_uint64,
                                  C.c_void_p]),
    "ks_verify_sample": (C.c_int, [C.c_void_p, C.c_int32, C.POINTER(KsSampling), C.c_uint64, C.c_void_p,
                                   C.c_void_p, C.c_void_p]),
    "ks_verify": (C.c_int, [C.c_void_p, C.c_void_p, C.c_int32, C.POINTER(C.c_int32), C.c_void_p,
                            C.POINTER(C.c_int32)]),
    "ks_decode_greedy": (C.c_int, [C.c_void_p, C.c_int32, C.c_void_p]),
    "ks_model_position": (C.c_int, [C.c_void_p, C.POINTER(C.c_int32), C.POINTER(C.c_int32)]),
    "ks_cosine": (C.c_int, [C.c_void_p, C.c_void_p, C.c_int32, C.c_int64, C.c_int32, C.c_int32, C.c_int64,
                            C.c_void_p, C.c_void_p, C.c_void_p]),
    "ks_history_similarities": (C.c_int, [C.c_void_p, C.c_void_p, C.POINTER(C.c_int32)]),
    "ks_select_scratch_bytes": (C.c_size_t, [C.c_int32, C.c_int32]),
    "ks_fit_latency": (C.c_int, [C.POINTER(C.c_double), C.POINTER(C.c_double), C.c_int32, C.POINTER(C.c_double),
                                 C.c_int32, C.POINTER(KsLatency)]),
    "ks_select_mask": (C.c_int, [C.POINTER(KsLatency), C.c_void_p, C.c_int64, C.c_int32, C.c_int32, C.c_void_p,
                                 C.c_void_p, C.c_void_p, C.c_void_p, C.c_size_t, C.c_void_p]),
    "ks_select_mask_static": (C.c_int, [C.POINTER(KsLatency), C.c_void_p, C.c_int64, C.c_int32, C.c_int32,
                                        C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p]),
    "ks_generate_speculative": (C.c_int, [C.c_void_p, C.POINTER(KsSpecParams), C.c_int32, C.c_void_p,
                                          C.POINTER(KsSpecStats), C.c_void_p]),
    "ks_debug_read": (C.c_int, [C.c_void_p, C.c_int32, C.c_int32, C.c_int32, C.c_int32, C.c_void_p, C.c_size_t]),
    "ks_debug_set_status": (C.c_int, [C.c_void_p, C.c_int32]),
    "ks_kernel_timing": (C.c_int, [C.c_void_p, C.c_int32, C.c_int32]),
    "ks_kernel_time": (C.c_int, [C.c_void_p, C.c_int32, C.POINTER(C.c_int64), C.POINTER(C.c_double)]),
    "ks_select_tpt": (C.c_int, [C.c_void_p, C.POINTER(KsLatency), C.c_int32, C.c_int32, C.c_void_p,
                                C.POINTER(C.c_int32), C.POINTER(C.c_double), C.c_void_p, C.c_void_p]),
    "ks_kernel_bytes": (C.c_int, [C.c_void_p, C.c_int32, C.POINTER(C.c_double)]),
    "ks_launch_count": (C.c_int64, [C.c_void_p]),
    "ks_transfer_bytes": (C.c_int, [C.c_void_p, C.POINTER(C.c_int64), C.POINTER(C.c_int64)]),
    "ks_status_str": (C.c_char_p, [C.c_int]),
    "ks_last_error": (C.c_char_p, []),
}


def load(path: str | None = None):
    """Load libknapspec.so (build it with ``paper_2602_20217_gb300.build``)."""
    global _lib
    if _lib is not None:
        return _lib
    path = path or LIB_PATH
    if not os.path.exists(path):
        raise RuntimeError(f"libknapspec.so not found at {path}: run "
                           "`python -c 'import __graft_entry__ as g; g.build()'` first")
    lib = C.CDLL(path)
    for name, (res, args) in _SIGS.items():
        f = getattr(lib, name)
        f.restype = res
        f.argtypes = args
    _lib = lib
    return lib


def _status_name(s: int) -> str:
    try:
        return load().ks_status_str(int(s)).decode()
    except Exception:
        return f"status {s}"


def check(status: int, where: str):
    if status != KS_OK:
        raise KsError(status, where, load().ks_last_error().decode())


def _ptr(x) -> int:
    """Device or host address of a torch tensor / numpy array / int."""
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if isinstance(x, np.ndarray):
        return x.ctypes.data
    return x.data_ptr()


def _stream_ptr(stream) -> int | None:
    if stream is None:
        return None
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


# ------------------------------------------------------------ model calls
def make_config(shape, max_seq: int, max_rows: int = 16, hist_steps: int = 5,
                hist_init_rows: int = 8) -> KsConfig:
    return KsConfig(shape.n_layers, shape.d_model, shape.n_q_heads, shape.n_kv_heads, shape.head_dim,
                    shape.d_ff, shape.vocab, int(shape.qk_norm),
                    KS_DTYPE_BF16 if shape.dtype == "bf16" else KS_DTYPE_F32, max_seq, max_rows,
                    hist_steps, hist_init_rows, float(shape.rms_eps), float(shape.rope_theta))


def ks_workspace_bytes(cfg: KsConfig) -> int:
    return int(load().ks_workspace_bytes(C.byref(cfg)))


def make_weights(w: dict, n_layers: int):
    """KsWeights plus the keep-alive pointer arrays from a dict of tensors."""
    def arr(kind):
        if kind not in w["layers"][0]:
            return None, None
        a = (C.c_void_p * n_layers)(*[_ptr(w["layers"][l][kind]) for l in range(n_layers)])
        return C.cast(a, PP), a

    keep = []
    fields = {}
    for kind in ("attn_norm", "w_qkv", "w_o", "q_norm", "k_norm", "mlp_norm", "w_gate_up", "w_down"):
        p, a = arr(kind)
        fields[kind] = p
        keep.append(a)
    kw = KsWeights(_ptr(w["embed"]), _ptr(w["lm_head"]), _ptr(w["final_norm"]), **{k: v for k, v in fields.items() if v is not None})
    return kw, keep


def ks_model_create(cfg: KsConfig, weights: KsWeights, workspace, workspace_bytes: int, stream=None) -> int:
    h = C.c_void_p()
    check(load().ks_model_create(C.byref(cfg), C.byref(weights), _ptr(workspace), workspace_bytes,
                                 _stream_ptr(stream), C.byref(h)), "ks_model_create")
    return h.value


def ks_model_destroy(h: int):
    check(load().ks_model_destroy(h), "ks_model_destroy")


def ks_prefill(h: int, tokens) -> int:
    t = np.ascontiguousarray(tokens, dtype=np.int32)
    nxt = C.c_int32()
    check(load().ks_prefill(h, t.ctypes.data, len(t), C.byref(nxt)), "ks_prefill")
    return nxt.value


def ks_rewind(h: int) -> int:
    nxt = C.c_int32()
    check(load().ks_rewind(h, C.byref(nxt)), "ks_rewind")
    return nxt.value


def ks_draft(h: int, mask, gamma: int, want_tokens: bool = True):
    m = np.ascontiguousarray(mask, dtype=np.uint8)
    out = np.zeros(gamma, np.int32) if want_tokens else None
    check(load().ks_draft(h, m.ctypes.data, gamma, out.ctypes.data if want_tokens else None), "ks_draft")
    return out


def ks_draft_dynamic(h: int, mask, gamma: int, tau_conf: float, want_outputs: bool = True):
    """Drafts with the dynamic exit: (n_drafted, confidences[n], tokens[n]), or
    None without waiting when want_outputs is False."""
    m = np.ascontiguousarray(mask, dtype=np.uint8)
    if not want_outputs:
        check(load().ks_draft_dynamic(h, m.ctypes.data, gamma, float(tau_conf), None, None, None),
              "ks_draft_dynamic")
        return None
    n = C.c_int32()
    conf = np.zeros(gamma, np.float32)
    toks = np.zeros(gamma, np.int32)
    check(load().ks_draft_dynamic(h, m.ctypes.data, gamma, float(tau_conf), C.byref(n), conf.ctypes.data,
                                  toks.ctypes.data), "ks_draft_dynamic")
    return n.value, conf[: n.value], toks[: n.value]


def sampling(temperature: float = 0.7, top_k: int = 50, top_p: float = 0.95, seed: int = 0) -> KsSampling:
    return KsSampling(float(temperature), int(top_k), float(top_p), int(seed))


def ks_draft_sample(h: int, mask, gamma: int, samp: KsSampling, step: int, want_tokens: bool = True):
    m = np.ascontiguousarray(mask, dtype=np.uint8)
    out = np.zeros(gamma, np.int32) if want_tokens else None
    check(load().ks_draft_sample(h, m.ctypes.data, gamma, C.byref(samp), int(step),
                                 out.ctypes.data if want_tokens else None), "ks_draft_sample")
    return out


def ks_verify_sample(h: int, gamma: int, samp: KsSampling, step: int):
    """Returns (n_accepted, new tokens array)."""
    a, n = C.c_int32(), C.c_int32()
    out = np.zeros(gamma + 1, np.int32)
    check(load().ks_verify_sample(h, gamma, C.byref(samp), int(step), C.byref(a), out.ctypes.data, C.byref(n)),
          "ks_verify_sample")
    return a.value, out[: n.value]


def ks_sample_dists(h: int, which: str, start: int, count: int):
    """Sampling distributions on the device: which = "draft" (q of positions
    start..) or "target" (p of the last verify rows start..); a list of
    (ids, probs) per row."""
    raw = np.zeros((count, 1 + 2 * 64), np.int32)
    check(load().ks_debug_read(h, 5 if which == "draft" else 6, 0, start, count, raw.ctypes.data, raw.nbytes),
          "ks_debug_read")
    out = []
    for r in range(count):
        n = int(raw[r, 0])
        out.append((raw[r, 1:1 + n].astype(np.int64), raw[r, 65:65 + n].view(np.float32).astype(np.float32)))
    return out


def ks_select_dp(h: int, lat: KsLatency, n_sublayers: int, tau: float, max_gamma: int, max_states: int,
                 max_rows: int, scratch_ptr: int, scratch_bytes: int):
    """Alg. 1 + the TPT grid: (mask, gamma, tpt, js, alphas, candidate masks)."""
    mask = np.zeros(n_sublayers, np.uint8)
    g, tpt, n = C.c_int32(), C.c_double(), C.c_int32()
    js = np.zeros(max_states, np.int32)
    alphas = np.zeros(max_states, np.float64)
    cands = np.zeros((max_states, n_sublayers), np.uint8)
    check(load().ks_select_dp(h, C.byref(lat), float(tau), max_gamma, max_states, max_rows, scratch_ptr,
                              scratch_bytes, mask.ctypes.data, C.byref(g), C.byref(tpt), C.byref(n), js.ctypes.data,
                              alphas.ctypes.data, cands.ctypes.data), "ks_select_dp")
    k = n.value
    return mask, g.value, tpt.value, js[:k].copy(), alphas[:k].copy(), cands[:k].copy()


def ks_verify(h: int, draft_tokens, gamma: int):
    """Returns (n_accepted, new tokens array)."""
    d = None if draft_tokens is None else np.ascontiguousarray(draft_tokens, dtype=np.int32)
    a, n = C.c_int32(), C.c_int32()
    out = np.zeros(gamma + 1, np.int32)
    check(load().ks_verify(h, None if d is None else d.ctypes.data, gamma, C.byref(a), out.ctypes.data,
                           C.byref(n)), "ks_verify")
    return a.value, out[: n.value]


def ks_decode_greedy(h: int, n_tokens: int, out=None):
    out = np.zeros(n_tokens, np.int32) if out is None else out
    check(load().ks_decode_greedy(h, n_tokens, out.ctypes.data), "ks_decode_greedy")
    return out


def ks_model_position(h: int):
    p, t = C.c_int32(), C.c_int32()
    check(load().ks_model_position(h, C.byref(p), C.byref(t)), "ks_model_position")
    return p.value, t.value


def ks_cosine(X, Y, dtype: int, n_pairs: int, rows: int, d: int, pair_stride: int, row_index, out, stream=None):
    check(load().ks_cosine(_ptr(X), _ptr(Y), dtype, n_pairs, rows, d, pair_stride, _ptr(row_index), _ptr(out),
                           _stream_ptr(stream)), "ks_cosine")


def ks_history_similarities(h: int, sims) -> int:
    r = C.c_int32()
    check(load().ks_history_similarities(h, _ptr(sims), C.byref(r)), "ks_history_similarities")
    return r.value


def latency(kind: int = 0, c1: float = 0.0, c2: float = 0.0, c3: float = 0.0, units=None):
    """KsLatency plus the keep-alive units array."""
    u = None
    if units is not None:
        u = np.ascontiguousarray(units, dtype=np.int32)
    lat = KsLatency(kind, c1, c2, c3, u.ctypes.data_as(C.POINTER(C.c_int32)) if u is not None else None)
    return lat, u


def ks_fit_latency(ns, t_attn, t_mlp):
    """App. C least-squares fit in the library: returns a kind-0 KsLatency."""
    n = np.ascontiguousarray(ns, np.float64)
    ta = np.ascontiguousarray(t_attn, np.float64)
    tm = np.ascontiguousarray(np.atleast_1d(t_mlp), np.float64)
    out = KsLatency()
    check(load().ks_fit_latency(n.ctypes.data_as(C.POINTER(C.c_double)), ta.ctypes.data_as(C.POINTER(C.c_double)),
                                len(n), tm.ctypes.data_as(C.POINTER(C.c_double)), len(tm), C.byref(out)),
          "ks_fit_latency")
    return out


def ks_select_scratch_bytes(n_sublayers: int, budget_units: int) -> int:
    return int(load().ks_select_scratch_bytes(n_sublayers, budget_units))


def ks_select_mask(lat: KsLatency, sims, context_len: int, n_sublayers: int, budget_units: int, mask_out,
                   objective_out, weights_out, scratch, scratch_bytes: int, stream=None):
    check(load().ks_select_mask(C.byref(lat), _ptr(sims), context_len, n_sublayers, budget_units,
                                _ptr(mask_out), _ptr(objective_out), _ptr(weights_out), _ptr(scratch),
                                scratch_bytes, _stream_ptr(stream)), "ks_select_mask")


KS_SELECT_STATIC_MAX_BUDGET = 4095


def ks_select_mask_static(lat: KsLatency, sims, context_len: int, n_sublayers: int, budget_units: int, mask_out,
                          objective_out, weights_out, stream=None):
    """ks_select_mask with the library's built-in work tables (no scratch argument)."""
    check(load().ks_select_mask_static(C.byref(lat), _ptr(sims), context_len, n_sublayers, budget_units,
                                       _ptr(mask_out), _ptr(objective_out), _ptr(weights_out),
                                       _stream_ptr(stream)), "ks_select_mask_static")


def ks_generate_speculative(h: int, params: KsSpecParams, n_tokens: int):
    out = np.zeros(n_tokens, np.int32)
    acc = np.zeros(n_tokens, np.int32)
    st = KsSpecStats()
    check(load().ks_generate_speculative(h, C.byref(params), n_tokens, out.ctypes.data, C.byref(st),
                                         acc.ctypes.data), "ks_generate_speculative")
    return out, st, acc[: st.steps]


def ks_debug_read(h: int, what: int, layer: int, start: int, count: int, out: np.ndarray):
    check(load().ks_debug_read(h, what, layer, start, count, out.ctypes.data, out.nbytes), "ks_debug_read")
    return out


def ks_debug_set_status(h: int, code: int):
    """Host-side fault injection: write `code` into the device status word (0 clears it)."""
    check(load().ks_debug_set_status(h, int(code)), "ks_debug_set_status")


def ks_kernel_timing(h: int, klass: int, enable: bool):
    check(load().ks_kernel_timing(h, klass, int(enable)), "ks_kernel_timing")


def ks_kernel_time(h: int, klass: int):
    n, ms = C.c_int64(), C.c_double()
    check(load().ks_kernel_time(h, klass, C.byref(n), C.byref(ms)), "ks_kernel_time")
    return n.value, ms.value


def ks_kernel_bytes(h: int, klass: int) -> float:
    b = C.c_double()
    check(load().ks_kernel_bytes(h, klass, C.byref(b)), "ks_kernel_bytes")
    return b.value


def ks_select_tpt(h: int, lat: "KsLatency", n_sublayers: int, n_candidates: int, max_gamma: int):
    """TPT stage on the model's history: (mask, gamma, tpt, alphas, candidates)."""
    mask = np.zeros(n_sublayers, np.uint8)
    cand = np.zeros((n_candidates, n_sublayers), np.uint8)
    alphas = np.zeros(n_candidates, np.float64)
    g = C.c_int32()
    t = C.c_double()
    check(load().ks_select_tpt(h, C.byref(lat), n_candidates, max_gamma, mask.ctypes.data, C.byref(g),
                               C.byref(t), alphas.ctypes.data, cand.ctypes.data), "ks_select_tpt")
    return mask, g.value, t.value, alphas, cand


def ks_launch_count(h: int) -> int:
    return int(load().ks_launch_count(h))


def ks_transfer_bytes(h: int):
    a, b = C.c_int64(), C.c_int64()
    check(load().ks_transfer_bytes(h, C.byref(a), C.byref(b)), "ks_transfer_bytes")
    return a.value, b.value
