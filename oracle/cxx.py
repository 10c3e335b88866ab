"""ctypes face of the plain fp32 C++ oracle (oracle/cpp/ksoracle.cpp).

TEST INFRASTRUCTURE ONLY: imported by tests/, __graft_entry__ and the bench's
CPU-baseline leg, never by the library.  The C++ oracle follows the same
passages as the numpy oracle (Sec. 2, 2.1, 3.3, 3.4, App. C) in single-threaded
fp32 loops; ``build()`` compiles it with g++ (no CUDA, no BLAS)."""
from __future__ import annotations

import ctypes as C
import os
import subprocess

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "cpp", "ksoracle.cpp")
LIB = os.path.join(HERE, "cpp", "libksoracle.so")
_lib = None


def build(force: bool = False) -> str:
    """Compile libksoracle.so if it is missing or older than its source."""
    if force or not os.path.exists(LIB) or os.path.getmtime(LIB) < os.path.getmtime(SRC):
        tmp = LIB + ".tmp"
        cmd = ["g++", "-O2", "-std=c++17", "-shared", "-fPIC", "-o", tmp, SRC]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError("g++ failed:\n" + r.stdout + r.stderr)
        os.replace(tmp, LIB)
    return LIB


class KoConfig(C.Structure):
    _fields_ = [("n_layers", C.c_int32), ("d_model", C.c_int32), ("n_q_heads", C.c_int32),
                ("n_kv_heads", C.c_int32), ("head_dim", C.c_int32), ("d_ff", C.c_int32),
                ("vocab", C.c_int32), ("qk_norm", C.c_int32), ("rms_eps", C.c_float),
                ("rope_theta", C.c_double)]


_FP = C.POINTER(C.c_float)
_PP = C.POINTER(_FP)


class KoWeights(C.Structure):
    _fields_ = [("embed", _FP), ("lm_head", _FP), ("final_norm", _FP), ("attn_norm", _PP), ("w_qkv", _PP),
                ("w_o", _PP), ("q_norm", _PP), ("k_norm", _PP), ("mlp_norm", _PP), ("w_gate_up", _PP),
                ("w_down", _PP)]


def load():
    global _lib
    if _lib is None:
        build()
        lib = C.CDLL(LIB)
        i32p, u8p = C.POINTER(C.c_int32), C.POINTER(C.c_uint8)
        vp = C.c_void_p
        lib.ko_attn_sublayer.argtypes = [vp, vp, C.c_int, _FP, C.c_int, i32p, _FP, _FP, C.c_int]
        lib.ko_mlp_sublayer.argtypes = [vp, vp, C.c_int, _FP, C.c_int]
        lib.ko_final_logits.argtypes = [vp, vp, _FP, C.c_int, _FP, C.c_int, C.c_int]
        lib.ko_argmax.argtypes = [_FP, C.c_int]
        lib.ko_matrix_cos.argtypes = [_FP, _FP, C.c_int, C.c_int]
        lib.ko_matrix_cos.restype = C.c_double
        lib.ko_integer_weights.argtypes = [C.c_double, C.c_double, i32p, i32p]
        lib.ko_knapsack.argtypes = [i32p, C.POINTER(C.c_int64), C.c_int, C.c_int, u8p]
        lib.ko_knapsack.restype = C.c_int64
        lib.ko_knapsack_brute.argtypes = lib.ko_knapsack.argtypes
        lib.ko_knapsack_brute.restype = C.c_int64
        lib.ko_session_create.argtypes = [vp, vp, C.c_int, C.c_int, C.c_int]
        lib.ko_session_create.restype = vp
        lib.ko_session_destroy.argtypes = [vp]
        lib.ko_forward.argtypes = [vp, i32p, C.c_int, C.c_int, u8p, _FP, _FP]
        lib.ko_prefill.argtypes = [vp, i32p, C.c_int, C.c_int]
        lib.ko_ar_step.argtypes = [vp]
        lib.ko_draft.argtypes = [vp, u8p, C.c_int, i32p]
        lib.ko_verify.argtypes = [vp, i32p, C.c_int, i32p, i32p]
        lib.ko_position.argtypes = [vp, i32p]
        lib.ko_history.argtypes = [vp, _FP]
        _lib = lib
    return _lib


def _f(a):
    return a.ctypes.data_as(_FP)


def _i(a):
    return a.ctypes.data_as(C.POINTER(C.c_int32))


class Model:
    """Config + fp32 host weights (from synth.np_model_weights, or any dict of
    the same keys) marshalled for the C++ oracle; the arrays stay alive here."""

    def __init__(self, shape, weights: dict):
        self.shape = shape
        self.cfg = KoConfig(shape.n_layers, shape.d_model, shape.n_q_heads, shape.n_kv_heads, shape.head_dim,
                            shape.d_ff, shape.vocab, int(bool(shape.qk_norm)), float(shape.rms_eps),
                            float(shape.rope_theta))
        c32 = lambda a: np.ascontiguousarray(a, np.float32)
        self.glob = {k: c32(weights[k]) for k in ("embed", "lm_head", "final_norm")}
        self.layers = [{k: c32(v) for k, v in lw.items()} for lw in weights["layers"]]
        L = shape.n_layers

        def arr(kind):
            a = (_FP * L)()
            for l in range(L):
                a[l] = _f(self.layers[l][kind]) if kind in self.layers[l] else None
            return a
        self._arrs = {k: arr(k) for k in ("attn_norm", "w_qkv", "w_o", "q_norm", "k_norm", "mlp_norm",
                                          "w_gate_up", "w_down")}
        self.w = KoWeights(_f(self.glob["embed"]), _f(self.glob["lm_head"]), _f(self.glob["final_norm"]),
                           *[C.cast(self._arrs[k], _PP) for k in ("attn_norm", "w_qkv", "w_o", "q_norm", "k_norm",
                                                                  "mlp_norm", "w_gate_up", "w_down")])

    # sublayers on the caller's rows and caches
    def attn_sublayer(self, layer: int, x: np.ndarray, pos, k_cache: np.ndarray, v_cache: np.ndarray) -> np.ndarray:
        y = np.ascontiguousarray(x, np.float32).copy()
        p = np.ascontiguousarray(pos, np.int32)
        assert k_cache.dtype == np.float32 and k_cache.flags.c_contiguous and v_cache.flags.c_contiguous
        load().ko_attn_sublayer(C.byref(self.cfg), C.byref(self.w), layer, _f(y), y.shape[0], _i(p), _f(k_cache),
                                _f(v_cache), k_cache.shape[1])
        return y

    def mlp_sublayer(self, layer: int, x: np.ndarray) -> np.ndarray:
        y = np.ascontiguousarray(x, np.float32).copy()
        load().ko_mlp_sublayer(C.byref(self.cfg), C.byref(self.w), layer, _f(y), y.shape[0])
        return y

    def final_logits(self, x: np.ndarray, rows=None) -> np.ndarray:
        x = np.ascontiguousarray(x, np.float32)
        r0, r1 = (0, self.shape.vocab) if rows is None else rows
        out = np.zeros((x.shape[0], self.shape.vocab), np.float32)
        load().ko_final_logits(C.byref(self.cfg), C.byref(self.w), _f(x), x.shape[0], _f(out), r0, r1)
        return out


class Session:
    """One sequence in the C++ oracle (KV cache, committed length, pending
    token, history of the last hist_steps verify passes)."""

    def __init__(self, model: Model, n_max: int, hist_steps: int = 5, hist_init_rows: int = 8):
        self.m = model
        self.h = load().ko_session_create(C.byref(model.cfg), C.byref(model.w), n_max, hist_steps, hist_init_rows)

    def close(self):
        if self.h:
            load().ko_session_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def forward(self, tokens, pos0: int, mask=None, capture: bool = False):
        sh = self.m.shape
        t = np.ascontiguousarray(tokens, np.int32)
        R = len(t)
        logits = np.zeros((R, sh.vocab), np.float32)
        states = np.zeros((2 * sh.n_layers + 1, R, sh.d_model), np.float32) if capture else None
        mk = None if mask is None else np.ascontiguousarray(mask, np.uint8)
        rc = load().ko_forward(self.h, _i(t), R, pos0, None if mk is None else mk.ctypes.data_as(C.POINTER(C.c_uint8)),
                               _f(logits), _f(states) if capture else None)
        if rc:
            raise ValueError("KV capacity exceeded")
        return logits, states

    def prefill(self, prompt, chunk: int = 256) -> int:
        p = np.ascontiguousarray(prompt, np.int32)
        return int(load().ko_prefill(self.h, _i(p), len(p), chunk))

    def ar_step(self) -> int:
        return int(load().ko_ar_step(self.h))

    def draft(self, mask, gamma: int) -> list:
        mk = np.ascontiguousarray(mask, np.uint8)
        out = np.zeros(gamma, np.int32)
        if load().ko_draft(self.h, mk.ctypes.data_as(C.POINTER(C.c_uint8)), gamma, _i(out)):
            raise ValueError("KV capacity exceeded")
        return [int(t) for t in out]

    def verify(self, drafts) -> tuple:
        d = np.ascontiguousarray(drafts, np.int32)
        a = np.zeros(1, np.int32)
        new = np.zeros(len(d) + 1, np.int32)
        if load().ko_verify(self.h, _i(d), len(d), _i(a), _i(new)):
            raise ValueError("KV capacity exceeded")
        return int(a[0]), [int(t) for t in new[: int(a[0]) + 1]]

    def position(self):
        pend = np.zeros(1, np.int32)
        p = load().ko_position(self.h, _i(pend))
        return int(p), int(pend[0])

    def history(self) -> np.ndarray:
        sh = self.m.shape
        r = int(load().ko_history(self.h, None))
        out = np.zeros((2 * sh.n_layers + 1, r, sh.d_model), np.float32)
        load().ko_history(self.h, _f(out))
        return out


def matrix_cos(x: np.ndarray, y: np.ndarray) -> float:
    x = np.ascontiguousarray(x, np.float32)
    y = np.ascontiguousarray(y, np.float32)
    return float(load().ko_matrix_cos(_f(x), _f(y), x.shape[0] if x.ndim > 1 else 1, x.shape[-1]))


def integer_weights(ta: float, tm: float) -> tuple:
    wa, wm = np.zeros(1, np.int32), np.zeros(1, np.int32)
    load().ko_integer_weights(ta, tm, _i(wa), _i(wm))
    return int(wa[0]), int(wm[0])


def knapsack(weights, values, budget: int, brute: bool = False):
    w = np.ascontiguousarray(weights, np.int32)
    q = np.ascontiguousarray(values, np.int64)
    mask = np.zeros(len(w), np.uint8)
    fn = load().ko_knapsack_brute if brute else load().ko_knapsack
    best = fn(_i(w), q.ctypes.data_as(C.POINTER(C.c_int64)), len(w), int(budget), mask.ctypes.data_as(C.POINTER(C.c_uint8)))
    return mask, int(best)
