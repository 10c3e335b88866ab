"""Seeded synthetic inputs: decoder weights, prompts and latency-unit tables.

This module is the only code shared by the CUDA path's callers and by the
oracle's callers.  It holds no step of the decoding method: it only turns
(seed, tensor id, element index) into numbers.

Generator
---------
SplitMix64 (Steele, Lea & Flood, "Fast splittable pseudorandom number
generators", OOPSLA 2014): the k-th output of a generator whose state starts
at ``key`` is ``mix(key + (k + 1) * 0x9E3779B97F4A7C15)`` with

    z ^= z >> 30; z *= 0xBF58476D1CE4E5B9
    z ^= z >> 27; z *= 0x94D049BB133111EB
    z ^= z >> 31                                  (all mod 2**64)

The generator is counter based, so any element can be regenerated from its
index alone: the oracle re-creates single weight rows of a 16 GB model on the
host without copying anything from the device.

Normal-like weights
-------------------
The four 16-bit lanes u0..u3 of one output are summed (an Irwin-Hall sum of
four uniforms, mean 131070, variance (2**32 - 1) / 3) and scaled to the
requested standard deviation in fp32:

    w = float32(S - 131070) * float32(std / sqrt((2**32 - 1) / 3))

Every step is exact integer arithmetic followed by one correctly rounded fp32
multiply, then (for bf16 models) round-to-nearest-even to bf16, so the host
(numpy) and device (torch) implementations below give bit-identical values.
The distribution has the mean and standard deviation of N(0, std**2) and
excess kurtosis -0.3.

Token ids are ``(z >> 11) % vocab`` (uniform up to a bias below 2**-40).
"""
from __future__ import annotations

import numpy as np

MASK64 = (1 << 64) - 1
GOLDEN = 0x9E3779B97F4A7C15
MIX1 = 0xBF58476D1CE4E5B9
MIX2 = 0x94D049BB133111EB
IH_MEAN = 131070  # mean of the sum of four uniform 16-bit lanes
IH_SD = float(np.sqrt((2.0 ** 32 - 1.0) / 3.0))

# Tensor ids: per layer l (0-based) the id is 16 * l + kind; global tensors use
# layer index GLOBAL_LAYER.
GLOBAL_LAYER = 1 << 20
KIND = {
    "attn_norm": 0, "w_qkv": 1, "w_o": 2, "q_norm": 3, "k_norm": 4,
    "mlp_norm": 5, "w_gate_up": 6, "w_down": 7,
    "embed": 8, "lm_head": 9, "final_norm": 10,
    "prompt": 11, "units": 12, "hidden": 13, "kv": 14, "misc": 15,
}


def _mix_int(z: int) -> int:
    z &= MASK64
    z = ((z ^ (z >> 30)) * MIX1) & MASK64
    z = ((z ^ (z >> 27)) * MIX2) & MASK64
    return z ^ (z >> 31)


def stream_key(seed: int, layer: int, kind: str) -> int:
    """64-bit key of one tensor's stream (a SplitMix64 output of the ids)."""
    return _mix_int((seed & 0xFFFFFFFF) * GOLDEN + (layer * 16 + KIND[kind]) * MIX2 + 1)


# ---------------------------------------------------------------- numpy side
def _np_mix(z: np.ndarray) -> np.ndarray:
    z = z ^ (z >> np.uint64(30))
    z = z * np.uint64(MIX1)
    z = z ^ (z >> np.uint64(27))
    z = z * np.uint64(MIX2)
    return z ^ (z >> np.uint64(31))


def np_bits(key: int, idx: np.ndarray) -> np.ndarray:
    """SplitMix64 outputs number idx (0-based) of the stream with state ``key``."""
    idx = np.asarray(idx, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = np.uint64(key) + (idx + np.uint64(1)) * np.uint64(GOLDEN)
        return _np_mix(z)


def np_normal32(key: int, idx: np.ndarray, std: float) -> np.ndarray:
    """fp32 normal-like values for element indices ``idx`` (see module doc)."""
    z = np_bits(key, idx)
    m = np.uint64(0xFFFF)
    s = (z & m) + ((z >> np.uint64(16)) & m) + ((z >> np.uint64(32)) & m) + (z >> np.uint64(48))
    centred = (s.astype(np.int64) - IH_MEAN).astype(np.float32)
    return centred * np.float32(std / IH_SD)


def np_tokens(key: int, n: int, vocab: int, start: int = 0) -> np.ndarray:
    z = np_bits(key, np.arange(start, start + n, dtype=np.uint64))
    return ((z >> np.uint64(11)) % np.uint64(vocab)).astype(np.int32)


def to_bf16_np(x32: np.ndarray) -> np.ndarray:
    """Round fp32 to the nearest bf16 (ties to even); returns the values as fp32."""
    u = np.ascontiguousarray(x32, dtype=np.float32).view(np.uint32).astype(np.uint64)
    r = (u + np.uint64(0x7FFF) + ((u >> np.uint64(16)) & np.uint64(1))) >> np.uint64(16)
    return (r << np.uint64(16)).astype(np.uint32).view(np.float32)


# ---------------------------------------------------------------- torch side
def _signed(c: int) -> int:
    return c - (1 << 64) if c >= (1 << 63) else c


def _t_lsr(z, s: int):
    """Logical right shift of int64 tensors holding 64-bit unsigned patterns."""
    return (z >> s) & ((1 << (64 - s)) - 1)


def torch_bits(key: int, start: int, n: int, device):
    import torch
    idx = torch.arange(start + 1, start + n + 1, dtype=torch.int64, device=device)
    z = idx * _signed(GOLDEN) + _signed(key)
    z = z ^ _t_lsr(z, 30)
    z = z * _signed(MIX1)
    z = z ^ _t_lsr(z, 27)
    z = z * _signed(MIX2)
    return z ^ _t_lsr(z, 31)


def torch_normal_(out, key: int, std: float, chunk: int = 1 << 25, start: int = 0):
    """Fill a contiguous fp32/bf16 tensor with the generator's values for
    element indices start, start + 1, ... (a slice of a larger tensor's
    stream when start > 0), in chunks."""
    import torch
    flat = out.view(-1)
    total = flat.numel()
    scale = float(np.float32(std / IH_SD))
    for s in range(0, total, chunk):
        n = min(chunk, total - s)
        z = torch_bits(key, start + s, n, out.device)
        lanes = (z & 0xFFFF) + (_t_lsr(z, 16) & 0xFFFF) + (_t_lsr(z, 32) & 0xFFFF) + _t_lsr(z, 48)
        v = (lanes - IH_MEAN).to(torch.float32) * scale
        flat[s:s + n].copy_(v.to(flat.dtype))
        del z, lanes, v
    return out


def torch_tokens(key: int, n: int, vocab: int, device, start: int = 0):
    import torch
    z = torch_bits(key, start, n, device)
    return (_t_lsr(z, 11) % vocab).to(torch.int32)


# ------------------------------------------------------------- model inputs
def weight_shapes(cfg) -> dict:
    """Per-layer and global weight shapes, row-major [out, in]."""
    d, hd = cfg.d_model, cfg.head_dim
    nq = (cfg.n_q_heads + 2 * cfg.n_kv_heads) * hd
    per_layer = {
        "attn_norm": (d,), "w_qkv": (nq, d), "w_o": (d, cfg.n_q_heads * hd),
        "mlp_norm": (d,), "w_gate_up": (2 * cfg.d_ff, d), "w_down": (d, cfg.d_ff),
    }
    if cfg.qk_norm:
        per_layer["q_norm"] = (hd,)
        per_layer["k_norm"] = (hd,)
    glob = {"embed": (cfg.vocab, d), "lm_head": (cfg.vocab, d), "final_norm": (d,)}
    return {"layer": per_layer, "global": glob}


NORM_KINDS = ("attn_norm", "mlp_norm", "q_norm", "k_norm", "final_norm")


def np_weight_rows(cfg, seed: int, layer: int, kind: str, rows, std: float = 0.02) -> np.ndarray:
    """Selected rows of one weight tensor as fp32 (bf16-rounded for bf16 models).

    Norm gains are all ones.  ``layer`` is ignored for global tensors."""
    shapes = weight_shapes(cfg)
    is_global = kind in shapes["global"]
    shape = shapes["global"][kind] if is_global else shapes["layer"][kind]
    if kind in NORM_KINDS:
        return np.ones((len(np.atleast_1d(rows)),) + shape[1:] if len(shape) > 1 else shape, np.float32)
    rows = np.atleast_1d(np.asarray(rows, dtype=np.int64))
    ncol = shape[1]
    key = stream_key(seed, GLOBAL_LAYER if is_global else layer, kind)
    idx = (rows[:, None] * ncol + np.arange(ncol)[None, :]).astype(np.uint64)
    v = np_normal32(key, idx, std)
    return to_bf16_np(v) if cfg.dtype == "bf16" else v


def np_weight(cfg, seed: int, layer: int, kind: str, std: float = 0.02) -> np.ndarray:
    shapes = weight_shapes(cfg)
    shape = shapes["global"][kind] if kind in shapes["global"] else shapes["layer"][kind]
    if kind in NORM_KINDS:
        return np.ones(shape, np.float32)
    return np_weight_rows(cfg, seed, layer, kind, np.arange(shape[0]), std)


def np_model_weights(cfg, seed: int = 0, std: float = 0.02) -> dict:
    """All weights on the host (small models only): {'layers': [dict], 'embed': ...}."""
    shapes = weight_shapes(cfg)
    layers = [{k: np_weight(cfg, seed, l, k, std) for k in shapes["layer"]} for l in range(cfg.n_layers)]
    out = {k: np_weight(cfg, seed, 0, k, std) for k in shapes["global"]}
    out["layers"] = layers
    return out


def torch_model_weights(cfg, seed: int = 0, device="cuda", std: float = 0.02) -> dict:
    """All weights as device tensors with the same values as ``np_model_weights``."""
    import torch
    dt = torch.bfloat16 if cfg.dtype == "bf16" else torch.float32
    shapes = weight_shapes(cfg)

    def make(layer, kind, shape):
        t = torch.empty(shape, dtype=dt, device=device)
        if kind in NORM_KINDS:
            return t.fill_(1.0)
        is_global = kind in shapes["global"]
        key = stream_key(seed, GLOBAL_LAYER if is_global else layer, kind)
        return torch_normal_(t, key, std)

    layers = [{k: make(l, k, s) for k, s in shapes["layer"].items()} for l in range(cfg.n_layers)]
    out = {k: make(0, k, s) for k, s in shapes["global"].items()}
    out["layers"] = layers
    return out


def prompt_tokens(cfg, n: int, seed: int = 1) -> np.ndarray:
    return np_tokens(stream_key(seed, GLOBAL_LAYER, "prompt"), n, cfg.vocab)


def unit_table(n_items: int, seed: int = 2, lo: int = 1, hi: int = 4) -> np.ndarray:
    """Seeded integer latency units, uniform on {lo..hi}, one per sublayer."""
    z = np_bits(stream_key(seed, GLOBAL_LAYER, "units"), np.arange(n_items, dtype=np.uint64))
    return (lo + (z >> np.uint64(11)) % np.uint64(hi - lo + 1)).astype(np.int32)


def np_uniform01(key: int, idx) -> np.ndarray:
    """Uniform doubles in [0, 1) from the top 53 bits."""
    z = np_bits(key, idx)
    return (z >> np.uint64(11)).astype(np.float64) * (2.0 ** -53)
