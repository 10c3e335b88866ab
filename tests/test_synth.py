"""The seeded input generator: host (numpy) and torch implementations agree bit
for bit, bf16 rounding matches torch's round-to-nearest-even, SplitMix64 matches
its published first outputs, and the weights have the stated mean and std."""
import numpy as np
import torch

from paper_2602_20217_gb300 import synth
from paper_2602_20217_gb300.configs import TINY


def test_splitmix64_reference_outputs():
    # SplitMix64 seeded with 1234567: first outputs of the reference generator
    # (Vigna's splitmix64.c): 6457827717110365317, 3203168211198807973
    got = synth.np_bits(1234567, np.arange(2, dtype=np.uint64))
    assert [int(v) for v in got] == [6457827717110365317, 3203168211198807973]


def test_numpy_and_torch_streams_agree():
    key = synth.stream_key(0, 3, "w_qkv")
    idx = np.arange(1000, 1000 + 4096, dtype=np.uint64)
    a = synth.np_bits(key, idx).view(np.int64)
    b = synth.torch_bits(key, 1000, 4096, "cpu").numpy()
    assert np.array_equal(a, b)
    t = torch.empty(4096, dtype=torch.float32)
    synth.torch_normal_(t, key, 0.02, chunk=1000)
    assert np.array_equal(t.numpy(), synth.np_normal32(key, np.arange(4096, dtype=np.uint64), 0.02))
    # a slice of the stream from an element offset equals the same slice of the whole
    u = torch.empty(1500, dtype=torch.float32)
    synth.torch_normal_(u, key, 0.02, chunk=700, start=2000)
    assert np.array_equal(u.numpy(), t.numpy()[2000:3500])


def test_bf16_rounding_matches_torch():
    x = np.random.default_rng(0).standard_normal(100000).astype(np.float32) * 0.02
    x[:4] = [1.00390625, 1.01171875, -1.00390625, 3.0e-39]   # exact ties, subnormal
    ref = torch.tensor(x).to(torch.bfloat16).to(torch.float32).numpy()
    assert np.array_equal(synth.to_bf16_np(x), ref)


def test_weight_statistics_and_row_access():
    w = synth.np_weight(TINY, 0, 1, "w_gate_up")
    assert w.shape == (2 * 688, 256) and w.dtype == np.float32
    assert abs(w.mean()) < 2e-4 and abs(w.std() - 0.02) < 2e-4
    rows = synth.np_weight_rows(TINY, 0, 1, "w_gate_up", [5, 900])
    assert np.array_equal(rows, w[[5, 900]])
    toks = synth.prompt_tokens(TINY, 256)
    assert toks.min() >= 0 and toks.max() < TINY.vocab and len(set(toks.tolist())) > 150
