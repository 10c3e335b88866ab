"""Model shapes and decode workloads (seeded, random-init, synthetic).

Five workloads: a tiny fp32 Llama-style decoder for exhaustive parity, and
Llama-3-8B, Qwen3-8B and Qwen3-32B shaped bf16 decoders at 4k-128k context.
Weights are drawn from the generator in ``synth`` with std 0.02, norm gains 1,
untied LM head; prompts are uniform random token ids.
"""
from __future__ import annotations

from dataclasses import dataclass, field, replace


@dataclass(frozen=True)
class ModelShape:
    name: str
    n_layers: int
    d_model: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    d_ff: int
    vocab: int
    qk_norm: bool = False
    dtype: str = "bf16"          # "f32" or "bf16"
    rms_eps: float = 1e-5
    rope_theta: float = 10000.0

    @property
    def n_sublayers(self) -> int:
        return 2 * self.n_layers

    @property
    def group(self) -> int:
        return self.n_q_heads // self.n_kv_heads

    @property
    def qkv_rows(self) -> int:
        return (self.n_q_heads + 2 * self.n_kv_heads) * self.head_dim

    @property
    def elem_bytes(self) -> int:
        return 2 if self.dtype == "bf16" else 4

    def attn_weight_bytes(self) -> int:
        d = self.d_model
        return self.elem_bytes * (self.qkv_rows * d + d * self.n_q_heads * self.head_dim)

    def mlp_weight_bytes(self) -> int:
        return self.elem_bytes * 3 * self.d_ff * self.d_model

    def kv_bytes_per_layer(self, n: int) -> int:
        """K and V bytes one Attn sublayer reads at context length n."""
        return 2 * self.n_kv_heads * self.head_dim * self.elem_bytes * n

    def lm_head_bytes(self) -> int:
        return self.elem_bytes * self.vocab * self.d_model


@dataclass(frozen=True)
class Workload:
    name: str
    shape: ModelShape
    prompt_len: int
    new_tokens: int
    gammas: tuple
    note: str = ""
    weight_seed: int = 0
    prompt_seed: int = 1
    units_seed: int = 2
    budget_units: int | None = None   # explicit knapsack budget (tiny config)
    resolve_every: int = 64           # optimisation interval T (verify steps)


TINY = ModelShape("tiny-llama-fp32", 4, 256, 4, 2, 64, 688, 1024, dtype="f32",
                  rope_theta=10000.0)
LLAMA3_8B = ModelShape("llama3-8b-shape", 32, 4096, 32, 8, 128, 14336, 128256,
                       rope_theta=500000.0)
QWEN3_8B = ModelShape("qwen3-8b-shape", 36, 4096, 32, 8, 128, 12288, 151936,
                      qk_norm=True, rope_theta=1000000.0)
QWEN3_32B = ModelShape("qwen3-32b-shape", 64, 5120, 64, 8, 128, 25600, 151936,
                       qk_norm=True, rope_theta=1000000.0)

WORKLOADS = {
    "tiny": Workload("tiny", TINY, 256, 32, (4,), budget_units=5,
                     note="exhaustive parity; 8 sublayers with seeded integer units"),
    "llama8b-4k": Workload("llama8b-4k", LLAMA3_8B, 4096, 256, (4,)),
    "qwen8b-32k": Workload("qwen8b-32k", QWEN3_8B, 32768, 256, (2, 4, 6)),
    "llama8b-128k": Workload("llama8b-128k", LLAMA3_8B, 131072, 128, (4,)),
    "qwen32b-64k": Workload("qwen32b-64k", QWEN3_32B, 65536, 128, (4,), resolve_every=1),
}


def truncated(shape: ModelShape, n_layers: int) -> ModelShape:
    """Same shape with fewer layers (for oracle-sized parity runs)."""
    return replace(shape, n_layers=n_layers, name=f"{shape.name}-L{n_layers}")
