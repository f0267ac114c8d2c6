"""Linear-layer shapes of the Qwen2.5-shaped stacks used as workloads.

Only shapes: the weights are random-init stand-ins (no trained checkpoint is
used).  Every projection is ``[N_out, K_in]`` row-major, head_dim 128.  The
q/k/v projections share their input and are stored as one concatenated
``qkv`` matrix; gate and up share theirs and are stored as one ``gate_up``
matrix whose first ``I`` rows are the gate and last ``I`` rows the up
projection (Sec. III-D.2/3: the draft and verify passes run every projection
plus lm_head).
"""
from __future__ import annotations

from dataclasses import dataclass


@dataclass(frozen=True)
class StackShape:
    name: str
    hidden: int
    q_heads: int
    kv_heads: int
    intermediate: int
    vocab: int
    layers: int
    head_dim: int = 128

    @property
    def q_out(self) -> int:
        return self.q_heads * self.head_dim

    @property
    def kv_out(self) -> int:
        return self.kv_heads * self.head_dim

    def projections(self):
        """(name, N_out, K_in) for one decoder layer's linear layers."""
        h, i = self.hidden, self.intermediate
        return [
            ("qkv", self.q_out + 2 * self.kv_out, h),
            ("o", h, self.q_out),
            ("gate_up", 2 * i, h),
            ("down", h, i),
        ]

    def lm_head(self):
        return ("lm_head", self.vocab, self.hidden)

    def linear_params(self) -> int:
        per_layer = sum(n * k for _, n, k in self.projections())
        _, n, k = self.lm_head()
        return self.layers * per_layer + n * k


QWEN25_0P5B_MLP = StackShape("qwen2.5-0.5b-mlp", 896, 14, 2, 4864, 151936, 1)
QWEN25_1P5B = StackShape("qwen2.5-1.5b", 1536, 12, 2, 8960, 151936, 28)
QWEN25_7B = StackShape("qwen2.5-7b", 3584, 28, 4, 18944, 152064, 28)
QWEN25_14B = StackShape("qwen2.5-14b", 5120, 40, 8, 13824, 152064, 48)

STACKS = {s.name: s for s in (QWEN25_0P5B_MLP, QWEN25_1P5B, QWEN25_7B, QWEN25_14B)}
