"""Host-side query-complexity router (Sec. III-B): which parent drafts.

The paper routes each prompt by an estimate of its complexity built from the
prompt's length, its syntactic depth and its named-entity density: low
complexity drafts with the INT4 variant (Q4), medium with the FP8 variant
(Q8), and high complexity decodes directly with the FP16 parent (Q16).  The
paper gives no formula, weights or thresholds (and reports only the routing
shares of its benchmark mix, Sec. IV), so the estimator below is this
library's own: each feature is scaled to [0, 1] by a fixed reference value
and clipped, the score is their weighted mean, and two fixed cut points
split the score into the three classes.

  length          prompt tokens, reference 512 (a long prompt is a harder
                  prompt for a small draft to follow)
  depth           syntactic depth (deepest clause nesting), reference 8
  entity_density  named entities per token, reference 0.2

  score = 0.4 * length' + 0.3 * depth' + 0.3 * entity_density'
  score < 1/3 -> "int4";  score < 2/3 -> "fp8";  otherwise "fp16"

The router runs on the host, outside the hot path; it sees features, not
text: computing syntactic depth or named-entity density needs a parser and
a tagger that are not part of this library, so the caller supplies them.
"""
from __future__ import annotations

import math
from dataclasses import dataclass

LENGTH_REF = 512.0
DEPTH_REF = 8.0
ENTITY_REF = 0.2
WEIGHTS = (0.4, 0.3, 0.3)
CUTS = (1.0 / 3.0, 2.0 / 3.0)
ROUTES = ("int4", "fp8", "fp16")


@dataclass(frozen=True)
class PromptFeatures:
    """Complexity features of one prompt."""

    length: int              # prompt tokens
    depth: float = 0.0       # syntactic depth
    entity_density: float = 0.0  # named entities per token

    def __post_init__(self):
        if not isinstance(self.length, (int,)) or self.length < 0:
            raise ValueError("length must be a non-negative integer")
        for name in ("depth", "entity_density"):
            v = getattr(self, name)
            if not isinstance(v, (int, float)) or not math.isfinite(v) or v < 0:
                raise ValueError(f"{name} must be a finite non-negative number")


def _unit(v: float, ref: float) -> float:
    return min(1.0, max(0.0, v / ref))


def complexity(f: PromptFeatures) -> float:
    """Complexity score in [0, 1]."""
    parts = (_unit(f.length, LENGTH_REF), _unit(f.depth, DEPTH_REF), _unit(f.entity_density, ENTITY_REF))
    return sum(w * p for w, p in zip(WEIGHTS, parts))


def route(f: PromptFeatures) -> str:
    """"int4" (draft with the INT4 variant), "fp8" (draft with the FP8
    variant) or "fp16" (decode directly with the FP16 parent)."""
    s = complexity(f)
    if s < CUTS[0]:
        return ROUTES[0]
    if s < CUTS[1]:
        return ROUTES[1]
    return ROUTES[2]


def route_batch(features) -> dict:
    """Indices of `features` per route, in input order."""
    out = {r: [] for r in ROUTES}
    for i, f in enumerate(features):
        out[route(f)].append(i)
    return out
