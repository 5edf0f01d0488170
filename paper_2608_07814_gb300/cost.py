"""Algorithmic byte and FLOP counts of the amortised compressed-MoE forward.

These are the counts the method must move or compute (never the uncompressed
work), used as the numerators of the roofline fractions.

Per token and projection, an anchor (a dominant or a tree root) costs ``2*I*H``
FLOPs and ``I*H`` weight elements; a rank-r correction costs ``2*r*(I+H)``
FLOPs and ``r*(I+H)`` elements (``x V`` then ``(x V) U^T``).  The amortised
forward evaluates each anchor once per (token, anchor) and each correction once
per (token, correction node) -- Sec. 5.1 (a shared product is evaluated one
time per token and reused by every selected expert below it) and the Sec. 5.2
display equation:

    speedup = k * 2IH / (2IH + k * 2r(I+H))      (gate_proj, k co-selected
                                                  members of one cluster)

which gives 1.9227x for Mixtral-8x7B's gate_proj (k=2, I=14336, H=4096, r=64),
235 M vs 122 M FLOPs and 235 MB vs 122 MB of bf16 weights (Fig. 3).
"""
from __future__ import annotations

from typing import Dict, Sequence

import numpy as np


def dense_proj_flops(I: int, H: int, k: int) -> int:
    """k full experts, one projection: k * 2IH (Sec. 5.2)."""
    return k * 2 * I * H


def amortised_proj_flops(I: int, H: int, k: int, r: int) -> int:
    """Shared dominant once plus k rank-r corrections: 2IH + k * 2r(I+H)."""
    return 2 * I * H + k * 2 * r * (I + H)


def proj_speedup(I: int, H: int, k: int, r: int) -> float:
    return dense_proj_flops(I, H, k) / amortised_proj_flops(I, H, k, r)


def anchor_elems(H: int, I: int) -> int:
    """gate + up + down of one anchor."""
    return 3 * I * H


def correction_elems(H: int, I: int, r: int) -> int:
    """Ug, Vg, Uu, Vu, Ud, Vd of one rank-r correction node."""
    return 3 * r * (I + H)


def layer_elems(H: int, I: int, node_parent: Sequence[int], node_rank: Sequence[int]) -> int:
    return int(sum(anchor_elems(H, I) if p < 0 else correction_elems(H, I, r)
                   for p, r in zip(node_parent, node_rank)))


def kept_fraction(H: int, I: int, E: int, node_parent, node_rank) -> float:
    """Stored expert parameters / uncompressed expert parameters (Sec. 3.3)."""
    return layer_elems(H, I, node_parent, node_rank) / (E * anchor_elems(H, I))


def step_counts(H: int, I: int, E: int, node_parent: Sequence[int], node_rank: Sequence[int],
                node_tokens: Sequence[int], T: int, w_bytes: int, x_bytes: int) -> Dict[str, float]:
    """Algorithmic work of one forward over T tokens with the realised routing.

    ``node_tokens[n]`` = |T_n|, the number of tokens whose selected experts'
    paths contain node n (zero = untouched).  Weight bytes count every touched
    node once (the streaming minimum); FLOPs count each (token, node) pair once.
    The router reads W_r [E, H] once and computes T*E*H multiply-adds.
    """
    node_tokens = np.asarray(node_tokens, np.int64)
    wb = 0
    fl = 0
    for p, r, c in zip(node_parent, node_rank, node_tokens):
        if c <= 0:
            continue
        if p < 0:
            wb += anchor_elems(H, I) * w_bytes
            fl += int(c) * 2 * anchor_elems(H, I)
        else:
            wb += correction_elems(H, I, int(r)) * w_bytes
            fl += int(c) * 2 * correction_elems(H, I, int(r))
    router_bytes = E * H * w_bytes
    io_bytes = 2 * T * H * x_bytes
    return dict(weight_bytes=float(wb), router_bytes=float(router_bytes),
                io_bytes=float(io_bytes), bytes=float(wb + router_bytes + io_bytes),
                expert_flops=float(fl), router_flops=float(2 * T * E * H),
                flops=float(fl + 2 * T * E * H))
