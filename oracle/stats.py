"""CPU oracle for the router profiling statistics.

TEST INFRASTRUCTURE ONLY (like the rest of ``oracle``): imported by the tests,
``__graft_entry__.smoke()`` and the CPU-baseline legs of ``bench.py``.

What it computes, from top-k assignments ``ids [T, k]`` (Sec. 3.2 Stage 1
accumulates per-layer firing counts N_e from the router; Sec. 2.2 builds the
expert co-activation graph weighted by normalised pointwise mutual information
and Sec. 3.2 Stage 2 clusters on 1 - NPMI):

* ``fire[e]``: the number of tokens whose selected set contains e (N_e);
* ``coact[i, j]``: the number of tokens whose selected set contains both i and
  j (i != j); ``coact[i, i] = fire[i]``.  A token's selected set is the set of
  its valid ids (ids outside [0, E) are ignored, a repeated id counts once);
* ``npmi[i, j]`` over n tokens, with ``p_i = coact[i, i] / n`` and
  ``p_ij = coact[i, j] / n``:  ``ln(p_ij / (p_i p_j)) / (-ln p_ij)`` when
  0 < p_ij < 1, -1 when p_ij = 0 (never together), +1 when p_ij = 1 (always
  together).  Floating point in float64.

Written as plain loops over tokens and pairs; pinned by
``tests/test_oracle_stats_pins.py``.
"""
from __future__ import annotations

import math

import numpy as np

__all__ = ["coact_counts", "npmi"]


def coact_counts(ids: np.ndarray, E: int):
    """(fire uint64 [E], coact uint64 [E, E]) of the assignments ids [T, k]."""
    ids = np.asarray(ids)
    fire = np.zeros(E, np.uint64)
    coact = np.zeros((E, E), np.uint64)
    for row in ids:
        sel = sorted({int(e) for e in row if 0 <= int(e) < E})
        for i in sel:
            fire[i] += 1
            for j in sel:
                coact[i, j] += 1
    return fire, coact


def npmi(coact: np.ndarray, n_tokens: int) -> np.ndarray:
    """float64 [E, E] NPMI matrix from co-activation counts over n_tokens."""
    E = coact.shape[0]
    out = np.empty((E, E), np.float64)
    n = float(n_tokens)
    for i in range(E):
        for j in range(E):
            cij = int(coact[i, j])
            if cij == 0:
                out[i, j] = -1.0
                continue
            p_ij = cij / n
            if p_ij >= 1.0:
                out[i, j] = 1.0
                continue
            p_i = int(coact[i, i]) / n
            p_j = int(coact[j, j]) / n
            out[i, j] = math.log(p_ij / (p_i * p_j)) / (-math.log(p_ij))
    return out
