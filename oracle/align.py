"""CPU oracle for neuron alignment (Sec. 3.2 Stage 3 (i)).

TEST INFRASTRUCTURE ONLY (like the rest of ``oracle``): imported by the tests,
``__graft_entry__.smoke()`` and the CPU-baseline legs of ``bench.py``.

An expert's intermediate neurons have no canonical order, so a member is
permuted to match its dominant before the residual is decomposed:

* neuron i of an expert is one vector: its gate, up and down weights joined
  end to end (in the ``x W^T`` storage used here: row i of gate [I, H], row i of up
  [I, H] and column i of down [H, I]), a vector of length 3H;
* the cost of matching dominant neuron i with member neuron j is the squared
  distance ``C[i, j] = ||a_i - b_j||^2`` (Eq. cost), computed here from the
  definition (the difference, squared and summed; float64);
* the permutation P minimising ``sum_i C[i, P(i)]`` (Eq. assign) is found
  exactly; the paper uses the Jonker-Volgenant algorithm, the oracle calls
  SciPy's exact linear-assignment solver (a library routine);
* applying P gives the aligned member: its neuron i is the member's neuron
  P(i), i.e. gate/up rows P(i) and down column P(i).  Permuting the hidden
  neurons of a SwiGLU FFN leaves its function unchanged.

Pinned by ``tests/test_oracle_align_pins.py``.
"""
from __future__ import annotations

import numpy as np

__all__ = ["neuron_vectors", "cost_matrix", "assign", "assignment_cost", "permute_expert"]


def neuron_vectors(gate: np.ndarray, up: np.ndarray, down: np.ndarray) -> np.ndarray:
    """[I, 3H] float64: row i = (gate[i, :], up[i, :], down[:, i])."""
    g = np.asarray(gate, np.float64)
    u = np.asarray(up, np.float64)
    d = np.asarray(down, np.float64)
    return np.concatenate([g, u, d.T], axis=1)


def cost_matrix(dom, mem, rows=None) -> np.ndarray:
    """C[i, j] = ||a_i - b_j||^2 for dom = (gate, up, down), mem likewise;
    only the dominant neurons ``rows`` (all by default), in that order."""
    A = neuron_vectors(*dom)
    B = neuron_vectors(*mem)
    rows = np.arange(A.shape[0]) if rows is None else np.asarray(rows, np.int64)
    C = np.empty((len(rows), B.shape[0]), np.float64)
    for q, i in enumerate(rows):
        diff = B - A[i]
        C[q] = np.sum(diff * diff, axis=1)
    return C


def assign(C: np.ndarray) -> np.ndarray:
    """P [n] int32 with P[i] = the member neuron matched to dominant neuron i,
    minimising sum_i C[i, P[i]] exactly."""
    from scipy.optimize import linear_sum_assignment
    rows, cols = linear_sum_assignment(np.asarray(C, np.float64))
    P = np.empty(C.shape[0], np.int32)
    P[rows] = cols
    return P


def assignment_cost(C: np.ndarray, P: np.ndarray) -> float:
    return float(sum(float(C[i, int(P[i])]) for i in range(C.shape[0])))


def permute_expert(gate, up, down, P):
    """The aligned member: neuron i takes the member's neuron P[i]."""
    P = np.asarray(P, np.int64)
    return (np.ascontiguousarray(np.asarray(gate)[P]), np.ascontiguousarray(np.asarray(up)[P]),
            np.ascontiguousarray(np.asarray(down)[:, P]))
