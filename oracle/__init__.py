"""CPU oracle for the LorExperts / BTExperts compressed-MoE forward.

TEST INFRASTRUCTURE ONLY.  Only the test-suite, ``__graft_entry__.smoke()`` and
the CPU-baseline leg of ``bench.py`` may import this package.  It shares no code
with the CUDA library: it reads the synthetic layer (``synth``) and computes,
slowly and plainly, what the paper defines.

What it computes (all floating point in float64 from the exact stored values,
except the router logits, see below):

1. Expert weights, by reconstruction (Sec. 3.1 display ``W_m ~ W_dom + B_m A_m``;
   Sec. 3.2 Stage 3(iii) "installation"; Sec. 5 tree: an expert's weights are the
   sum of the contributions on its root path).  For every projection
   p in {gate, up, down}:  ``W_e^p = W_anchor^p + sum_{n on path(e), n != anchor}
   s_n U_n^p (V_n^p)^T``  with ``U = B`` ([out, r]), ``V = A^T`` ([in, r]) and
   ``s_n`` in {+1, -1} the label of the edge into n (Fig. 2; +1 when the layer
   carries no signs).
2. Routing (Sec. 1 and Fig. 1: top-k over all E experts by the unchanged
   router; Sec. 5.2 names the routing top-k).  Logits ``l = x W_r^T (+ b)`` in the
   canonical fp32 order of ``router_canonical.c``; top-k by (logit descending,
   expert id ascending); gates = softmax over the k selected logits (float64).
3. The standard MoE forward on the reconstructed experts (Sec. 5.1, the
   quantity the amortised forward reproduces): for every token t and slot s
   with expert e = id[t, s] and gate g = gate[t, s],
   ``out[t, s] = g * W_e^down (silu(W_e^gate x_t) * (W_e^up x_t))``,
   ``silu(z) = z / (1 + exp(-z))``, and ``y_t = sum_s out[t, s]`` in slot order.
4. Bucketing (what Sec. 5.1's one evaluation per token of each shared product needs):
   per node n, the ascending list of tokens whose selected experts' root paths
   contain n; per (assignment, path level) the row of that (token, node) pair;
   per expert, its assignments in ascending token order.  Written as plain
   loops.

Parity of every function here is pinned by ``tests/test_oracle_pins.py``
against closed forms, library routines and invariants (full-rank SVD
reconstruction, dominant zero-correction, router invariance, tree == flat,
brute-force top-k and bucketing, Fig. 3 closed forms).
"""
from __future__ import annotations

from typing import Dict, List, Optional, Sequence

import numpy as np

from synth import CompressedLayer, from_storage
from . import _clib

__all__ = [
    "router_logits", "topk", "gates", "route", "expert_weights", "silu",
    "expert_output", "moe_forward", "buckets", "build", "edge_sign",
]


def build() -> None:
    """Compile the oracle's C part (gcc)."""
    _clib.build()


# ----------------------------------------------------------------------------
# 2. routing
# ----------------------------------------------------------------------------
def router_logits(layer: CompressedLayer, x: np.ndarray) -> np.ndarray:
    """fp32 [T, E] logits in the canonical order (see router_canonical.c)."""
    if layer.dtype not in ("f32", "bf16"):
        raise ValueError("canonical router logits need f32 or bf16 storage")
    T, H = x.shape
    E = layer.n_experts
    assert H == layer.d_model and H % 8 == 0
    want = np.uint16 if layer.dtype == "bf16" else np.float32
    xs = np.ascontiguousarray(x, dtype=want)
    ws = np.ascontiguousarray(layer.router_w, dtype=want)
    bias = None if layer.router_bias is None else np.ascontiguousarray(layer.router_bias, np.float32)
    out = np.empty((T, E), np.float32)
    rc = _clib.lib().oracle_router_logits(
        xs.ctypes.data, ws.ctypes.data, None if bias is None else bias.ctypes.data,
        1 if layer.dtype == "bf16" else 0, T, E, H, out.ctypes.data)
    if rc != 0:
        raise ValueError("oracle_router_logits rejected its arguments")
    return out


def topk(logits: np.ndarray, k: int) -> np.ndarray:
    """Per token, the k experts with the largest logits; ties go to the lower
    expert id; slot order = (logit descending, id ascending).  int32 [T, k]."""
    T, E = logits.shape
    ids = np.broadcast_to(np.arange(E), (T, E))
    # lexsort: last key is primary.  -logit ascending == logit descending.
    order = np.lexsort((ids, -logits.astype(np.float64)), axis=1)
    return np.ascontiguousarray(order[:, :k].astype(np.int32))


def gates(logits: np.ndarray, ids: np.ndarray) -> np.ndarray:
    """Softmax over the selected logits, float64 [T, k]."""
    sel = np.take_along_axis(logits.astype(np.float64), ids.astype(np.int64), axis=1)
    z = np.exp(sel - sel.max(axis=1, keepdims=True))
    return z / z.sum(axis=1, keepdims=True)


def route(layer: CompressedLayer, x: np.ndarray, k: Optional[int] = None):
    """Returns (topk_id int32 [T,k], gates float64 [T,k], logits float32 [T,E])."""
    k = layer.top_k if k is None else k
    l = router_logits(layer, x)
    ids = topk(l, k)
    return ids, gates(l, ids), l


# ----------------------------------------------------------------------------
# 1. reconstruction and 3. the standard MoE forward
# ----------------------------------------------------------------------------
def _path(layer: CompressedLayer, e: int) -> List[int]:
    out = []
    n = int(layer.expert_node[e])
    while n >= 0:
        out.append(n)
        n = int(layer.node_parent[n])
    return out


def _correction(layer: CompressedLayer, n: int, p: int) -> np.ndarray:
    """U_n^p (V_n^p)^T for projection p (0 gate, 1 up, 2 down), float64 [out, in]."""
    w = layer.node_w[n]
    U = from_storage(w[2 * p], layer.dtype)
    V = from_storage(w[2 * p + 1], layer.dtype)
    return U @ V.T


def edge_sign(layer: CompressedLayer, n: int) -> float:
    """Sign of the edge into node n (Fig. 2's -1/+1 labels); +1 without signs."""
    signs = getattr(layer, "node_sign", None)
    return 1.0 if signs is None else float(signs[n])


def expert_weights(layer: CompressedLayer, e: int):
    """(W_gate [I,H], W_up [I,H], W_down [H,I]) of expert e, float64."""
    path = _path(layer, e)
    anchor = path[-1]
    Ws = [from_storage(a, layer.dtype).copy() for a in layer.node_w[anchor]]
    for n in path[:-1]:
        s = edge_sign(layer, n)
        for p in range(3):
            Ws[p] += s * _correction(layer, n, p)
    return tuple(Ws)


def silu(z: np.ndarray) -> np.ndarray:
    return z / (1.0 + np.exp(-z))


def expert_output(Wg: np.ndarray, Wu: np.ndarray, Wd: np.ndarray, xs: np.ndarray) -> np.ndarray:
    """SwiGLU expert applied to rows xs [n, H] -> [n, H] (x W^T convention)."""
    return (silu(xs @ Wg.T) * (xs @ Wu.T)) @ Wd.T


def reconstruct(layer: CompressedLayer, experts: Sequence[int]) -> Dict[int, tuple]:
    """{e: expert_weights(layer, e)} for the given experts (step 1 done ahead of
    the forward, so that a timing of the forward can leave it out)."""
    return {int(e): expert_weights(layer, int(e)) for e in np.unique(np.asarray(experts))}


def moe_forward(layer: CompressedLayer, x: np.ndarray, k: Optional[int] = None,
                token_subset: Optional[Sequence[int]] = None, routing=None,
                experts: Optional[Dict[int, tuple]] = None) -> np.ndarray:
    """y [T, H] float64 (or [len(token_subset), H]).

    Routing is decided on all T tokens' canonical logits (only the subset's rows
    are needed, and routing is per token, so only those rows are routed).
    ``experts`` may hold reconstructed weights from ``reconstruct``; an expert
    missing from it is reconstructed here."""
    k = layer.top_k if k is None else k
    toks = np.arange(x.shape[0]) if token_subset is None else np.asarray(token_subset, np.int64)
    xs = x[toks]
    if routing is None:
        ids, g, _ = route(layer, xs, k)
    else:
        ids, g = routing[0][toks], routing[1][toks]
    X = from_storage(xs, layer.dtype)
    n, H = X.shape
    out = np.zeros((n, k, H), np.float64)
    for e in np.unique(ids):
        if experts is not None and int(e) in experts:
            Wg, Wu, Wd = experts[int(e)]
        else:
            Wg, Wu, Wd = expert_weights(layer, int(e))
        rows, slots = np.nonzero(ids == e)
        out[rows, slots] = g[rows, slots][:, None] * expert_output(Wg, Wu, Wd, X[rows])
    y = np.zeros((n, H), np.float64)
    for s in range(k):
        y += out[:, s]
    return y


# ----------------------------------------------------------------------------
# 4. bucketing
# ----------------------------------------------------------------------------
def max_depth(layer: CompressedLayer) -> int:
    return max(len(_path(layer, e)) for e in range(layer.n_experts))


def buckets(layer: CompressedLayer, ids: np.ndarray) -> Dict[str, np.ndarray]:
    """Plain-loop bucketing of the assignments ids [T, k].

    node_off   [n_nodes+1]  exclusive prefix of |T_n|
    node_tok   [sum |T_n|]  tokens of node n ascending, nodes in id order
    node_row   [T*k*D]      row of (t, path(e)[l]) for a = t*k+s, level l; -1 past the path
    expert_off [E+1]        exclusive prefix of the firing counts N_e
    perm       [T*k]        assignment indices a = t*k+s, by (expert, token) ascending
    """
    T, k = ids.shape
    N = layer.n_nodes
    E = layer.n_experts
    D = max_depth(layer)
    paths = [_path(layer, e) for e in range(E)]
    node_tokens: List[List[int]] = [[] for _ in range(N)]
    for t in range(T):
        used = set()
        for s in range(k):
            for n in paths[int(ids[t, s])]:
                used.add(n)
        for n in sorted(used):
            node_tokens[n].append(t)          # t ascending by construction
    node_off = np.zeros(N + 1, np.int32)
    for n in range(N):
        node_off[n + 1] = node_off[n] + len(node_tokens[n])
    node_tok = np.zeros(int(node_off[N]), np.int32)
    where: Dict[tuple, int] = {}
    for n in range(N):
        for i, t in enumerate(node_tokens[n]):
            node_tok[node_off[n] + i] = t
            where[(t, n)] = int(node_off[n]) + i
    node_row = np.full(T * k * D, -1, np.int32)
    for t in range(T):
        for s in range(k):
            for l, n in enumerate(paths[int(ids[t, s])]):
                node_row[(t * k + s) * D + l] = where[(t, n)]
    expert_asg: List[List[int]] = [[] for _ in range(E)]
    for t in range(T):
        for s in range(k):
            expert_asg[int(ids[t, s])].append(t * k + s)
    expert_off = np.zeros(E + 1, np.int32)
    for e in range(E):
        expert_off[e + 1] = expert_off[e] + len(expert_asg[e])
    perm = np.asarray([a for e in range(E) for a in expert_asg[e]], np.int32)
    return dict(node_off=node_off, node_tok=node_tok, node_row=node_row,
                expert_off=expert_off, perm=perm, max_depth=D)
