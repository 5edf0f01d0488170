"""Seeded synthetic workloads for the compressed-MoE forward.

This module only draws random numbers and lays them out; it holds none of the
forward pass's arithmetic.  Both the CPU oracle and the CUDA library consume the
layers and token batches made here, so the two sides always see identical
inputs.

A layer is described by a *node table* (LorExperts Sec. 3.1; BTExperts Sec. 5):

* an **anchor** node (parent -1, rank 0) stores full gate/up/down matrices,
  ``gate, up: [I, H]`` and ``down: [H, I]`` in ``nn.Linear`` ``[out, in]`` order
  (the paper's ``W_e in R^{I x H}``, applied as ``x W^T``, Sec. 2 and 5.1);
* a **correction** node (parent >= 0, rank r > 0) stores, per projection, the
  pair ``U = B_m  [out, r]`` and ``V = A_m^T  [in, r]`` of the paper's
  ``W_m ~ W_dom + B_m A_m`` (Sec. 3.1), in the order
  ``(Ug [I,r], Vg [H,r], Uu [I,r], Vu [H,r], Ud [H,r], Vd [I,r])``;
* ``expert_node[e]`` names the node whose root path defines expert ``e``.

The flat LorExperts layout has one anchor per cluster (the dominant expert maps
to it directly) and one rank-r child per member.  The BTExperts layout used here
has non-expert root anchors, rank-192 sub-dominant children (experts) and rank-64
leaf grandchildren (experts).  Two further layouts: a binary BTExperts tree in the
shape of Fig. 2 (non-expert root and internal corrections, experts at the
leaves, optionally with the figure's -1/+1 edge signs), and a single shared base
(one non-expert anchor, every expert a rank-r correction to it: the
single-shared-component layout the paper contrasts with, Sec. 5.2).

Edge signs: ``node_sign[n]`` in {+1, -1} multiplies correction n's contribution
``U_n V_n^T`` (the label on the edge from n's parent to n in Fig. 2); ``None``
means every edge is +1.  Anchors always carry +1.

Storage dtypes: ``'f32'`` (float32 arrays), ``'bf16'`` (uint16 arrays holding
bfloat16 bit patterns) and ``'f64'`` (float64; accepted by the oracle only, used
by pins that need exact arithmetic).

Routing statistics.  Router rows of experts in one co-activation group share a
common direction (correlation ``rho``), so tokens pick several experts of one
cluster; a per-expert bias ``-beta * s * log(rank)`` over Zipf ranks (the
cluster's dominant holds the cluster's best rank, mirroring the paper's choice of
the highest-firing member as dominant, Sec. 3.2 Stage 2) skews the loads, and a
fixed set of members gets a -4 logit offset so that they are effectively never
routed.  With the default constants the 128-expert layer gives a top-64 visit
share of ~0.949, 25 dead experts and ~3.6 clusters per token, matching the
routing concentration of Table 3 (0.945, 24.6 dead).
"""
from __future__ import annotations

import dataclasses
from typing import List, Optional, Sequence, Tuple

import numpy as np

__all__ = [
    "CompressedLayer", "bf16_bits", "bf16_to_f32", "to_storage", "from_storage",
    "tiny_layer", "flat_layer", "tree_layer", "qwen_decode_layer",
    "qwen_prefill_layer", "high_e_layer", "btexperts_tree_layer", "binary_tree_layer",
    "single_base_layer", "btexperts_binary_layer", "d2moe_base_layer", "tokens", "CONFIGS",
]

ANCHOR_SLOTS = ("gate", "up", "down")
CORR_SLOTS = ("Ug", "Vg", "Uu", "Vu", "Ud", "Vd")


# ----------------------------------------------------------------------------
# bfloat16 storage helpers (bit-pattern conversions only)
# ----------------------------------------------------------------------------
def bf16_bits(a: np.ndarray) -> np.ndarray:
    """Round float32 values to bfloat16 (round-to-nearest-even); return uint16 bits."""
    a = np.ascontiguousarray(a, dtype=np.float32)
    u = a.view(np.uint32)
    # in uint32 (no overflow for any finite or infinite value): t = (u + 0x7FFF
    # + lsb) >> 16, lsb the lowest kept bit, in place to keep it to a few passes
    t = u >> 16
    t &= 1
    t += u
    t += np.uint32(0x7FFF)
    t >>= 16
    return t.astype(np.uint16)


def bf16_to_f32(b: np.ndarray) -> np.ndarray:
    """Exact widening of bfloat16 bit patterns (uint16) to float32."""
    b = np.ascontiguousarray(b, dtype=np.uint16)
    return (b.astype(np.uint32) << 16).view(np.float32)


def to_storage(a: np.ndarray, dtype: str) -> np.ndarray:
    if dtype == "bf16":
        return bf16_bits(a)
    if dtype == "f32":
        return np.ascontiguousarray(a, dtype=np.float32)
    if dtype == "f64":
        return np.ascontiguousarray(a, dtype=np.float64)
    raise ValueError(f"unknown storage dtype {dtype!r}")


def from_storage(a: np.ndarray, dtype: str) -> np.ndarray:
    """Storage array -> float64 (exact)."""
    if dtype == "bf16":
        return bf16_to_f32(a).astype(np.float64)
    return np.asarray(a, dtype=np.float64)


# ----------------------------------------------------------------------------
# layer container
# ----------------------------------------------------------------------------
@dataclasses.dataclass
class CompressedLayer:
    d_model: int
    d_ff: int
    n_experts: int
    dtype: str
    node_parent: np.ndarray          # int32 [n_nodes]
    node_rank: np.ndarray            # int32 [n_nodes]
    expert_node: np.ndarray          # int32 [n_experts]
    node_w: List[Tuple[np.ndarray, ...]]
    router_w: np.ndarray             # [E, H] storage dtype
    router_bias: Optional[np.ndarray]  # float32 [E] or None
    top_k: int
    name: str = ""
    meta: dict = dataclasses.field(default_factory=dict)
    node_sign: Optional[np.ndarray] = None   # int8 [n_nodes] of +1/-1, or None (all +1)

    @property
    def n_nodes(self) -> int:
        return int(self.node_parent.shape[0])

    def is_anchor(self, n: int) -> bool:
        return int(self.node_parent[n]) < 0

    def path(self, e: int) -> List[int]:
        """Nodes from expert e's own node up to its anchor (inclusive)."""
        out = []
        n = int(self.expert_node[e])
        while n >= 0:
            out.append(n)
            n = int(self.node_parent[n])
        return out

    def weight_bytes(self) -> int:
        return int(sum(a.nbytes for w in self.node_w for a in w))


# ----------------------------------------------------------------------------
# drawing helpers
# ----------------------------------------------------------------------------
def _normal(rng: np.random.Generator, shape, std: float) -> np.ndarray:
    return (rng.standard_normal(shape, dtype=np.float32) * np.float32(std))


def _router(rng, E: int, H: int, groups: Sequence[Sequence[int]], rho: float,
            outer: Optional[Sequence[Sequence[int]]] = None, rho_outer: float = 0.0,
            std: float = 0.02) -> np.ndarray:
    """Router rows N(0, std^2) marginally; rows in one group share a direction."""
    W = _normal(rng, (E, H), std) * np.float32(np.sqrt(max(0.0, 1.0 - rho - rho_outer)))
    for g in groups:
        u = _normal(rng, (H,), std) * np.float32(np.sqrt(rho))
        W[list(g)] += u
    if outer is not None:
        for g in outer:
            u = _normal(rng, (H,), std) * np.float32(np.sqrt(rho_outer))
            W[list(g)] += u
    return W


def _zipf_bias(rng, E: int, groups: Sequence[Sequence[int]], s: float, beta: float,
               dead: Sequence[int]) -> np.ndarray:
    """Per-expert logit bias -beta*s*log(rank); groups get consecutive ranks in a
    seeded popularity order and each group's first expert its best rank."""
    order = rng.permutation(len(groups))
    ranks = np.zeros(E, np.float64)
    base = 0
    pos = np.empty(len(groups), np.int64)
    pos[order] = np.arange(len(groups))
    starts = np.cumsum([0] + [len(groups[g]) for g in order])
    for gi, g in enumerate(groups):
        base = starts[pos[gi]]
        for j, e in enumerate(g):
            ranks[e] = base + j + 1
    b = -beta * s * np.log(ranks)
    b[list(dead)] -= 4.0
    return b.astype(np.float32)


def _n_dead(n_dead: int, n_candidates: int) -> int:
    """Dead experts of a skewed router: the calibrated count (25 of the 96
    members of E = 128, Table 3), but at most a third of the candidates, so
    that a small test layer keeps members the router can select."""
    return min(n_dead, n_candidates // 3)


def _factor_std(rank: int, factor_std) -> float:
    if factor_std is None:
        return 0.02 / np.sqrt(rank)            # "N(0, 0.02/sqrt(r))" read as std
    if factor_std == "visible":
        return float(np.sqrt(0.02) / rank ** 0.25)   # U V^T entries ~ N(0, 0.02^2)
    return float(factor_std)


def _corr_factors(rng, H, I, r, std, dtype, zero=False):
    # always draw, so that zeroed variants keep the same random stream
    shapes = [(I, r), (H, r), (I, r), (H, r), (H, r), (I, r)]
    ws = [_normal(rng, s, std) for s in shapes]
    return tuple(to_storage(w * np.float32(0.0 if zero else 1.0), dtype) for w in ws)


def _anchor(rng, H, I, dtype, std=0.02, zero=False):
    shapes = [(I, H), (I, H), (H, I)]
    ws = [_normal(rng, s, std) for s in shapes]
    return tuple(to_storage(w * np.float32(0.0 if zero else 1.0), dtype) for w in ws)


# ----------------------------------------------------------------------------
# flat LorExperts layer (Sec. 3.1): one dominant + members per cluster
# ----------------------------------------------------------------------------
def flat_layer(H: int, I: int, cluster_sizes: Sequence[int], rank, top_k: int,
               dtype: str = "bf16", seed: int = 0, factor_std=None,
               zero_dominants: bool = False, zero_factors: bool = False,
               skew: Optional[Tuple[float, float, float, int]] = None,
               shuffle_experts: bool = True, name: str = "flat") -> CompressedLayer:
    """Flat layer.  ``cluster_sizes[c]`` experts in cluster c (size 1 = a
    protection-set singleton: an anchor with no children).  ``rank`` is an int or
    a per-member sequence.  ``skew = (s, beta, rho, n_dead)`` enables the Zipf /
    co-activation router; ``None`` gives a plain N(0, 0.02) router."""
    rng = np.random.default_rng(seed)
    E = int(sum(cluster_sizes))
    C = len(cluster_sizes)
    ids = rng.permutation(E) if shuffle_experts else np.arange(E)
    groups, pos = [], 0
    for m in cluster_sizes:
        groups.append([int(e) for e in ids[pos:pos + m]])
        pos += m
    n_members = E - C
    ranks = list(rank) if isinstance(rank, (list, tuple, np.ndarray)) else [int(rank)] * n_members
    assert len(ranks) == n_members
    parent = [-1] * C
    nrank = [0] * C
    expert_node = np.zeros(E, np.int32)
    node_w = [_anchor(rng, H, I, dtype, zero=zero_dominants) for _ in range(C)]
    mi = 0
    for c, g in enumerate(groups):
        expert_node[g[0]] = c
        for e in g[1:]:
            r = ranks[mi]
            mi += 1
            parent.append(c)
            nrank.append(r)
            expert_node[e] = len(parent) - 1
            node_w.append(_corr_factors(rng, H, I, r, _factor_std(r, factor_std), dtype,
                                        zero=zero_factors))
    if skew is None:
        Wr = _normal(rng, (E, H), 0.02)
        bias = None
    else:
        s, beta, rho, n_dead = skew
        Wr = _router(rng, E, H, groups, rho)
        members = [e for g in groups for e in g[1:]]
        dead = rng.choice(members, size=_n_dead(n_dead, len(members)), replace=False) if n_dead else []
        bias = _zipf_bias(rng, E, groups, s, beta, dead)
    return CompressedLayer(
        d_model=H, d_ff=I, n_experts=E, dtype=dtype,
        node_parent=np.asarray(parent, np.int32), node_rank=np.asarray(nrank, np.int32),
        expert_node=expert_node, node_w=node_w, router_w=to_storage(Wr, dtype),
        router_bias=bias, top_k=top_k, name=name,
        meta={"clusters": groups, "seed": seed})


# ----------------------------------------------------------------------------
# BTExperts depth-2 tree (Sec. 5, Fig. 2): root anchors, sub-dominant and leaf
# corrections.  Roots are not experts.
# ----------------------------------------------------------------------------
def tree_layer(H: int, I: int, n_roots: int, subs_per_root: int, leaves_per_sub: int,
               r_sub: int, r_leaf: int, top_k: int, dtype: str = "bf16", seed: int = 0,
               factor_std=None, zero_dominants: bool = False, zero_factors: bool = False,
               skew: Optional[Tuple[float, float, float, int]] = None,
               name: str = "tree") -> CompressedLayer:
    rng = np.random.default_rng(seed)
    n_subs = n_roots * subs_per_root
    n_leaves = n_subs * leaves_per_sub
    E = n_subs + n_leaves
    ids = [int(e) for e in rng.permutation(E)]
    parent = [-1] * n_roots
    nrank = [0] * n_roots
    node_w = [_anchor(rng, H, I, dtype, zero=zero_dominants) for _ in range(n_roots)]
    expert_node = np.zeros(E, np.int32)
    sub_groups, root_groups = [], [[] for _ in range(n_roots)]
    it = iter(ids)
    sub_nodes = []
    for rt in range(n_roots):
        for _ in range(subs_per_root):
            parent.append(rt)
            nrank.append(r_sub)
            node_w.append(_corr_factors(rng, H, I, r_sub, _factor_std(r_sub, factor_std),
                                        dtype, zero=zero_factors))
            sn = len(parent) - 1
            sub_nodes.append(sn)
            e = next(it)
            expert_node[e] = sn
            sub_groups.append([e])
            root_groups[rt].append(e)
    for si, sn in enumerate(sub_nodes):
        rt = parent[sn]
        for _ in range(leaves_per_sub):
            parent.append(sn)
            nrank.append(r_leaf)
            node_w.append(_corr_factors(rng, H, I, r_leaf, _factor_std(r_leaf, factor_std),
                                        dtype, zero=zero_factors))
            e = next(it)
            expert_node[e] = len(parent) - 1
            sub_groups[si].append(e)
            root_groups[rt].append(e)
    if skew is None:
        Wr = _normal(rng, (E, H), 0.02)
        bias = None
    else:
        s, beta, rho, n_dead = skew
        Wr = _router(rng, E, H, sub_groups, rho * 0.5, outer=root_groups, rho_outer=rho * 0.45)
        leaves = [e for g in sub_groups for e in g[1:]]
        dead = rng.choice(leaves, size=_n_dead(n_dead, len(leaves)), replace=False) if n_dead else []
        bias = _zipf_bias(rng, E, sub_groups, s, beta, dead)
    return CompressedLayer(
        d_model=H, d_ff=I, n_experts=E, dtype=dtype,
        node_parent=np.asarray(parent, np.int32), node_rank=np.asarray(nrank, np.int32),
        expert_node=expert_node, node_w=node_w, router_w=to_storage(Wr, dtype),
        router_bias=bias, top_k=top_k, name=name,
        meta={"subs": sub_groups, "roots": root_groups, "seed": seed})


# ----------------------------------------------------------------------------
# BTExperts binary tree (Fig. 2): per root anchor a complete binary tree of
# corrections; internal corrections are shared, the leaves are the experts.
# ----------------------------------------------------------------------------
def binary_tree_layer(H: int, I: int, n_roots: int, levels: int, ranks: Sequence[int],
                      top_k: int, dtype: str = "bf16", seed: int = 0, factor_std=None,
                      signed: bool = False, zero_dominants: bool = False,
                      zero_factors: bool = False,
                      skew: Optional[Tuple[float, float, float, int]] = None,
                      name: str = "binary-tree") -> CompressedLayer:
    """``levels`` correction levels below each root (level 1 has 2 nodes, level
    ``levels`` has 2**levels leaves, the experts); ``ranks[l-1]`` is the rank of
    level l.  ``signed`` labels the edge to every left child -1 and to every
    right child +1, as Fig. 2 does for the internal levels (the figure gives the
    leaf edges no label; here they carry the same alternation)."""
    assert 1 <= levels and len(ranks) == levels
    rng = np.random.default_rng(seed)
    leaves_per_root = 2 ** levels
    E = n_roots * leaves_per_root
    ids = [int(e) for e in rng.permutation(E)]
    parent = [-1] * n_roots
    nrank = [0] * n_roots
    sign = [1] * n_roots
    node_w = [_anchor(rng, H, I, dtype, zero=zero_dominants) for _ in range(n_roots)]
    expert_node = np.zeros(E, np.int32)
    it = iter(ids)
    root_groups, pair_groups = [], []
    for rt in range(n_roots):
        frontier = [rt]
        for lev in range(1, levels + 1):
            nxt = []
            for pn in frontier:
                for side in (0, 1):
                    parent.append(pn)
                    r = int(ranks[lev - 1])
                    nrank.append(r)
                    sign.append((-1 if side == 0 else 1) if signed else 1)
                    node_w.append(_corr_factors(rng, H, I, r, _factor_std(r, factor_std),
                                                dtype, zero=zero_factors))
                    nxt.append(len(parent) - 1)
            frontier = nxt
        leaves = []
        for ln in frontier:
            e = next(it)
            expert_node[e] = ln
            leaves.append(e)
        root_groups.append(leaves)
        # co-activation groups: the leaves below each level-(levels-1) node
        # (pairs of siblings; the whole root's leaves when levels == 1)
        step = 2 if levels > 1 else leaves_per_root
        for j in range(0, leaves_per_root, step):
            pair_groups.append(leaves[j:j + step])
    if skew is None:
        Wr = _normal(rng, (E, H), 0.02)
        bias = None
    else:
        s, beta, rho, n_dead = skew
        Wr = _router(rng, E, H, pair_groups, rho * 0.5, outer=root_groups, rho_outer=rho * 0.45)
        cand = [e for g in pair_groups for e in g[1:]]
        dead = rng.choice(cand, size=_n_dead(n_dead, len(cand)), replace=False) if n_dead else []
        bias = _zipf_bias(rng, E, pair_groups, s, beta, dead)
    return CompressedLayer(
        d_model=H, d_ff=I, n_experts=E, dtype=dtype,
        node_parent=np.asarray(parent, np.int32), node_rank=np.asarray(nrank, np.int32),
        expert_node=expert_node, node_w=node_w, router_w=to_storage(Wr, dtype),
        router_bias=bias, top_k=top_k, name=name,
        meta={"roots": root_groups, "pairs": pair_groups, "seed": seed},
        node_sign=np.asarray(sign, np.int8) if signed else None)


# ----------------------------------------------------------------------------
# single shared base: one non-expert anchor, every expert a rank-r correction
# ----------------------------------------------------------------------------
def single_base_layer(H: int, I: int, E: int, rank, top_k: int, dtype: str = "bf16",
                      seed: int = 0, factor_std=None, group: int = 4,
                      zero_dominants: bool = False, zero_factors: bool = False,
                      skew: Optional[Tuple[float, float, float, int]] = None,
                      name: str = "single-base") -> CompressedLayer:
    """One shared base anchor (not an expert) and E rank-r experts below it.
    Router co-activation groups of ``group`` consecutive shuffled experts."""
    rng = np.random.default_rng(seed)
    ids = [int(e) for e in rng.permutation(E)]
    ranks = list(rank) if isinstance(rank, (list, tuple, np.ndarray)) else [int(rank)] * E
    parent, nrank = [-1], [0]
    node_w = [_anchor(rng, H, I, dtype, zero=zero_dominants)]
    expert_node = np.zeros(E, np.int32)
    for j, e in enumerate(ids):
        r = int(ranks[j])
        parent.append(0)
        nrank.append(r)
        node_w.append(_corr_factors(rng, H, I, r, _factor_std(r, factor_std), dtype,
                                    zero=zero_factors))
        expert_node[e] = len(parent) - 1
    groups = [ids[j:j + group] for j in range(0, E, group)]
    if skew is None:
        Wr = _normal(rng, (E, H), 0.02)
        bias = None
    else:
        s, beta, rho, n_dead = skew
        Wr = _router(rng, E, H, groups, rho)
        cand = [e for g in groups for e in g[1:]]
        dead = rng.choice(cand, size=_n_dead(n_dead, len(cand)), replace=False) if n_dead else []
        bias = _zipf_bias(rng, E, groups, s, beta, dead)
    return CompressedLayer(
        d_model=H, d_ff=I, n_experts=E, dtype=dtype,
        node_parent=np.asarray(parent, np.int32), node_rank=np.asarray(nrank, np.int32),
        expert_node=expert_node, node_w=node_w, router_w=to_storage(Wr, dtype),
        router_bias=bias, top_k=top_k, name=name, meta={"groups": groups, "seed": seed})


# ----------------------------------------------------------------------------
# the five workloads
# ----------------------------------------------------------------------------
def _svd_factors(R: np.ndarray, r: int):
    """Rank-r truncated SVD of R with the symmetric singular-value split of
    Eq. (factors): B = U_r S^1/2, A = S^1/2 V_r^T.  Returns (B [out,r], A^T [in,r]).
    Sign convention: the largest-magnitude entry of each left singular vector is
    positive.  (Input construction for the tiny workload; the forward never
    factorises anything.)"""
    U, S, Vt = np.linalg.svd(R.astype(np.float64), full_matrices=False)
    U, S, Vt = U[:, :r], S[:r], Vt[:r]
    sgn = np.sign(U[np.argmax(np.abs(U), axis=0), np.arange(r)])
    sgn[sgn == 0] = 1.0
    U = U * sgn
    Vt = Vt * sgn[:, None]
    sq = np.sqrt(S)
    return U * sq, (Vt.T * sq)


def tiny_layer(seed: int = 0, rank: int = 8, dtype: str = "f32", H: int = 64, I: int = 128,
               clusters: int = 2, cluster_size: int = 4, top_k: int = 2,
               return_dense: bool = False):
    """Tiny fp32 LorExperts layer: members' corrections are the exact rank-``rank``
    truncated SVD of (independent N(0, 0.02) expert - dominant), per projection.

    With ``return_dense`` also returns the uncompressed expert weights
    ``dense[e] = (gate, up, down)`` as float64 (the matrices the factors
    approximate; exact at full rank)."""
    rng = np.random.default_rng(seed)
    E = clusters * cluster_size
    dense = [tuple(_normal(rng, s, 0.02).astype(np.float64)
                   for s in [(I, H), (I, H), (H, I)]) for _ in range(E)]
    parent, nrank, node_w = [], [], []
    expert_node = np.zeros(E, np.int32)
    for c in range(clusters):
        parent.append(-1)
        nrank.append(0)
        dom = c * cluster_size
        node_w.append(tuple(to_storage(w, dtype) for w in dense[dom]))
        expert_node[dom] = len(parent) - 1
    for c in range(clusters):
        dom = c * cluster_size
        domw = [from_storage(w, dtype) for w in node_w[c]]
        for e in range(dom + 1, dom + cluster_size):
            fac = []
            for p in range(3):
                B, At = _svd_factors(dense[e][p] - domw[p], rank)
                fac += [B, At]
            parent.append(c)
            nrank.append(rank)
            expert_node[e] = len(parent) - 1
            node_w.append(tuple(to_storage(f, dtype) for f in fac))
    Wr = _normal(rng, (E, H), 0.02)
    layer = CompressedLayer(
        d_model=H, d_ff=I, n_experts=E, dtype=dtype,
        node_parent=np.asarray(parent, np.int32), node_rank=np.asarray(nrank, np.int32),
        expert_node=expert_node, node_w=node_w, router_w=to_storage(Wr, dtype),
        router_bias=None, top_k=top_k, name="tiny",
        meta={"clusters": [list(range(c * cluster_size, (c + 1) * cluster_size))
                           for c in range(clusters)], "seed": seed})
    if return_dense:
        return layer, dense
    return layer


QWEN_SKEW = (1.1, 0.6, 0.95, 25)
HIGH_E_SKEW = (1.2, 0.5, 0.95, 50)
TREE_SKEW = (1.1, 0.6, 0.95, 25)


def qwen_decode_layer(seed: int = 2, factor_std=None, **kw) -> CompressedLayer:
    """Qwen3-30B-A3B-shaped layer: H=2048, I=768, E=128 top-8, 32 clusters of 4,
    rank-128 members, bf16, Zipf(1.1) loads with in-cluster co-activation."""
    return flat_layer(2048, 768, [4] * 32, 128, 8, "bf16", seed, factor_std,
                      skew=QWEN_SKEW, name="qwen3-30b-a3b-layer", **kw)


def qwen_prefill_layer(seed: int = 3, factor_std=None, **kw) -> CompressedLayer:
    return flat_layer(2048, 768, [4] * 32, 128, 8, "bf16", seed, factor_std,
                      skew=QWEN_SKEW, name="qwen3-30b-a3b-layer", **kw)


def high_e_layer(seed: int = 4, factor_std=None, **kw) -> CompressedLayer:
    """H=2560, I=1536, E=256 top-8, 32 clusters of 8, rank-64 members, Zipf(1.2)."""
    return flat_layer(2560, 1536, [8] * 32, 64, 8, "bf16", seed, factor_std,
                      skew=HIGH_E_SKEW, name="high-e-layer", **kw)


def btexperts_tree_layer(seed: int = 5, factor_std=None, **kw) -> CompressedLayer:
    """H=2048, I=768, 8 root anchors x 4 rank-192 sub-dominants x 3 rank-64 leaves."""
    return tree_layer(2048, 768, 8, 4, 3, 192, 64, 8, "bf16", seed, factor_std,
                      skew=TREE_SKEW, name="btexperts-tree-layer", **kw)


def btexperts_binary_layer(seed: int = 6, factor_std=None, signed: bool = True,
                           **kw) -> CompressedLayer:
    """H=2048, I=768, E=128 top-8: 16 root anchors, each a Fig. 2 binary tree of
    rank-128 / rank-64 internal corrections and rank-64 leaf experts (8 per root,
    root paths of 4 nodes), edge signs -1/+1."""
    return binary_tree_layer(2048, 768, 16, 3, [128, 64, 64], 8, "bf16", seed, factor_std,
                             signed=signed, skew=TREE_SKEW, name="btexperts-binary-layer",
                             **kw)


def d2moe_base_layer(seed: int = 7, factor_std=None, **kw) -> CompressedLayer:
    """H=2048, I=768, E=128 top-8 rank-128 experts over one shared base."""
    return single_base_layer(2048, 768, 128, 128, 8, "bf16", seed, factor_std,
                             skew=QWEN_SKEW, name="single-base-layer", **kw)


def tokens(layer: CompressedLayer, T: int, seed: int = 0) -> np.ndarray:
    """x ~ N(0, 1), [T, H], in the layer's storage dtype."""
    rng = np.random.default_rng(10_000 + seed)
    return to_storage(rng.standard_normal((T, layer.d_model), dtype=np.float32), layer.dtype)


CONFIGS = {
    1: dict(name="tiny-fp32", make=tiny_layer, T=256),
    2: dict(name="qwen3-decode", make=qwen_decode_layer, T=(1, 8, 32, 64)),
    3: dict(name="qwen3-prefill", make=qwen_prefill_layer, T=8192),
    4: dict(name="high-e", make=high_e_layer, T=4096),
    5: dict(name="btexperts-tree", make=btexperts_tree_layer, T=2048),
}
