"""GPU parity of liblx against the CPU oracle, through the C ABI.

Bar (per output tensor): routing ids, bucketing and permutation bit-exact;
router logits bit-exact (same canonical fp32 order on both sides); gates within
1e-6; y within max|y - y_ref| / max|y_ref| <= 2e-2 for bf16 layers and 1e-5 for
fp32 layers.  Sizes span several GEMM tiles with ragged tails; the full-size
workloads are checked on sampled tokens (the oracle is per token) plus bit-exact
routing and bucketing of every token.
"""
import numpy as np
import pytest
import torch

import oracle
import synth
from paper_2608_07814_gb300 import lx

pytestmark = pytest.mark.gpu

TOL = {"bf16": 2e-2, "f32": 1e-5}


def _dev(a, dtype):
    return lx.host_to_torch(a, dtype).cuda()


def _rel(y, ref):
    return float(np.max(np.abs(y - ref)) / max(np.max(np.abs(ref)), 1e-30))


def elementwise(y, ref):
    """Element-wise relative error |y - ref| / max(|ref|, 1e-3 rms(ref)): its
    median, 99th percentile and maximum.  A diagnostic beside the per-tensor
    bar: a wrong small-magnitude element shows here and not there."""
    floor = 1e-3 * float(np.sqrt(np.mean(ref ** 2))) if ref.size else 0.0
    e = np.abs(y - ref) / np.maximum(np.abs(ref), max(floor, 1e-30))
    if e.size == 0:
        return dict(p50=0.0, p99=0.0, max=0.0)
    return dict(p50=float(np.median(e)), p99=float(np.quantile(e, 0.99)), max=float(e.max()))


# element-wise diagnostics of every forward checked in this session (printed
# at the end of the run by the terminal-summary hook in conftest.py)
DIAG = []


def _y_host(y):
    return y.float().cpu().numpy().astype(np.float64)


_cache = {}


def installed(key, make):
    """(synth layer, lx.Layer) cached per test session."""
    if key not in _cache:
        src = make()
        _cache[key] = (src, lx.Layer(src))
    return _cache[key]


def check_route(src, L, x, k):
    xd = _dev(x, src.dtype)
    ids, w, logits = L.route(xd, k, want_logits=True)
    torch.cuda.synchronize()
    o_ids, o_g, o_l = oracle.route(src, x, k)
    assert np.array_equal(logits.cpu().numpy(), o_l), "logits not bit-exact"
    assert np.array_equal(ids.cpu().numpy(), o_ids), "top-k ids not bit-exact"
    assert np.max(np.abs(w.cpu().numpy() - o_g)) < 1e-6
    return o_ids, o_g


def check_buckets(src, L, ids_host):
    L.bucket(torch.from_numpy(ids_host).cuda())
    b = L.get_buckets()
    torch.cuda.synchronize()
    ref = oracle.buckets(src, ids_host)
    for key in ("node_off", "node_tok", "node_row", "expert_off", "perm"):
        got = b[key].cpu().numpy()
        assert np.array_equal(got, ref[key]), key


def check_forward(src, L, x, k, sample=None, path=lx.LX_PATH_AUTO, tol=None):
    L.set_path(path)
    xd = _dev(x, src.dtype)
    y = L.moe_forward(xd, k)
    torch.cuda.synchronize()
    yh = _y_host(y)
    toks = np.arange(x.shape[0]) if sample is None else np.asarray(sample)
    ref = oracle.moe_forward(src, x, k, token_subset=toks)
    err = _rel(yh[toks], ref)
    ew = elementwise(yh[toks], ref)
    DIAG.append((f"H={src.d_model} I={src.d_ff} E={src.n_experts} N={src.n_nodes} "
                 f"T={x.shape[0]} k={k} path={path}", err, ew))
    assert L.info()["device_error"] == 0
    assert np.all(np.isfinite(yh))
    bar = tol or TOL[src.dtype]
    assert err <= bar, f"rel err {err}"
    # the typical element meets the same bar element-wise
    assert ew["p50"] <= bar, f"element-wise median rel err {ew['p50']}"
    return err


# ----------------------------------------------------------------------------
# small layers: every output element
# ----------------------------------------------------------------------------
SMALL = {
    "tiny_fp32": lambda: synth.tiny_layer(seed=0),
    "tiny_fp32_fullrank": lambda: synth.tiny_layer(seed=1, rank=64),
    "flat_bf16_visible": lambda: synth.flat_layer(512, 384, [4] * 8, 32, 8, "bf16", seed=3,
                                                  factor_std="visible", skew=synth.QWEN_SKEW),
    "flat_bf16_zero_dom": lambda: synth.flat_layer(512, 384, [4] * 8, 32, 8, "bf16", seed=3,
                                                   factor_std="visible", zero_dominants=True,
                                                   skew=synth.QWEN_SKEW),
    "flat_bf16_zero_fac": lambda: synth.flat_layer(512, 384, [4] * 8, 32, 8, "bf16", seed=3,
                                                   zero_factors=True, skew=synth.QWEN_SKEW),
    "flat_fp32_singletons": lambda: synth.flat_layer(136, 72, [1, 3, 1, 5, 1, 2, 1], 24, 3,
                                                     "f32", seed=5, factor_std="visible"),
    "flat_fp32_mixed_rank": lambda: synth.flat_layer(64, 96, [4, 4, 4], [8, 16, 24, 40, 8, 64,
                                                                         1, 2, 3], 4, "f32",
                                                     seed=6, factor_std="visible"),
    "tree_bf16": lambda: synth.tree_layer(256, 192, 2, 4, 3, 48, 16, 8, "bf16", seed=7,
                                          factor_std="visible", skew=synth.TREE_SKEW),
    "tree_fp32": lambda: synth.tree_layer(128, 64, 2, 2, 3, 24, 8, 4, "f32", seed=8,
                                          factor_std="visible", skew=synth.TREE_SKEW),
    # served by the weight-streaming (TMA) kernels: dims and ranks multiples of 64
    "stream_flat": lambda: synth.flat_layer(512, 384, [4] * 8, 64, 8, "bf16", seed=13,
                                            factor_std="visible", skew=synth.QWEN_SKEW),
    "stream_flat_zero_dom": lambda: synth.flat_layer(512, 384, [4] * 8, 64, 8, "bf16", seed=13,
                                                     factor_std="visible", zero_dominants=True,
                                                     skew=synth.QWEN_SKEW),
    "stream_flat_zero_fac": lambda: synth.flat_layer(512, 384, [4] * 8, 64, 8, "bf16", seed=13,
                                                     zero_factors=True, skew=synth.QWEN_SKEW),
    "stream_singletons_mixed": lambda: synth.flat_layer(320, 448, [1, 3, 1, 5, 2], [64, 128, 192,
                                                        64, 64, 128, 192], 3, "bf16",
                                                        seed=14, factor_std="visible"),
    "stream_tree": lambda: synth.tree_layer(256, 192, 2, 4, 3, 128, 64, 8, "bf16", seed=15,
                                            factor_std="visible", skew=synth.TREE_SKEW),
    # K long enough for split-K anchor tiles on the streaming path (ragged last split)
    "stream_split_ragged": lambda: synth.flat_layer(1088, 448, [4] * 4, 64, 4, "bf16", seed=16,
                                                    factor_std="visible", skew=synth.QWEN_SKEW),
    "stream_split_tree": lambda: synth.tree_layer(1024, 640, 2, 4, 3, 128, 64, 8, "bf16",
                                                  seed=17, factor_std="visible",
                                                  skew=synth.TREE_SKEW),
    # Fig. 2 binary trees with -1/+1 edges (root paths of four nodes: k * depth = 32)
    "stream_binary_signed": lambda: synth.binary_tree_layer(
        256, 192, 2, 3, [128, 64, 64], 8, "bf16", seed=18, factor_std="visible", signed=True,
        skew=synth.TREE_SKEW),
    "binary_signed_fp32": lambda: synth.binary_tree_layer(
        128, 64, 2, 3, [16, 8, 8], 4, "f32", seed=19, factor_std="visible", signed=True,
        skew=synth.TREE_SKEW),
    # one shared base below which every expert is a correction
    "stream_single_base": lambda: synth.single_base_layer(
        512, 384, 24, 64, 8, "bf16", seed=20, factor_std="visible", skew=synth.QWEN_SKEW),
    "single_base_fp32_mixed_rank": lambda: synth.single_base_layer(
        64, 96, 12, [8, 16, 24, 40, 8, 64, 1, 2, 3, 5, 7, 9], 4, "f32", seed=21,
        factor_std="visible"),
}

STREAM = [n for n in SMALL if n.startswith("stream")]


@pytest.mark.parametrize("name", sorted(SMALL))
@pytest.mark.parametrize("T", [1, 37, 200])
def test_small_route_bucket_forward(name, T):
    src, L = installed(name, SMALL[name])
    x = synth.tokens(src, T, seed=T)
    ids, _ = check_route(src, L, x, src.top_k)
    check_buckets(src, L, ids)
    check_forward(src, L, x, src.top_k)
    check_forward(src, L, x, src.top_k, path=lx.LX_PATH_GENERIC)


@pytest.mark.parametrize("name", STREAM)
def test_stream_path_serves_layer(name):
    src, L = installed(name, SMALL[name])
    assert L.info()["stream_path"] == 1


@pytest.mark.parametrize("name", STREAM)
@pytest.mark.parametrize("T", [1, 37, 200, 256])
def test_forward_buckets(name, T):
    """The bucketing a streaming forward runs (fused with the router for small
    batches) is bit-exact too: read back after the forward."""
    src, L = installed(name, SMALL[name])
    x = synth.tokens(src, T, seed=900 + T)
    check_forward(src, L, x, src.top_k)
    b = L.get_buckets()
    torch.cuda.synchronize()
    o_ids, _, _ = oracle.route(src, x, src.top_k)
    ref = oracle.buckets(src, o_ids)
    for key in ("node_off", "node_tok", "node_row", "expert_off", "perm"):
        assert np.array_equal(b[key].cpu().numpy(), ref[key]), key


@pytest.mark.parametrize("T", [64, 256, 257])
def test_stream_generic_boundary(T):
    src, L = installed("stream_flat", SMALL["stream_flat"])
    x = synth.tokens(src, T, seed=300 + T)
    ids, _ = check_route(src, L, x, src.top_k)
    check_buckets(src, L, ids)
    check_forward(src, L, x, src.top_k)


@pytest.mark.parametrize("name", STREAM)
@pytest.mark.parametrize("T", [300, 1031])
def test_tensor_core_path(name, T):
    """Batches above the streaming limit run on the tcgen05 kernels."""
    src, L = installed(name, SMALL[name])
    x = synth.tokens(src, T, seed=500 + T)
    ids, _ = check_route(src, L, x, src.top_k)
    check_buckets(src, L, ids)
    check_forward(src, L, x, src.top_k)


BF16_SMALL = [n for n in sorted(SMALL) if "fp32" not in n]


@pytest.mark.parametrize("name", BF16_SMALL)
@pytest.mark.parametrize("T", [1217, 2003])
def test_router_large_batch(name, T):
    """Batches of >= 152 8-token tiles take the register-tiled router: logits,
    top-k and gates stay bit-exact (ragged expert groups and chunk counts)."""
    src, L = installed(name, SMALL[name])
    x = synth.tokens(src, T, seed=700 + T)
    ids, _ = check_route(src, L, x, src.top_k)
    check_buckets(src, L, ids)


def test_tensor_core_one_cluster_many_token_blocks():
    """Every token on one cluster: each node bucket spans several 128-row blocks."""
    src = synth.flat_layer(256, 128, [4] * 4, 64, 4, "bf16", seed=12, factor_std="visible")
    src.router_bias = np.zeros(16, np.float32)
    src.router_bias[src.meta["clusters"][1]] = 50.0
    L = lx.Layer(src)
    x = synth.tokens(src, 700, seed=4)
    ids, _ = check_route(src, L, x, 4)
    check_buckets(src, L, ids)
    check_forward(src, L, x, 4)


def test_tiny_fp32_config_full():
    """The tiny fp32 workload: 256 tokens, top-2, rank-8 SVD members."""
    src, L = installed("tiny_fp32", SMALL["tiny_fp32"])
    x = synth.tokens(src, 256, seed=0)
    check_route(src, L, x, 2)
    check_forward(src, L, x, 2)


@pytest.mark.parametrize("name", ["flat_bf16_visible", "stream_flat"])
@pytest.mark.parametrize("k", [1, 3, 8])
def test_other_k(name, k):
    src, L = installed(name, SMALL[name])
    x = synth.tokens(src, 64, seed=100 + k)
    check_route(src, L, x, k)
    check_forward(src, L, x, k)


def test_ties_go_to_lower_id():
    src = synth.flat_layer(64, 32, [4, 4], 8, 3, "f32", seed=9)
    src.router_w[5] = src.router_w[2]      # experts 2 and 5 tie on every token
    src.router_w[7] = src.router_w[2]
    L = lx.Layer(src)
    x = synth.tokens(src, 50, seed=1)
    ids, _ = check_route(src, L, x, 3)
    for row in ids:
        if 2 in row or 5 in row or 7 in row:
            pos = {e: list(row).index(e) for e in (2, 5, 7) if e in row}
            assert sorted(pos, key=pos.get) == sorted(pos)


@pytest.mark.parametrize("T", [70, 255, 256])
def test_all_tokens_on_one_cluster(T):
    """Every token on one cluster of a streaming-capable layer: each of its
    nodes' buckets spans up to the largest number of 32-token work items the
    streaming path takes (8 at 256 tokens, one ragged at 255)."""
    src = synth.flat_layer(256, 128, [4] * 4, 64, 4, "bf16", seed=10, factor_std="visible")
    src.router_bias = np.zeros(16, np.float32)
    src.router_bias[src.meta["clusters"][2]] = 50.0
    L = lx.Layer(src)
    assert L.info()["stream_path"] == 1
    x = synth.tokens(src, T, seed=2)
    ids, _ = check_route(src, L, x, 4)
    assert set(np.unique(ids)) == set(src.meta["clusters"][2])
    check_buckets(src, L, ids)
    check_forward(src, L, x, 4)
    assert L.info()["device_error"] == 0


def test_zero_tokens_is_noop():
    src, L = installed("tiny_fp32", SMALL["tiny_fp32"])
    x = torch.empty((0, src.d_model), dtype=torch.float32, device="cuda")
    y = L.moe_forward(x, 2)
    assert y.shape == (0, src.d_model)


def test_call_errors():
    src, L = installed("tiny_fp32", SMALL["tiny_fp32"])
    x = _dev(synth.tokens(src, 4), "f32")
    with pytest.raises(lx.LxError) as e:
        L.moe_forward(x, src.n_experts + 1)
    assert e.value.status == lx.LX_ERR_ARG
    with pytest.raises(lx.LxError) as e:
        L.moe_forward(x, 0)
    assert e.value.status == lx.LX_ERR_ARG
    big = torch.zeros(4 * 64 + 1, dtype=torch.float32, device="cuda")
    with pytest.raises(lx.LxError) as e:
        L.moe_forward(big[1:].view(4, 64), 2)      # misaligned x
    assert e.value.status == lx.LX_ERR_ARG
    with pytest.raises(lx.LxError) as e:
        L.moe_forward(x, 2, y=x)                   # aliasing
    assert e.value.status == lx.LX_ERR_ARG
    ybig = torch.zeros(4 * 64 + 1, dtype=torch.float32, device="cuda")
    with pytest.raises(lx.LxError) as e:
        L.moe_forward(x, 2, y=ybig[1:].view(4, 64))  # misaligned y
    assert e.value.status == lx.LX_ERR_ARG
    xy = torch.zeros(8 * 64, dtype=torch.float32, device="cuda")
    with pytest.raises(lx.LxError) as e:
        L.moe_forward(xy[:4 * 64].view(4, 64), 2, y=xy[2 * 64:6 * 64].view(4, 64))  # overlap
    assert e.value.status == lx.LX_ERR_ARG


# ----------------------------------------------------------------------------
# full-size workloads
# ----------------------------------------------------------------------------
FULL = {
    "qwen": lambda: synth.qwen_decode_layer(),
    "qwen_visible": lambda: synth.qwen_decode_layer(factor_std="visible"),
    # dominants zeroed: the output is the pure correction path (rank-128 x V and
    # P U^T at K = 2048, z Vd and Q Ud^T at K = 768)
    "qwen_zero_dom": lambda: synth.qwen_decode_layer(factor_std="visible", zero_dominants=True),
    "high_e": lambda: synth.high_e_layer(),
    "high_e_visible": lambda: synth.high_e_layer(factor_std="visible"),
    "tree": lambda: synth.btexperts_tree_layer(factor_std="visible"),
    "binary": lambda: synth.btexperts_binary_layer(factor_std="visible"),
    "single_base": lambda: synth.d2moe_base_layer(factor_std="visible"),
}


@pytest.mark.parametrize("T", [1, 8, 32, 64])
def test_qwen_decode_batches(T):
    src, L = installed("qwen", FULL["qwen"])
    x = synth.tokens(src, T, seed=T)
    ids, _ = check_route(src, L, x, 8)
    check_buckets(src, L, ids)
    check_forward(src, L, x, 8)


@pytest.mark.parametrize("name", ["high_e", "tree", "binary", "single_base"])
@pytest.mark.parametrize("T", [1, 32, 64])
def test_full_layers_decode(name, T):
    """Decode batches of the other full-size layers (depth-3 tree paths; split-K
    anchor tiles where the streaming path splits them: the high-expert-count
    layer at T = 32, gate/up in four K ranges and down in two, the d_ff = 768
    layers at T = 64, gate/up in four)."""
    src, L = installed(name, FULL[name])
    x = synth.tokens(src, T, seed=40 + T)
    ids, _ = check_route(src, L, x, 8)
    check_buckets(src, L, ids)
    check_forward(src, L, x, 8)


@pytest.mark.parametrize("name", ["stream_split_ragged", "stream_split_tree"])
def test_stream_split_band(name):
    """A batch inside the band where the streaming path splits the anchors'
    products along K (tokens x gate/up column tiles between 1.5 and 3.1 times
    the streaming grid of 5 CTAs per SM): three K ranges with a ragged last one,
    and two on a tree layer."""
    src, L = installed(name, SMALL[name])
    grid = 5 * torch.cuda.get_device_properties(0).multi_processor_count
    ct = (2 * src.d_ff + 63) // 64
    T = -(-3 * grid // (2 * ct)) + 1
    assert 10 * T * ct <= 31 * grid and T <= 256
    x = synth.tokens(src, T, seed=60)
    ids, _ = check_route(src, L, x, src.top_k)
    check_buckets(src, L, ids)
    check_forward(src, L, x, src.top_k)


def test_qwen_decode_correction_visible():
    src, L = installed("qwen_visible", FULL["qwen_visible"])
    x = synth.tokens(src, 64, seed=3)
    check_route(src, L, x, 8)
    check_forward(src, L, x, 8)


@pytest.mark.parametrize("name", ["qwen_visible", "qwen_zero_dom", "high_e_visible"])
@pytest.mark.parametrize("T", [1, 8, 32, 64])
def test_full_size_correction_visible_decode(name, T):
    """Full-size layers whose corrections are visible under the bf16 bar (or
    the only term), every token of a decode batch."""
    src, L = installed(name, FULL[name])
    x = synth.tokens(src, T, seed=60 + T)
    ids, _ = check_route(src, L, x, 8)
    check_buckets(src, L, ids)
    check_forward(src, L, x, 8)


def _sample(T, n=24, seed=0):
    rng = np.random.default_rng(seed)
    return np.unique(np.concatenate([[0, T - 1], rng.choice(T, n, replace=False)]))


@pytest.mark.parametrize("name,T", [("qwen", 8192), ("high_e", 4096), ("tree", 2048),
                                    ("binary", 2048), ("single_base", 2048),
                                    ("qwen_visible", 8192), ("qwen_zero_dom", 8192),
                                    ("high_e_visible", 4096)])
def test_full_size_sampled(name, T):
    src, L = installed(name, FULL[name])
    x = synth.tokens(src, T, seed=11)
    ids, _ = check_route(src, L, x, 8)
    check_buckets(src, L, ids)
    check_forward(src, L, x, 8, sample=_sample(T))
