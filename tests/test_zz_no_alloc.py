"""lx_bucket_noalloc: bucketing without any device allocation during the call.

Some callers may not call cudaMalloc at all while they run -- serving runtimes
whose device memory belongs to their own pooling allocator or a fixed budget,
and latency-critical loops where cudaMalloc/cudaFree could synchronise the
device.  lx_bucket_noalloc serves them: its temporary buffers live in one
static device array of the library, and the caller passes every output.

This file runs last (its name sorts last), so that a run stopping at its first
failure has already run every other test; it also passes on its own in a fresh
process.  Each case calls the new entry point twice in a row through the C ABI
(the second call smaller than the first, so stale scratch contents from the
first call would show) and compares every output bit for bit with the oracle's
plain-loop bucketing and with the existing lx_bucket + lx_get_buckets path.
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle
import synth
from paper_2608_07814_gb300 import lx

pytestmark = pytest.mark.gpu

KEYS = ("node_off", "node_tok", "node_row", "expert_off", "perm")


def _r256(v):
    return (v + 255) // 256 * 256


def scratch_need(n_nodes, E, T, k, D):
    """Scratch bytes of one call, by the formula the header states."""
    keys, Tp = n_nodes + E, (T + 15) // 16 * 16
    return (_r256(keys * Tp) + _r256(4 * keys * Tp) + _r256(4 * keys) + _r256(4 * (keys + 2))
            + _r256(4 * T * k * D))


def largest_T(n_nodes, E, k, D):
    T = 1
    while scratch_need(n_nodes, E, T + 1, k, D) <= lx.LX_NOALLOC_SCRATCH_BYTES:
        T += 1
    return T


def _outputs(layer, T, k):
    D = layer.info()["max_depth"]
    full = lambda n: torch.full((n,), -7, dtype=torch.int32, device="cuda")
    return dict(node_off=full(layer.info()["n_nodes"] + 1), node_tok=full(max(1, T * k * D)),
                node_row=full(max(1, T * k * D)), expert_off=full(layer.n_experts + 1),
                perm=full(max(1, T * k)))


def _noalloc(layer, ids, out, T=None, k=None):
    """Call lx_bucket_noalloc on outputs allocated by the caller before the call."""
    T = ids.shape[0] if T is None else T
    k = ids.shape[1] if k is None else k
    p = lambda t: ctypes.c_void_p(t.data_ptr())
    st = lx.lib().lx_bucket_noalloc(layer.handle, p(ids), T, k, p(out["node_off"]),
                                    p(out["node_tok"]), p(out["node_row"]), p(out["expert_off"]),
                                    p(out["perm"]),
                                    ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    if st != lx.LX_OK:
        raise lx.LxError(st, lx.lib().lx_last_error().decode())
    return out


def _check_against_oracle(src, got, ids_host):
    ref = oracle.buckets(src, ids_host)
    rows = int(ref["node_off"][-1])
    for key in KEYS:
        g = got[key].cpu().numpy()
        if key == "node_tok":
            g = g[:rows]
        assert np.array_equal(g, ref[key]), key


CASES = {
    "flat_qwen_like": lambda: synth.flat_layer(512, 256, [4] * 32, 16, 8, "bf16", seed=21,
                                               skew=synth.QWEN_SKEW),
    "tree": lambda: synth.tree_layer(256, 128, 4, 4, 3, 16, 8, 8, "bf16", seed=22,
                                     skew=synth.TREE_SKEW),
}


@pytest.mark.parametrize("name", sorted(CASES))
def test_noalloc_matches_oracle_and_existing_bucketing_twice(name):
    src = CASES[name]()
    layer = lx.Layer(src)
    for call, T in enumerate((3000, 257)):
        x = lx.host_to_torch(synth.tokens(src, T, seed=50 + call), src.dtype).cuda()
        ids, _ = layer.route(x, src.top_k)
        out = _outputs(layer, T, src.top_k)
        torch.cuda.synchronize()
        free0 = torch.cuda.mem_get_info()[0]
        got = _noalloc(layer, ids, out)
        torch.cuda.synchronize()
        # the property the entry point exists for: no device memory taken
        assert torch.cuda.mem_get_info()[0] == free0
        _check_against_oracle(src, got, ids.cpu().numpy())
        layer.bucket(ids)
        ref = layer.get_buckets()
        torch.cuda.synchronize()
        rows = int(ref["node_off"][-1])
        for key in KEYS:
            g, r = got[key], ref[key]
            if key == "node_tok":
                g, r = g[:rows], r[:rows]
            assert torch.equal(g, r), key
    layer.free()


def test_noalloc_largest_admitted_batch_and_the_next_size():
    """The largest T the fixed array admits for this layer (computed from the
    header's formula) runs and matches the oracle; the next 16-token size is
    rejected with LX_ERR_SHAPE before any launch."""
    src = CASES["flat_qwen_like"]()
    layer = lx.Layer(src)
    k, D = src.top_k, layer.info()["max_depth"]
    Tmax = largest_T(src.n_nodes, src.n_experts, k, D)
    assert Tmax == 12480   # keys = 256, k = 8, D = 2, the Qwen3-30B-A3B-shaped layer's sizes
    x = lx.host_to_torch(synth.tokens(src, Tmax, seed=77), src.dtype).cuda()
    ids, _ = layer.route(x, k)
    out = _outputs(layer, Tmax, k)
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    got = _noalloc(layer, ids, out)
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info()[0] == free0
    _check_against_oracle(src, got, ids.cpu().numpy())
    T2 = Tmax + 1    # rounds up to the next 16-token size
    assert scratch_need(src.n_nodes, src.n_experts, T2, k, D) > lx.LX_NOALLOC_SCRATCH_BYTES
    ids2 = torch.zeros((T2, k), dtype=torch.int32, device="cuda")
    with pytest.raises(lx.LxError) as e:
        _noalloc(layer, ids2, _outputs(layer, T2, k))
    assert e.value.status == lx.LX_ERR_SHAPE
    assert "scratch" in str(e.value)
    layer.free()


def test_noalloc_zero_tokens_zeroes_the_offsets():
    src = CASES["tree"]()
    layer = lx.Layer(src)
    out = _outputs(layer, 0, src.top_k)
    ids = torch.zeros((1, src.top_k), dtype=torch.int32, device="cuda")
    _noalloc(layer, ids, out, T=0)
    torch.cuda.synchronize()
    assert int(out["node_off"].abs().sum()) == 0
    assert int(out["expert_off"].abs().sum()) == 0
    assert int(out["perm"][0]) == -7     # nothing else written
    layer.free()
