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
first call would show) and compares every output with the existing
lx_bucket + lx_get_buckets path, bit for bit (integer outputs).
"""
import ctypes

import numpy as np
import pytest
import torch

import synth
from paper_2608_07814_gb300 import lx

pytestmark = pytest.mark.gpu


def _noalloc(layer, ids):
    """Call lx_bucket_noalloc with outputs allocated here, before the call."""
    T, k = ids.shape
    D = layer.info()["max_depth"]
    dev = ids.device
    out = dict(node_off=torch.full((layer.info()["n_nodes"] + 1,), -7, dtype=torch.int32, device=dev),
               node_tok=torch.full((T * k * D,), -7, dtype=torch.int32, device=dev),
               node_row=torch.full((T * k * D,), -7, dtype=torch.int32, device=dev),
               expert_off=torch.full((layer.n_experts + 1,), -7, dtype=torch.int32, device=dev),
               perm=torch.full((T * k,), -7, dtype=torch.int32, device=dev))
    p = lambda t: ctypes.c_void_p(t.data_ptr())
    st = lx.lib().lx_bucket_noalloc(layer.handle, p(ids), T, k, p(out["node_off"]),
                                    p(out["node_tok"]), p(out["node_row"]), p(out["expert_off"]),
                                    p(out["perm"]),
                                    ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    if st != lx.LX_OK:
        raise lx.LxError(st, lx.lib().lx_last_error().decode())
    return out


def _existing(layer, ids):
    layer.bucket(ids)
    return layer.get_buckets()


CASES = {
    "flat_qwen_like": lambda: synth.flat_layer(512, 256, [4] * 32, 16, 8, "bf16", seed=21,
                                               skew=synth.QWEN_SKEW),
    "tree": lambda: synth.tree_layer(256, 128, 4, 4, 3, 16, 8, 8, "bf16", seed=22,
                                     skew=synth.TREE_SKEW),
}


@pytest.mark.parametrize("name", sorted(CASES))
def test_noalloc_matches_existing_bucketing_twice(name):
    src = CASES[name]()
    layer = lx.Layer(src)
    for call, T in enumerate((3000, 257)):
        x = lx.host_to_torch(synth.tokens(src, T, seed=50 + call), src.dtype).cuda()
        ids, _ = layer.route(x, src.top_k)
        got = _noalloc(layer, ids)
        ref = _existing(layer, ids)
        torch.cuda.synchronize()
        rows = int(ref["node_off"][-1])
        assert torch.equal(got["node_off"], ref["node_off"])
        assert torch.equal(got["expert_off"], ref["expert_off"])
        assert torch.equal(got["node_tok"][:rows], ref["node_tok"][:rows])
        assert torch.equal(got["node_row"], ref["node_row"])
        assert torch.equal(got["perm"], ref["perm"])
    layer.free()


def test_noalloc_rejects_sizes_beyond_the_array():
    src = CASES["flat_qwen_like"]()
    layer = lx.Layer(src)
    T = 40000     # 5 bytes * 256 keys * 40000 tokens > 16 MiB
    ids = torch.zeros((T, src.top_k), dtype=torch.int32, device="cuda")
    with pytest.raises(lx.LxError) as e:
        _noalloc(layer, ids)
    assert e.value.status == lx.LX_ERR_SHAPE
    assert "scratch" in str(e.value)
    layer.free()
