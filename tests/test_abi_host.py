"""Host-side checks of the C ABI: the library loads, exports every symbol that
include/lx.h declares, and rejects invalid layers and calls on the host before
touching the GPU (so these run without one)."""
import copy
import ctypes
import os
import re

import numpy as np
import pytest
import torch

import synth
from paper_2608_07814_gb300 import build as lxbuild
from paper_2608_07814_gb300 import lx

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def L():
    if not os.path.exists(lx.LIB_PATH):
        lxbuild.build()
    return lx.lib()


def declared_symbols():
    src = open(os.path.join(ROOT, "include", "lx.h")).read()
    return sorted(set(re.findall(r"LX_API\s+[\w\s\*]+?\b(lx_\w+)\s*\(", src)))


def test_exports_every_declared_symbol(L):
    names = declared_symbols()
    assert len(names) >= 12
    for n in names:
        assert hasattr(L, n), n
    assert sorted(lx.EXPORTS) == names


def test_last_error_empty_initially(L):
    assert isinstance(L.lx_last_error(), bytes)


def _load_status(layer):
    try:
        lx.Layer(layer).free()
        return lx.LX_OK
    except lx.LxError as e:
        return e.status


def _base():
    return synth.flat_layer(64, 32, [4, 4], 8, 2, "f32", seed=0)


@pytest.mark.parametrize("mutate,status", [
    (lambda l: setattr(l, "d_model", 60), lx.LX_ERR_SHAPE),          # not a multiple of 8
    (lambda l: setattr(l, "n_experts", 0), lx.LX_ERR_SHAPE),
    (lambda l: l.node_parent.__setitem__(2, 99), lx.LX_ERR_SHAPE),   # parent out of range
    (lambda l: l.node_parent.__setitem__(2, 2), lx.LX_ERR_SHAPE),    # self parent
    (lambda l: l.node_rank.__setitem__(0, 4), lx.LX_ERR_SHAPE),      # anchor with rank
    (lambda l: l.node_rank.__setitem__(3, 0), lx.LX_ERR_SHAPE),      # correction rank 0
    (lambda l: l.node_rank.__setitem__(3, 33), lx.LX_ERR_SHAPE),     # rank > min(I,H)
    (lambda l: l.expert_node.__setitem__(1, 99), lx.LX_ERR_SHAPE),
    (lambda l: setattr(l, "node_sign", np.asarray([1, 1, 2, 1, 1, 1, 1, 1], np.int8)),
     lx.LX_ERR_SHAPE),                                                # sign not +-1
    (lambda l: setattr(l, "node_sign", np.asarray([-1, 1, 1, 1, 1, 1, 1, 1], np.int8)),
     lx.LX_ERR_SHAPE),                                                # negative anchor edge
])
def test_invalid_layers_rejected_on_host(L, mutate, status):
    layer = copy.deepcopy(_base())
    mutate(layer)
    assert _load_status(layer) == status


def test_cycle_and_depth_rejected(L):
    layer = copy.deepcopy(_base())
    # nodes 2 -> 3 -> 2 (cycle among corrections)
    layer.node_parent[2] = 3
    layer.node_parent[3] = 2
    assert _load_status(layer) == lx.LX_ERR_SHAPE
    deep = synth.tree_layer(64, 32, 1, 1, 1, 4, 4, 2, "f32", seed=0)
    # chain of depth 5: anchor <- a <- b <- c <- d
    n = deep.n_nodes
    parent = list(deep.node_parent) + [n - 1, n]
    rank = list(deep.node_rank) + [4, 4]
    deep.node_parent = np.asarray(parent, np.int32)
    deep.node_rank = np.asarray(rank, np.int32)
    deep.node_w = deep.node_w + [deep.node_w[-1], deep.node_w[-1]]
    deep.expert_node[0] = n + 1
    assert _load_status(deep) == lx.LX_ERR_SHAPE


def test_null_arguments(L):
    st = L.lx_load_compressed_layer(None, None, None, None, None, ctypes.byref(ctypes.c_void_p()))
    assert st == lx.LX_ERR_ARG
    assert b"NULL" in L.lx_last_error()
    assert L.lx_moe_forward(None, None, 1, 1, None, None) == lx.LX_ERR_ARG
    assert L.lx_route(None, None, 1, 1, None, None, None, None) == lx.LX_ERR_ARG
    assert L.lx_free_layer(None) == lx.LX_ERR_ARG
    n = ctypes.c_int32()
    assert L.lx_read_profile(None, None, 0, ctypes.byref(n)) == lx.LX_ERR_ARG


@pytest.mark.skipif(torch.cuda.is_available(), reason="checks the no-GPU error path")
def test_valid_layer_without_gpu_reports_cuda_error(L):
    assert _load_status(_base()) == lx.LX_ERR_CUDA
    signed = synth.binary_tree_layer(64, 32, 1, 3, [8, 8, 8], 2, "f32", seed=0, signed=True)
    assert _load_status(signed) == lx.LX_ERR_CUDA      # passes validation


def test_statistics_calls_rejected_on_host(L):
    """Argument checks of the router-statistics calls come before any CUDA call."""
    buf = ctypes.c_void_p(8)  # never dereferenced: every call below fails validation
    assert L.lx_coact_accumulate(buf, -1, 4, 16, buf, buf, None) == lx.LX_ERR_ARG
    assert L.lx_coact_accumulate(buf, 4, 0, 16, buf, buf, None) == lx.LX_ERR_ARG
    assert L.lx_coact_accumulate(buf, 4, 33, 16, buf, buf, None) == lx.LX_ERR_ARG
    assert L.lx_coact_accumulate(buf, 4, 4, 0, buf, buf, None) == lx.LX_ERR_ARG
    assert L.lx_coact_accumulate(buf, 4, 4, 1025, buf, buf, None) == lx.LX_ERR_ARG
    assert L.lx_coact_accumulate(buf, 4, 4, 16, None, None, None) == lx.LX_ERR_ARG
    assert L.lx_coact_accumulate(None, 4, 4, 16, buf, None, None) == lx.LX_ERR_ARG
    assert L.lx_coact_accumulate(None, 0, 4, 16, buf, None, None) == lx.LX_OK   # T = 0
    assert L.lx_coact_npmi(None, 16, 4, buf, None) == lx.LX_ERR_ARG
    assert L.lx_coact_npmi(buf, 0, 4, buf, None) == lx.LX_ERR_ARG
    assert L.lx_coact_npmi(buf, 16, -1, buf, None) == lx.LX_ERR_ARG


def _declared_arity():
    """{name: parameter count} of every LX_API function in include/lx.h."""
    src = open(os.path.join(ROOT, "include", "lx.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    out = {}
    for m in re.finditer(r"LX_API\s+[\w\s\*]+?\b(lx_\w+)\s*\(([^)]*)\)\s*;", src, flags=re.S):
        params = m.group(2).strip()
        out[m.group(1)] = 0 if params in ("", "void") else len(params.split(","))
    return out


def test_binding_arity_matches_header(L):
    arity = _declared_arity()
    assert sorted(arity) == sorted(lx.EXPORTS)
    for name, n in arity.items():
        f = getattr(L, name)
        got = len(f.argtypes) if f.argtypes is not None else 0
        assert got == n, f"{name}: binding declares {got} arguments, the header {n}"


def test_layer_desc_struct_matches_header():
    """lx_layer_desc's fields, in order, as the binding lays them out."""
    src = open(os.path.join(ROOT, "include", "lx.h")).read()
    body = re.search(r"typedef struct \{(.*?)\} lx_layer_desc;", src, flags=re.S).group(1)
    body = re.sub(r"/\*.*?\*/", "", body, flags=re.S)
    fields = re.findall(r"\b(\w+)\s*;", body)
    assert fields == [f for f, _ in lx.LayerDesc._fields_]


def test_wait_hooks_reject_bad_arguments(L):
    assert L.lx_set_wait_limit(None, 1000) == lx.LX_ERR_ARG
    assert L.lx_inject_unmet_wait(None, lx.LX_WAIT_STREAM_DEP) == lx.LX_ERR_ARG
    assert L.lx_clear_device_error(None) == lx.LX_ERR_ARG
