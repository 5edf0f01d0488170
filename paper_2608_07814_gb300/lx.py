"""Python binding of liblx (the C ABI declared in include/lx.h).

Argument marshalling only: every step of the forward runs in the CUDA library.
PyTorch provides device memory and the current stream.  There is no fallback:
if liblx.so is missing or cannot load, every call raises.
"""
from __future__ import annotations

import ctypes
import os
from typing import Dict, Optional

import numpy as np
import torch

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "liblx.so")

LX_OK, LX_ERR_ARG, LX_ERR_SHAPE, LX_ERR_CUDA, LX_ERR_OOM, LX_ERR_TIMEOUT, LX_ERR_STATE, \
    LX_ERR_UNSUPPORTED = range(8)
STATUS_NAMES = ["LX_OK", "LX_ERR_ARG", "LX_ERR_SHAPE", "LX_ERR_CUDA", "LX_ERR_OOM",
                "LX_ERR_TIMEOUT", "LX_ERR_STATE", "LX_ERR_UNSUPPORTED"]
LX_F32, LX_BF16 = 0, 1
LX_PATH_AUTO, LX_PATH_GENERIC = 0, 1
LX_MAX_DEPTH, LX_MAX_K, LX_MAX_EXPERTS = 4, 32, 1024

# every symbol include/lx.h declares
EXPORTS = [
    "lx_load_compressed_layer", "lx_free_layer", "lx_reserve", "lx_route", "lx_bucket",
    "lx_moe_forward", "lx_get_buckets", "lx_layer_info", "lx_set_path", "lx_set_profiling",
    "lx_read_profile", "lx_last_error", "lx_bucket_noalloc", "lx_coact_accumulate",
    "lx_coact_npmi", "lx_align_cost", "lx_lap_solve", "lx_lap_solve_batch", "lx_permute_neurons",
    "lx_compress_workspace", "lx_compress_factor", "lx_set_wait_limit", "lx_inject_unmet_wait",
    "lx_clear_device_error",
]
LX_WAIT_NONE, LX_WAIT_STREAM_DEP, LX_WAIT_TC_MMA = 0, 1, 2
LX_NOALLOC_SCRATCH_BYTES = 16 << 20


class LxError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"{STATUS_NAMES[status] if 0 <= status < 8 else status}: {msg}")
        self.status = status


class LayerDesc(ctypes.Structure):
    _fields_ = [("d_model", ctypes.c_int32), ("d_ff", ctypes.c_int32),
                ("n_experts", ctypes.c_int32), ("n_nodes", ctypes.c_int32),
                ("dtype", ctypes.c_int32), ("node_parent", ctypes.POINTER(ctypes.c_int32)),
                ("node_rank", ctypes.POINTER(ctypes.c_int32)),
                ("expert_node", ctypes.POINTER(ctypes.c_int32)),
                ("node_sign", ctypes.POINTER(ctypes.c_int8))]


class LayerInfo(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in (
        "d_model", "d_ff", "n_experts", "n_nodes", "dtype", "n_anchors", "n_corrections",
        "max_depth", "max_rank")] + [("weight_bytes", ctypes.c_int64)] + [
        (n, ctypes.c_int32) for n in ("last_T", "last_k", "last_rows", "device_error",
                                      "stream_path")]


class KernelTime(ctypes.Structure):
    _fields_ = [("name", ctypes.c_char_p), ("ms", ctypes.c_float)]


_lib = None


def lib() -> ctypes.CDLL:
    """Load liblx.so; raises if it is missing (no fallback exists)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(
                f"{LIB_PATH} is missing: build it with `python -m paper_2608_07814_gb300.build`")
        L = ctypes.CDLL(LIB_PATH)
        vp, i32 = ctypes.c_void_p, ctypes.c_int32
        sig = {
            "lx_load_compressed_layer": [ctypes.POINTER(LayerDesc), vp, vp, vp, vp,
                                         ctypes.POINTER(vp)],
            "lx_free_layer": [vp],
            "lx_reserve": [vp, i32, i32],
            "lx_route": [vp, vp, i32, i32, vp, vp, vp, vp],
            "lx_bucket": [vp, vp, i32, i32, vp],
            "lx_moe_forward": [vp, vp, i32, i32, vp, vp],
            "lx_get_buckets": [vp, vp, vp, vp, vp, vp, vp],
            "lx_layer_info": [vp, ctypes.POINTER(LayerInfo)],
            "lx_set_path": [vp, i32],
            "lx_set_profiling": [vp, i32],
            "lx_set_wait_limit": [vp, ctypes.c_uint64],
            "lx_inject_unmet_wait": [vp, i32],
            "lx_clear_device_error": [vp],
            "lx_read_profile": [vp, ctypes.POINTER(KernelTime), i32, ctypes.POINTER(i32)],
            "lx_bucket_noalloc": [vp, vp, i32, i32, vp, vp, vp, vp, vp, vp],
            "lx_coact_accumulate": [vp, i32, i32, i32, vp, vp, vp],
            "lx_coact_npmi": [vp, i32, ctypes.c_int64, vp, vp],
            "lx_align_cost": [i32, i32, i32, vp, vp, vp, vp, vp, vp, vp, vp],
            "lx_lap_solve": [vp, i32, vp, ctypes.POINTER(ctypes.c_double)],
            "lx_lap_solve_batch": [vp, i32, i32, vp, vp, i32],
            "lx_permute_neurons": [i32, i32, i32, vp, vp, vp, vp, vp, vp, vp, vp],
            "lx_compress_workspace": [i32, i32, i32, i32, ctypes.POINTER(ctypes.c_uint64)],
            "lx_compress_factor": [i32, i32, i32, vp, vp, vp, i32, i32, i32, vp, vp, vp, vp,
                                   ctypes.c_uint64, vp],
        }
        for name, args in sig.items():
            f = getattr(L, name)
            f.argtypes = args
            f.restype = ctypes.c_int
        L.lx_last_error.argtypes = []
        L.lx_last_error.restype = ctypes.c_char_p
        _lib = L
    return _lib


def _check(status: int) -> None:
    if status != LX_OK:
        raise LxError(status, lib().lx_last_error().decode())


def _stream(stream: Optional[torch.cuda.Stream]) -> ctypes.c_void_p:
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def host_to_torch(a: np.ndarray, dtype: str) -> torch.Tensor:
    """Storage array (bf16 as uint16 bits, or float32) -> CPU torch tensor."""
    if dtype == "bf16":
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16)
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32))


class Layer:
    """A compressed MoE layer installed on the current CUDA device.

    ``src`` is any object with the fields of ``synth.CompressedLayer``
    (d_model, d_ff, n_experts, dtype in {'f32','bf16'}, node_parent, node_rank,
    expert_node, node_w, router_w, router_bias, and optionally node_sign)."""

    def __init__(self, src, stream: Optional[torch.cuda.Stream] = None):
        L = lib()
        if src.dtype not in ("f32", "bf16"):
            raise ValueError("liblx stores f32 or bf16 layers")
        self.dtype = src.dtype
        self.torch_dtype = torch.bfloat16 if src.dtype == "bf16" else torch.float32
        self.d_model, self.d_ff, self.n_experts = src.d_model, src.d_ff, src.n_experts
        want = np.uint16 if src.dtype == "bf16" else np.float32
        self._keep = []
        parent = np.ascontiguousarray(src.node_parent, np.int32)
        rank = np.ascontiguousarray(src.node_rank, np.int32)
        enode = np.ascontiguousarray(src.expert_node, np.int32)
        self._keep += [parent, rank, enode]
        sign = getattr(src, "node_sign", None)
        if sign is not None:
            sign = np.ascontiguousarray(sign, np.int8)
            self._keep.append(sign)
        N = parent.shape[0]
        ptrs = (ctypes.c_void_p * (6 * N))()
        for n, ws in enumerate(src.node_w):
            for j, a in enumerate(ws):
                a = np.ascontiguousarray(a, dtype=want)
                self._keep.append(a)
                ptrs[6 * n + j] = a.ctypes.data
        rw = np.ascontiguousarray(src.router_w, dtype=want)
        self._keep.append(rw)
        bias = None
        if src.router_bias is not None:
            bias = np.ascontiguousarray(src.router_bias, np.float32)
            self._keep.append(bias)
        desc = LayerDesc(src.d_model, src.d_ff, src.n_experts, N,
                         LX_BF16 if src.dtype == "bf16" else LX_F32,
                         parent.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)),
                         rank.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)),
                         enode.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)),
                         None if sign is None else sign.ctypes.data_as(
                             ctypes.POINTER(ctypes.c_int8)))
        h = ctypes.c_void_p()
        st = L.lx_load_compressed_layer(ctypes.byref(desc), ptrs, ctypes.c_void_p(rw.ctypes.data),
                                        None if bias is None else ctypes.c_void_p(bias.ctypes.data),
                                        _stream(stream) if torch.cuda.is_available() else None,
                                        ctypes.byref(h))
        self._keep = None
        _check(st)
        self.handle = h
        self.info_cache = self.info()

    # ---- lifetime
    def free(self) -> None:
        if getattr(self, "handle", None):
            _check(lib().lx_free_layer(self.handle))
            self.handle = None

    def __del__(self):
        try:
            self.free()
        except Exception:
            pass

    # ---- calls
    def info(self) -> Dict[str, int]:
        inf = LayerInfo()
        _check(lib().lx_layer_info(self.handle, ctypes.byref(inf)))
        return {n: getattr(inf, n) for n, _ in LayerInfo._fields_}

    def reserve(self, max_tokens: int, k: int) -> None:
        _check(lib().lx_reserve(self.handle, max_tokens, k))

    def set_wait_limit(self, cycles: int) -> None:
        """Bound (SM clock cycles) of the kernels' device-side waits; 0 = default."""
        _check(lib().lx_set_wait_limit(self.handle, int(cycles)))

    def inject_unmet_wait(self, site: int) -> None:
        """Test hook: make the wait at `site` (LX_WAIT_*) run out."""
        _check(lib().lx_inject_unmet_wait(self.handle, int(site)))

    def clear_device_error(self) -> None:
        _check(lib().lx_clear_device_error(self.handle))

    def set_path(self, path: int) -> None:
        _check(lib().lx_set_path(self.handle, path))

    def set_profiling(self, on: bool) -> None:
        _check(lib().lx_set_profiling(self.handle, 1 if on else 0))

    def read_profile(self, cap: int = 4096):
        buf = (KernelTime * cap)()
        n = ctypes.c_int32()
        _check(lib().lx_read_profile(self.handle, buf, cap, ctypes.byref(n)))
        return [(buf[i].name.decode(), float(buf[i].ms)) for i in range(n.value)]

    def route(self, x: torch.Tensor, k: int, want_logits: bool = False, stream=None):
        T = x.shape[0]
        dev = x.device
        ids = torch.empty((T, k), dtype=torch.int32, device=dev)
        w = torch.empty((T, k), dtype=torch.float32, device=dev)
        logits = torch.empty((T, self.n_experts), dtype=torch.float32, device=dev) \
            if want_logits else None
        _check(lib().lx_route(self.handle, _ptr(x), T, k, _ptr(ids), _ptr(w), _ptr(logits),
                              _stream(stream)))
        return (ids, w, logits) if want_logits else (ids, w)

    def bucket(self, topk_id: torch.Tensor, stream=None) -> None:
        T, k = topk_id.shape
        _check(lib().lx_bucket(self.handle, _ptr(topk_id), T, k, _stream(stream)))

    def moe_forward(self, x: torch.Tensor, k: int, y: Optional[torch.Tensor] = None,
                    stream=None) -> torch.Tensor:
        if y is None:
            y = torch.empty_like(x)
        _check(lib().lx_moe_forward(self.handle, _ptr(x), x.shape[0], k, _ptr(y),
                                    _stream(stream)))
        return y

    def get_buckets(self, stream=None) -> Dict[str, torch.Tensor]:
        inf = self.info()
        T, k, D = inf["last_T"], inf["last_k"], inf["max_depth"]
        dev = torch.device("cuda", torch.cuda.current_device())
        z = lambda n: torch.empty(max(1, n), dtype=torch.int32, device=dev)
        out = dict(node_off=z(inf["n_nodes"] + 1), node_tok=z(T * k * D), node_row=z(T * k * D),
                   expert_off=z(self.n_experts + 1), perm=z(T * k))
        _check(lib().lx_get_buckets(self.handle, _ptr(out["node_off"]), _ptr(out["node_tok"]),
                                    _ptr(out["node_row"]), _ptr(out["expert_off"]),
                                    _ptr(out["perm"]), _stream(stream)))
        out["node_tok"] = out["node_tok"][:inf["last_rows"]]
        out["node_row"] = out["node_row"][:T * k * D]
        out["perm"] = out["perm"][:T * k]
        return out


# ----------------------------------------------------------------------------
# router profiling statistics (standalone calls, no layer)
# ----------------------------------------------------------------------------
def coact_accumulate(topk_id: torch.Tensor, E: int, fire: Optional[torch.Tensor] = None,
                     coact: Optional[torch.Tensor] = None, stream=None):
    """Adds the batch topk_id [T, k] (int32, device) to the uint64 counters
    fire [E] and coact [E, E] (int64 tensors holding the unsigned counts;
    allocated zeroed when omitted).  Returns (fire, coact)."""
    dev = topk_id.device
    if fire is None:
        fire = torch.zeros(E, dtype=torch.int64, device=dev)
    if coact is None:
        coact = torch.zeros((E, E), dtype=torch.int64, device=dev)
    T, k = topk_id.shape
    _check(lib().lx_coact_accumulate(_ptr(topk_id), T, k, E, _ptr(fire), _ptr(coact),
                                     _stream(stream)))
    return fire, coact


def coact_npmi(coact: torch.Tensor, n_tokens: int, stream=None) -> torch.Tensor:
    """float64 [E, E] NPMI of the counts coact [E, E] over n_tokens tokens."""
    E = coact.shape[0]
    out = torch.empty((E, E), dtype=torch.float64, device=coact.device)
    _check(lib().lx_coact_npmi(_ptr(coact), E, n_tokens, _ptr(out), _stream(stream)))
    return out


# ----------------------------------------------------------------------------
# neuron alignment (standalone calls on plain expert matrices)
# ----------------------------------------------------------------------------
def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return LX_BF16
    if t.dtype == torch.float32:
        return LX_F32
    raise ValueError("expert matrices must be bf16 or fp32")


def align_cost(dom, mem, stream=None) -> torch.Tensor:
    """fp32 [I, I] cost of matching dominant neurons (rows) with member neurons
    (columns); dom and mem are (gate [I,H], up [I,H], down [H,I]) device tensors."""
    g = dom[0]
    I, H = g.shape
    cost = torch.empty((I, I), dtype=torch.float32, device=g.device)
    _check(lib().lx_align_cost(_dtype_code(g), H, I, *[_ptr(t) for t in dom],
                               *[_ptr(t) for t in mem], _ptr(cost), _stream(stream)))
    return cost


def lap_solve(cost: np.ndarray):
    """(assign int32 [n], total float) of the exact assignment of a host cost."""
    c = np.ascontiguousarray(cost, dtype=np.float32)
    n = c.shape[0]
    out = np.empty(n, np.int32)
    tot = ctypes.c_double()
    _check(lib().lx_lap_solve(ctypes.c_void_p(c.ctypes.data), n,
                              ctypes.c_void_p(out.ctypes.data), ctypes.byref(tot)))
    return out, tot.value


def lap_solve_batch(costs: np.ndarray, threads: int = 0):
    """(assign int32 [count, n], totals float64 [count]) of independent host
    costs [count, n, n], solved on `threads` host threads (0: all cores)."""
    c = np.ascontiguousarray(costs, dtype=np.float32)
    count, n = c.shape[0], c.shape[1]
    out = np.empty((count, n), np.int32)
    tot = np.empty(count, np.float64)
    _check(lib().lx_lap_solve_batch(ctypes.c_void_p(c.ctypes.data), n, count,
                                    ctypes.c_void_p(out.ctypes.data),
                                    ctypes.c_void_p(tot.ctypes.data), threads))
    return out, tot


def permute_neurons(perm: torch.Tensor, gate: torch.Tensor, up: torch.Tensor,
                    down: torch.Tensor, stream=None, out=None):
    """(gate, up, down) of the member with neuron i taken from neuron perm[i]
    (into ``out`` when given)."""
    I, H = gate.shape
    outs = out if out is not None else (torch.empty_like(gate), torch.empty_like(up),
                                        torch.empty_like(down))
    _check(lib().lx_permute_neurons(_dtype_code(gate), H, I, _ptr(perm), _ptr(gate), _ptr(up),
                                    _ptr(down), *[_ptr(t) for t in outs], _stream(stream)))
    return outs


# ----------------------------------------------------------------------------
# compression of one member projection
# ----------------------------------------------------------------------------
def compress_workspace_bytes(rows: int, cols: int, l: int, r: int) -> int:
    b = ctypes.c_uint64()
    _check(lib().lx_compress_workspace(rows, cols, l, r, ctypes.byref(b)))
    return int(b.value)


def compress_factor(w_dom: torch.Tensor, w_mem: torch.Tensor, omega: torch.Tensor, r: int,
                    power_iters: int = 2, workspace: Optional[torch.Tensor] = None,
                    stream=None, out=None):
    """(U [rows, r], V [cols, r], s [r]) fp32 with U V^T ~ w_mem - w_dom; omega
    is the fp32 [cols, l] Gaussian test matrix.  ``out`` = preallocated
    (U, V, s); independent projections may run concurrently on their own
    streams, each with its own workspace."""
    rows, cols = w_dom.shape
    l = omega.shape[1]
    need = compress_workspace_bytes(rows, cols, l, r)
    if workspace is None:
        workspace = torch.empty(need, dtype=torch.uint8, device=w_dom.device)
    dev = w_dom.device
    if out is None:
        out = (torch.empty((rows, r), dtype=torch.float32, device=dev),
               torch.empty((cols, r), dtype=torch.float32, device=dev),
               torch.empty(r, dtype=torch.float32, device=dev))
    U, V, s = out
    _check(lib().lx_compress_factor(_dtype_code(w_dom), rows, cols, _ptr(w_dom), _ptr(w_mem),
                                    _ptr(omega), l, r, power_iters, _ptr(U), _ptr(V), _ptr(s),
                                    _ptr(workspace), workspace.numel(), _stream(stream)))
    return U, V, s


_MEMBER_STREAMS: Dict[int, list] = {}


def compress_member(w_doms, w_mems, omegas, r: int, power_iters: int = 2, workspaces=None,
                    outs=None):
    """The gate, up and down projections of one member, each through
    lx_compress_factor on a stream of its own (the three are independent), the
    calling stream waiting for all three.  Lists of three: dominant and member
    matrices, fp32 Gaussian test matrices, optional workspaces and outputs.
    Returns the three (U, V, s)."""
    dev = w_doms[0].device
    main = torch.cuda.current_stream(dev)
    key = dev.index if dev.index is not None else torch.cuda.current_device()
    if key not in _MEMBER_STREAMS:
        _MEMBER_STREAMS[key] = [torch.cuda.Stream(device=dev) for _ in range(3)]
    streams = _MEMBER_STREAMS[key]
    start = torch.cuda.Event()
    start.record(main)
    res = []
    for j in range(3):
        st = streams[j]
        st.wait_event(start)
        ws = workspaces[j] if workspaces is not None else None
        out = outs[j] if outs is not None else None
        with torch.cuda.stream(st):
            res.append(compress_factor(w_doms[j], w_mems[j], omegas[j], r, power_iters,
                                       workspace=ws, stream=st, out=out))
        done = torch.cuda.Event()
        done.record(st)
        main.wait_event(done)
        if out is None:
            for t in res[-1]:  # allocated on the side stream, used on the caller's
                t.record_stream(main)
    return res
