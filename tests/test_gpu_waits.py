"""The bounded device-side waits, made to run out on purpose.

A test hook (lx_inject_unmet_wait) makes one wait of the forward wait for a
condition nothing fulfils, and lx_set_wait_limit shortens the bound to about a
millisecond.  No fault, trap or endless loop is involved: the wait gives up,
records LX_ERR_TIMEOUT in the layer's device error word, the CTA's other roles
stop, its copies in flight land and its tensor memory is freed, and the launch
ends normally.  The test then checks that the host reads the status, that the
context is still usable, and that the next forward (hook off, default bound)
matches the oracle -- the tensor-core case also shows that every CTA released
its tensor memory, since the next launch allocates the same columns again.
"""
import numpy as np
import pytest
import torch

import oracle
import synth
from paper_2608_07814_gb300 import lx

pytestmark = pytest.mark.gpu

SHORT = 2_000_000   # SM clock cycles, about 1 ms


def _layer():
    # dims and ranks multiples of 64: decode batches stream, larger ones use tcgen05
    src = synth.flat_layer(512, 384, [4] * 8, 64, 8, "bf16", seed=31, factor_std="visible",
                           skew=synth.QWEN_SKEW)
    return src, lx.Layer(src)


def _forward_ok(src, L, T, seed):
    x = synth.tokens(src, T, seed=seed)
    y = L.moe_forward(lx.host_to_torch(x, "bf16").cuda(), src.top_k)
    torch.cuda.synchronize()
    ref = oracle.moe_forward(src, x)
    yh = y.float().cpu().numpy()
    err = float(np.max(np.abs(yh - ref)) / np.max(np.abs(ref)))
    assert err <= 2e-2, err
    assert L.info()["device_error"] == 0


@pytest.mark.parametrize("site,T", [(lx.LX_WAIT_STREAM_DEP, 64), (lx.LX_WAIT_TC_MMA, 300)])
def test_unmet_wait_times_out_and_the_next_forward_is_correct(site, T):
    src, L = _layer()
    assert L.info()["stream_path"] == 1
    _forward_ok(src, L, T, seed=1)             # warm: workspace sized, kernels loaded
    L.set_wait_limit(SHORT)
    L.inject_unmet_wait(site)
    x = lx.host_to_torch(synth.tokens(src, T, seed=2), "bf16").cuda()
    L.moe_forward(x, src.top_k)
    torch.cuda.synchronize()                   # the launch ended: no hang, no fault
    assert L.info()["device_error"] == lx.LX_ERR_TIMEOUT
    # the context is usable: a plain torch kernel runs and reads back
    assert float(torch.ones(1024, device="cuda").sum()) == 1024.0
    L.inject_unmet_wait(lx.LX_WAIT_NONE)
    L.set_wait_limit(0)
    L.clear_device_error()
    assert L.info()["device_error"] == 0
    _forward_ok(src, L, T, seed=3)
    _forward_ok(src, L, 64 if T > 256 else 300, seed=4)   # the other kernel family too
    L.free()


def test_short_bound_alone_does_not_fire():
    """A 1 ms bound is far above every wait of a healthy forward: nothing times out."""
    src, L = _layer()
    L.set_wait_limit(SHORT)
    for T in (1, 64, 300):
        _forward_ok(src, L, T, seed=10 + T)
    L.free()
