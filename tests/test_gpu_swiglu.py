"""SwiGLU experts (App. B: the paper's own FFN, (SiLU(x W1) * (x W3)) W2) through
moevie_moe_forward against the oracle: routing bit-exact, outputs within rel-L2 1e-2
and max |err| 5e-2 * RMS.  The up-projection runs gate and up as one N = 256 MMA per
128 output columns (W1 tiles on the pair's first CTA, W3 tiles on the second)."""
import numpy as np
import pytest

import oracle
import workloads
from paper_2608_17402_gb300 import moevie
from tests._gpu import assert_close, check_status, layer_to_device, to_np_f64, workspace_for

pytestmark = pytest.mark.gpu


def _run(lay):
    x, W = layer_to_device(lay)
    ws = workspace_for(lay)
    y, rt = moevie.moevie_moe_forward(W, x, ws, routing=True)
    check_status(ws)
    return to_np_f64(y), {k: v.cpu().numpy() for k, v in rt.items()}


@pytest.mark.parametrize("T,d,E,k,h", [
    (1, 64, 4, 2, 64), (130, 128, 8, 2, 128), (257, 256, 16, 4, 416), (300, 128, 16, 4, 96),
    (200, 192, 8, 8, 384),
])
def test_swiglu_forward_small(T, d, E, k, h):
    cfg = workloads.small_config(T, d, E, k, h, seed=T + h, act="swiglu")
    lay = workloads.make_layer(cfg)
    y, rt = _run(lay)
    want, oidx, _, _ = oracle.forward_tokens(lay.x, lay.Wr, lay.b, lay.W1, lay.W2, k, W3=lay.W3)
    assert np.array_equal(rt["idx"], oidx)
    assert_close(y, want)


def test_swiglu_forward_image_batch_layer():
    """The s1 workload (c1's routed shape, SwiGLU experts), every token."""
    lay = workloads.make_layer(workloads.CONFIGS["s1"])
    y, rt = _run(lay)
    c = lay.cfg
    want, oidx, _, _ = oracle.forward_tokens(lay.x, lay.Wr, lay.b, lay.W1, lay.W2, c.k, W3=lay.W3)
    assert np.array_equal(rt["idx"], oidx)
    rel, mx = assert_close(y, want)
    print(f"s1: rel-L2 {rel:.2e}, max|err|/RMS {mx:.2e}")


@pytest.mark.parametrize("T,d,E,k,h,hs", [
    (1, 64, 4, 2, 64, 64), (300, 128, 16, 4, 128, 256), (257, 64, 8, 2, 64, 96),
])
def test_swiglu_with_shared_expert(T, d, E, k, h, hs):
    """A SwiGLU shared expert (Ws1 gate, Ws3 up).  When h divides h_s it runs as h_s / h
    always-on groups of the routed launches (the first two cases: the gate chunks of Ws1
    on the pair's first CTA, those of Ws3 on the second); otherwise as its own GEMMs,
    the up-projection through the gather warps with contiguous rows, then lambda times
    its down-projection as the first value of the fp32 accumulator."""
    assert moevie.moevie_shared_groups(T, d, E, k, h, hs) == (hs // h if hs % h == 0 else 0)
    cfg = workloads.small_config(T, d, E, k, h, h_s=hs, lam=0.5, seed=T + hs, act="swiglu")
    lay = workloads.make_layer(cfg)
    y, rt = _run(lay)
    want, oidx, _, _ = oracle.forward_tokens(lay.x, lay.Wr, lay.b, lay.W1, lay.W2, k, lay.Ws1, lay.Ws2,
                                             cfg.lam, W3=lay.W3, Ws3=lay.Ws3)
    assert np.array_equal(rt["idx"], oidx)
    assert_close(y, want)
