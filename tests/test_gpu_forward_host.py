"""moevie_moe_forward_host: the layer from host memory to host memory over contiguous
token chunks, the copies overlapped with the compute.  Tokens are independent (Eqs. 4-7
act per token), so every chunk count gives the oracle's routing and outputs: small
layers against the oracle on every token (ragged last chunks, more chunks than tokens,
one chunk), the image layer with a shared expert against the one-call device forward,
and the argument checks."""
import numpy as np
import pytest
import torch

import oracle
import workloads
from paper_2608_17402_gb300 import moevie
from tests._gpu import assert_close, check_status, layer_to_device, to_np_f64

pytestmark = pytest.mark.gpu


def _host(bits, pinned=True):
    t = torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16)
    return t.pin_memory() if pinned else t.clone()


def _run_host(lay, chunks, pinned=True):
    c = lay.cfg
    x, W = layer_to_device(lay)
    Tc = -(-c.T // chunks)
    ws = moevie.Workspace(Tc, c.d, c.E, c.k, c.h, c.h_s)
    x_host = _host(lay.x, pinned)
    y_host = torch.empty_like(x_host)
    if pinned:
        y_host = y_host.pin_memory()
    xd, yd = torch.empty_like(x), torch.empty_like(x)
    moevie.moevie_moe_forward_host(W, x_host, y_host, xd, yd, ws, chunks)
    torch.cuda.synchronize()
    check_status(ws)
    return y_host.float().numpy().astype(np.float64)


@pytest.mark.parametrize("T,chunks,hs", [
    (300, 4, 0), (257, 16, 96), (20, 16, 0), (64, 1, 96), (1, 3, 0), (513, 5, 192),
])
def test_forward_host_small(T, chunks, hs):
    cfg = workloads.small_config(T, 128, 8, 2, 96, h_s=hs, lam=0.5 if hs else 1.0, seed=T + 3 * chunks)
    lay = workloads.make_layer(cfg)
    got = _run_host(lay, chunks)
    want, *_ = oracle.forward_tokens(lay.x, lay.Wr, lay.b, lay.W1, lay.W2, cfg.k, lay.Ws1, lay.Ws2, cfg.lam)
    assert_close(got, want)


def test_forward_host_pageable():
    """Host buffers that are not pinned: the copies are then synchronous, the result the same."""
    cfg = workloads.small_config(300, 128, 8, 2, 96, seed=9)
    lay = workloads.make_layer(cfg)
    got = _run_host(lay, 3, pinned=False)
    want, *_ = oracle.forward_tokens(lay.x, lay.Wr, lay.b, lay.W1, lay.W2, cfg.k)
    assert_close(got, want)


def test_forward_host_image_layer_matches_device_forward():
    """The image layer with its shared expert (T = 8192) in 4 chunks against one
    device-resident forward of all 8192 tokens: the same routing per token, outputs within
    the y accumulator's rounding (its fp32 sums are formed in another order)."""
    lay = workloads.make_layer(workloads.CONFIGS["c1"])
    c = lay.cfg
    x, W = layer_to_device(lay)
    ws = moevie.Workspace(c.T, c.d, c.E, c.k, c.h, c.h_s)
    y_one = to_np_f64(moevie.moevie_moe_forward(W, x, ws))
    check_status(ws)
    got = _run_host(lay, 4)
    assert_close(got, y_one)
    # outputs differ from the one-call forward only by fp32 summation order and the
    # bf16 rounding of y: at most a few bf16 ulps
    assert np.max(np.abs(got - y_one)) <= 4 * 2.0 ** -8 * np.max(np.abs(y_one))


def test_forward_host_rejects_bad_arguments():
    cfg = workloads.small_config(64, 64, 4, 2, 64, seed=1)
    lay = workloads.make_layer(cfg)
    x, W = layer_to_device(lay)
    x_host = _host(lay.x)
    y_host = torch.empty_like(x_host).pin_memory()
    xd, yd = torch.empty_like(x), torch.empty_like(x)
    n0 = moevie.moevie_launch_count()
    ws = moevie.Workspace(64, 64, 4, 2, 64)
    for chunks, code in ((0, 2), (moevie.HOST_MAX_CHUNKS + 1, 2)):
        with pytest.raises(moevie.MoevieError) as e:
            moevie.moevie_moe_forward_host(W, x_host, y_host, xd, yd, ws, chunks)
        assert e.value.code == code
    small = moevie.Workspace(8, 64, 4, 2, 64)   # room for 8 tokens, chunks of 32 asked
    with pytest.raises(moevie.MoevieError) as e:
        moevie.moevie_moe_forward_host(W, x_host, y_host, xd, yd, small, 2)
    assert e.value.code == 3
    assert moevie.moevie_launch_count() == n0
