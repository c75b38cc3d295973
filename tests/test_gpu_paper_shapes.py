"""The paper's own MoE-ViE-B / L / H layers (App. D, model table: 31 routed + 1 shared
SwiGLU experts of width 512 / 684 / 854, k = 3 / 3 / 7) and hidden widths that are not
multiples of 8 or 16, through moevie_moe_forward against the oracle: routing
bit-exact, outputs within rel-L2 1e-2 and max |err| 5e-2 * RMS.

W1, W3, Ws1 and Ws3 travel with rows padded to a multiple of 8 elements; the weight
tensor maps cover the first h columns only, so the up-projection's last column tile and
the down-projection's last K block read zeros past h."""
import numpy as np
import pytest
import torch

import oracle
import workloads
from paper_2608_17402_gb300 import moevie
from tests._gpu import (MARGIN_PINNED, assert_close, check_status, layer_to_device,
                        stratified_tokens, to_np_f64, workspace_for)

pytestmark = pytest.mark.gpu


def _run(lay, poison_pad=False):
    x, W = layer_to_device(lay)
    if poison_pad:   # the pad columns must never be read: fill them with NaN
        for name in ("W1", "W3", "Ws1", "Ws3"):
            w = getattr(W, name)
            if w is not None and w.shape[-1] % 8:
                h = w.shape[-1]
                full = w.as_strided(w.shape[:-1] + (moevie.row_ld(h),), w.stride())
                full[..., h:] = float("nan")
    ws = workspace_for(lay)
    y, rt = moevie.moevie_moe_forward(W, x, ws, routing=True)
    check_status(ws)
    return to_np_f64(y), {k: v.cpu().numpy() for k, v in rt.items()}


def _want(lay, tokens=None):
    c = lay.cfg
    return oracle.forward_tokens(lay.x, lay.Wr, lay.b, lay.W1, lay.W2, c.k, lay.Ws1, lay.Ws2, c.lam,
                                 tokens=tokens, W3=lay.W3, Ws3=lay.Ws3)


@pytest.mark.parametrize("T,d,E,k,h,hs,act", [
    (300, 256, 31, 3, 684, 684, "swiglu"),   # L widths at a small T and d (shared: one always-on group)
    (257, 128, 31, 7, 854, 854, "swiglu"),   # H widths
    (130, 192, 8, 2, 684, 0, "gelu"),
    (200, 128, 8, 3, 100, 300, "gelu"),      # h % 8 == 4; the shared expert runs as its own GEMMs
    (64, 64, 4, 2, 13, 5, "swiglu"),         # odd widths below one 8-column output group
])
def test_ragged_hidden_width_small(T, d, E, k, h, hs, act):
    cfg = workloads.small_config(T, d, E, k, h, h_s=hs, lam=0.5 if hs else 1.0, seed=T + h, act=act)
    lay = workloads.make_layer(cfg)
    y, rt = _run(lay, poison_pad=True)
    want, oidx, _, _ = _want(lay)
    assert np.array_equal(rt["idx"], oidx)
    assert_close(y, want)


@pytest.mark.parametrize("name", ["pB", "pL", "pH"])
def test_paper_layer_sampled(name):
    """Full-size layer, all routing outputs, and at least 1024 output rows chosen by
    stratum (as for the video and stress layers).  The shared expert (h_s = h) rides
    in the routed launches as one always-on group."""
    lay = workloads.make_layer(workloads.CONFIGS[name])
    c = lay.cfg
    assert moevie.moevie_shared_groups(c.T, c.d, c.E, c.k, c.h, c.h_s) == 1
    y, rt = _run(lay)
    oidx, ogate, margin = oracle.route(lay.x, lay.Wr, lay.b, c.k)
    assert (margin > MARGIN_PINNED).all()
    assert np.array_equal(rt["idx"], oidx)
    np.testing.assert_allclose(rt["gate"], ogate, rtol=0, atol=1e-5)
    oc, oo, op, oi = oracle.permute(oidx, c.E)
    for key, want in (("counts", oc), ("offsets", oo), ("perm", op), ("inv", oi)):
        assert np.array_equal(rt[key], want), key
    toks, strata = stratified_tokens(c.T, c.k, oc, oo, op, n_random=512, seed=2)
    assert toks.size >= 1024, toks.size
    want, *_ = _want(lay, tokens=toks)
    rel, mx = assert_close(y[toks], want)
    print(f"{name}: {toks.size} tokens by stratum {strata}, rel-L2 {rel:.2e}, max|err|/RMS {mx:.2e}")


def test_unpadded_weights_are_rejected():
    """A dense [E, d, h] W1 with h % 8 != 0 does not have the row stride the entry
    points take: the binding raises before any launch."""
    cfg = workloads.small_config(16, 64, 4, 2, 20)
    lay = workloads.make_layer(cfg)
    x, W = layer_to_device(lay)
    W.W1 = W.W1.contiguous()
    ws = workspace_for(lay)
    with pytest.raises(ValueError):
        moevie.moevie_moe_forward(W, x, ws)
