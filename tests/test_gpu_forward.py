"""Whole-layer parity (Eqs. 1, 4-7; Algorithm 1) of moevie_moe_forward against the
oracle: routing bit-exact, outputs within rel-L2 1e-2 and max |err| 5e-2 * RMS.

Small layers and the batch-1 / image layers are compared on every token; the
video (T = 32768) and stress (T = 65536) layers, in the launch configuration the
benchmark times, are compared on all routing outputs and on a sample of output
rows that the oracle computes token by token."""
import numpy as np
import pytest

import oracle
import workloads
from paper_2608_17402_gb300 import moevie
from tests._gpu import (MARGIN_PINNED, assert_close, check_status, layer_to_device,
                        stratified_tokens, to_np_f64, workspace_for)

pytestmark = pytest.mark.gpu


def _run(lay):
    x, W = layer_to_device(lay)
    ws = workspace_for(lay)
    y, rt = moevie.moevie_moe_forward(W, x, ws, routing=True)
    check_status(ws)
    return to_np_f64(y), {k: v.cpu().numpy() for k, v in rt.items()}


def _check_routing(lay, rt, tokens=None):
    c = lay.cfg
    oidx, ogate, margin = oracle.route(lay.x, lay.Wr, lay.b, c.k)
    pinned = margin > MARGIN_PINNED
    assert pinned.all(), f"{(~pinned).sum()} oracle near-ties"
    assert np.array_equal(rt["idx"], oidx)
    np.testing.assert_allclose(rt["gate"], ogate, rtol=0, atol=1e-5)
    oc, oo, op, oi = oracle.permute(oidx, c.E)
    assert np.array_equal(rt["counts"], oc)
    assert np.array_equal(rt["offsets"], oo)
    assert np.array_equal(rt["perm"], op)
    assert np.array_equal(rt["inv"], oi)
    return oc


@pytest.mark.parametrize("T,d,E,k,h,hs", [
    (1, 64, 4, 2, 64, 0), (130, 128, 8, 2, 128, 0), (257, 256, 16, 4, 416, 0),
    (200, 128, 8, 8, 64, 0), (100, 96, 4, 1, 48, 0), (300, 128, 16, 4, 96, 256),
    # h divides h_s: the shared expert runs as h_s / h always-on groups of the grouped GEMMs
    (1, 64, 4, 2, 64, 64), (300, 128, 16, 4, 128, 256), (257, 64, 8, 2, 64, 192),
])
def test_forward_small(T, d, E, k, h, hs):
    cfg = workloads.small_config(T, d, E, k, h, h_s=hs, lam=0.5 if hs else 1.0, seed=T + h)
    lay = workloads.make_layer(cfg)
    y, rt = _run(lay)
    _check_routing(lay, rt)
    want, *_ = oracle.forward_tokens(lay.x, lay.Wr, lay.b, lay.W1, lay.W2, k, lay.Ws1, lay.Ws2, cfg.lam)
    assert_close(y, want)


@pytest.mark.parametrize("name", ["c0", "c1", "c2"])
def test_forward_full_config(name):
    lay = workloads.make_layer(workloads.CONFIGS[name])
    y, rt = _run(lay)
    _check_routing(lay, rt)
    c = lay.cfg
    want, *_ = oracle.forward_tokens(lay.x, lay.Wr, lay.b, lay.W1, lay.W2, c.k, lay.Ws1, lay.Ws2, c.lam)
    rel, mx = assert_close(y, want)
    print(f"{name}: rel-L2 {rel:.2e}, max|err|/RMS {mx:.2e}")


@pytest.mark.parametrize("name", ["c3", "c4"])
def test_forward_large_config_stratified(name):
    """The video and stress layers in the launch configuration the benchmark times:
    every routing output bit-exact, and at least 1024 output rows against the oracle,
    chosen by stratum (every expert's last m-tile, the hot expert's tile boundaries,
    both sides of every possible token-band boundary, the least loaded experts, and a
    uniform sample)."""
    lay = workloads.make_layer(workloads.CONFIGS[name])
    y, rt = _run(lay)
    counts = _check_routing(lay, rt)
    c = lay.cfg
    assert (counts == 0).sum() >= 3, "the skewed layer must keep its empty experts"
    toks, strata = stratified_tokens(c.T, c.k, counts, rt["offsets"], rt["perm"])
    assert toks.size >= 1024, toks.size
    want, *_ = oracle.forward_tokens(lay.x, lay.Wr, lay.b, lay.W1, lay.W2, c.k, lay.Ws1, lay.Ws2,
                                     c.lam, tokens=toks)
    rel, mx = assert_close(y[toks], want)
    print(f"{name}: {toks.size} tokens by stratum {strata}, rel-L2 {rel:.2e}, max|err|/RMS {mx:.2e}")


def test_forward_is_deterministic_in_routing_and_repeatable():
    lay = workloads.make_layer(workloads.CONFIGS["c0"])
    y1, r1 = _run(lay)
    y2, r2 = _run(lay)
    for k in r1:
        assert np.array_equal(r1[k], r2[k]), k
    assert_close(y2, y1, "repeat")


def test_forward_empty_batch_launches_nothing():
    """T = 0 is a valid call: status OK, no kernel launched, nothing written."""
    cfg = workloads.small_config(4, 64, 4, 2, 64)
    lay = workloads.make_layer(cfg)
    x, W = layer_to_device(lay)
    ws = workspace_for(lay)
    n0 = moevie.moevie_launch_count()
    y = moevie.moevie_moe_forward(W, x[:0], ws)
    assert y.shape == (0, cfg.d)
    assert moevie.moevie_launch_count() == n0
    check_status(ws)


def test_forward_banded_with_shared_expert_sampled():
    """A layer whose fp32 accumulator exceeds 64 MiB (band-ordered down-projection)
    with a shared expert of width 2h: the shared expert runs as its own GEMMs, its
    hidden [T, h_s] in the workspace bytes that the always-on groups use otherwise."""
    T, d, E, k, h, hs = 16400, 1024, 16, 2, 256, 512
    assert moevie.moevie_shared_groups(T, d, E, k, h, hs) == 0
    assert moevie.moevie_shared_groups(T // 2, d, E, k, h, hs) == 2
    cfg = workloads.small_config(T, d, E, k, h, h_s=hs, lam=0.75, seed=7)
    lay = workloads.make_layer(cfg)
    y, rt = _run(lay)
    _check_routing(lay, rt)
    rng = np.random.default_rng(1)
    toks = np.unique(np.concatenate([[0, T - 1], rng.choice(T, 48, replace=False)])).astype(np.int32)
    want, *_ = oracle.forward_tokens(lay.x, lay.Wr, lay.b, lay.W1, lay.W2, k, lay.Ws1, lay.Ws2,
                                     cfg.lam, tokens=toks)
    assert_close(y[toks], want)
