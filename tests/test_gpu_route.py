"""Router parity (Eqs. 1, 7, 4-5): GPU selection bit-exact against the fp64 oracle,
gates within fp32 rounding, through the C ABI."""
import numpy as np
import pytest
import torch

import oracle
import workloads
from paper_2608_17402_gb300 import moevie
from tests._gpu import MARGIN_PINNED, check_status, dev, dev_bf16

pytestmark = pytest.mark.gpu


def _route_case(x, Wr, b, k):
    T, d = x.shape
    E = Wr.shape[1]
    ws = moevie.Workspace(T, d, E, k, 16)
    idx, gate = moevie.moevie_route(dev_bf16(x), dev(Wr), dev(b), k, ws)
    nfb = moevie.moevie_test_fallback_count(ws)
    check_status(ws)
    return idx.cpu().numpy(), gate.cpu().numpy().astype(np.float64), nfb


def _check_against_oracle(x, Wr, b, k):
    idx, gate, nfb = _route_case(x, Wr, b, k)
    oidx, ogate, margin = oracle.route(x, Wr, b, k)
    pinned = margin > MARGIN_PINNED
    assert pinned.mean() > 0.999, "too many oracle near-ties to pin the selection"
    assert np.array_equal(idx[pinned], oidx[pinned]), np.argwhere(np.any(idx != oidx, axis=1))[:8]
    np.testing.assert_allclose(gate, ogate, rtol=0, atol=1e-5)
    assert np.all(np.diff(idx, axis=1) > 0)
    return nfb


@pytest.mark.parametrize("T,d,E,k", [(1, 16, 8, 2), (37, 64, 16, 2), (129, 128, 64, 8),
                                     (200, 96, 1, 1), (64, 32, 4, 4), (50, 64, 1024, 4),
                                     (300, 256, 256, 8), (77, 48, 33, 5)])
def test_route_small_shapes(T, d, E, k):
    rng = np.random.default_rng(T * 7 + E)
    x = workloads.f32_to_bf16_bits(rng.standard_normal((T, d)).astype(np.float32))
    Wr = (rng.standard_normal((d, E)) * 0.02).astype(np.float32)
    b = rng.uniform(-0.1, 0.1, E).astype(np.float32)
    _check_against_oracle(x, Wr, b, k)


def test_route_exact_ties_go_to_lower_id():
    """Duplicated W_r columns with equal bias give exactly equal keys; the fast path
    cannot certify them and the exact re-decision must pick the lower id."""
    rng = np.random.default_rng(5)
    T, d, E, k = 256, 64, 16, 3
    x = workloads.f32_to_bf16_bits(rng.standard_normal((T, d)).astype(np.float32))
    Wr = (rng.standard_normal((d, E)) * 0.3).astype(np.float32)
    b = rng.uniform(-0.1, 0.1, E).astype(np.float32)
    for a, c in [(1, 9), (4, 5), (0, 15)]:
        Wr[:, c] = Wr[:, a]
        b[c] = b[a]
    idx, gate, nfb = _route_case(x, Wr, b, k)
    oidx, ogate, _ = oracle.route(x, Wr, b, k)
    assert np.array_equal(idx, oidx)
    assert nfb > 0
    np.testing.assert_allclose(gate, ogate, rtol=0, atol=1e-5)


def test_route_exact_redecision_stress():
    """Inputs that send almost every token through the exact re-decision and stress its
    long accumulator: two rows whose products cancel exactly (x[:, 1] = x[:, 0],
    W_r[1] = -W_r[0] = 1024 r), which makes the fast-path error bound large; rows of
    tiny (2^-40) and subnormal weights, whose products fall far below the others; and a
    near-duplicate column whose logit differs from its twin by x[:, 10] 2^-20 only."""
    rng = np.random.default_rng(12)
    T, d, E, k = 256, 96, 24, 4
    xf = rng.standard_normal((T, d)).astype(np.float32)
    x = workloads.f32_to_bf16_bits(xf)
    x[:, 1] = x[:, 0]
    Wr = (rng.standard_normal((d, E)) * 0.05).astype(np.float32)
    Wr[0] = (1024.0 * rng.uniform(0.5, 1.0, E) * rng.choice([-1.0, 1.0], E)).astype(np.float32)
    Wr[1] = -Wr[0]
    Wr[2:6] *= np.float32(2.0 ** -40)
    Wr[6:10] = (rng.standard_normal((4, E)) * 1e-40).astype(np.float32)   # subnormal fp32
    Wr[:, 17] = Wr[:, 3]
    Wr[10, 17] = Wr[10, 3] + np.float32(2.0 ** -20)
    b = rng.uniform(-0.1, 0.1, E).astype(np.float32)
    b[17] = b[3]
    nfb = _check_against_oracle(x, Wr, b, k)
    assert nfb > T // 2, nfb


def test_route_bias_only():
    """W_r = 0: every key is 1/2 + b; ties in b resolve to the lower id; gates 1/k."""
    T, d, E, k = 40, 32, 12, 4
    x = workloads.f32_to_bf16_bits(np.random.default_rng(1).standard_normal((T, d)).astype(np.float32))
    Wr = np.zeros((d, E), np.float32)
    b = np.array([0.0625, -0.5, 0.25, 0.25, 0.0, 0.25, 0.125, 0.25, -0.25, 0.0625, 0.5, 0.0],
                 np.float32)
    idx, gate, _ = _route_case(x, Wr, b, k)
    want = np.array([2, 3, 5, 10])   # 0.5 (id 10), then 0.25 at ids 2, 3, 5 (7 left out)
    assert np.all(idx == want)
    np.testing.assert_allclose(gate, 0.25, rtol=0, atol=1e-7)


@pytest.mark.parametrize("name", ["c0", "c1", "c2", "c3", "c4"])
def test_route_full_configs(name):
    lay = workloads.make_layer(workloads.CONFIGS[name])
    nfb = _check_against_oracle(lay.x, lay.Wr, lay.b, lay.cfg.k)
    print(f"{name}: {nfb} of {lay.cfg.T} tokens re-decided exactly")


def _split_hi_mid(Wr):
    """W_r's two leading bf16 pieces, hi = bf16(w) and mid = bf16(w - hi) (round to
    nearest even), summed in fp32 (exact), and the left-out remainder lo = w - hi - mid."""
    hi = workloads.bf16_bits_to_f32(workloads.f32_to_bf16_bits(Wr))
    r1 = (Wr - hi).astype(np.float32)
    mid = workloads.bf16_bits_to_f32(workloads.f32_to_bf16_bits(r1))
    return (hi + mid).astype(np.float32), (r1 - mid).astype(np.float32)


def _logit_error_units(x, Wr):
    """The fast logits' fp32 accumulation error, max over the layer of |s_fast - x . (hi +
    mid)| in units of 2^-24 |x_t| (|W_r[:, e]| + |lo_e|); also checks that the whole error
    |s_fast - s| stays inside the bound the router certifies with (its accumulation term
    with the constant ROUTE_TAU_C = 128, plus |x_t| |lo_e| for the left-out piece)."""
    T, d = x.shape
    E = Wr.shape[1]
    ws = moevie.Workspace(T, d, E, 1, 16)
    s = moevie.moevie_test_route_logits(dev_bf16(x), dev(Wr), ws).cpu().numpy().astype(np.float64)
    check_status(ws)
    w2, lo = _split_hi_mid(Wr)
    s2 = oracle.logits(x, w2)
    so = oracle.logits(x, Wr)
    xn = np.linalg.norm(workloads.bf16_bits_to_f32(x).astype(np.float64), axis=1)[:, None]
    wn = np.linalg.norm(Wr.astype(np.float64), axis=0)[None, :]
    ln = np.linalg.norm(lo.astype(np.float64), axis=0)[None, :]
    unit = 2.0 ** -24 * xn * (wn + ln)
    bound = 128 * unit + xn * ln
    assert np.all(np.abs(s - so) <= bound), float((np.abs(s - so) / bound).max())
    return float((np.abs(s - s2) / unit).max())


@pytest.mark.parametrize("name", ["c0", "c1", "c2", "c3", "c4", "s1", "pB", "pL", "pH"])
def test_fast_logit_error_within_bound(name):
    """The tensor-core logits' accumulation error stays far inside the bound the router
    certifies with (ROUTE_TAU_C = 128 units of 2^-24 |x_t| (|W_r[:, e]| + |lo_e|)):
    measured max below 1/4 of it over every token of every layer workload."""
    lay = workloads.make_layer(workloads.CONFIGS[name])
    r = _logit_error_units(lay.x, lay.Wr)
    print(f"{name}: max accumulation error {r:.3f} units of 2^-24 |x_t| (|W_r[:, e]| + |lo_e|)")
    assert r < 128 / 4


@pytest.mark.parametrize("E", [64, 256])
@pytest.mark.parametrize("pattern", ["same_sign", "alternating", "random_sign"])
def test_fast_logit_error_adversarial(pattern, E):
    """Inputs built to maximise the fp32 accumulation error of the logits at the
    stress layer's width (d = 1664): every product x_i w_i of nearly the same
    magnitude (x_i = +-1, w_i = 0.02 (1 + small) with all 24 significand bits of w in
    use, so all bf16 pieces of W_r are non-zero), with the signs all equal (the
    partial sums grow to d |x_i w_i|), alternating, or random.  E = 64 puts the two
    pieces side by side (summed in the epilogue), E = 256 one after another along K.
    The accumulation error must stay below 1/4 of the certified bound."""
    rng = np.random.default_rng(E + len(pattern))
    T, d = 256, 1664
    if pattern == "same_sign":
        xs = np.ones((T, d), np.float32)
    elif pattern == "alternating":
        xs = np.tile(np.array([1.0, -1.0], np.float32), (T, d // 2))
    else:
        xs = rng.choice(np.array([1.0, -1.0], np.float32), (T, d))
    x = workloads.f32_to_bf16_bits(xs)
    Wr = (0.02 * (1.0 + rng.uniform(0.0, 2.0 ** -6, (d, E)))).astype(np.float32)
    r = _logit_error_units(x, Wr)
    print(f"{pattern}, E={E}: max accumulation error {r:.3f} units of 2^-24 |x_t| (|W_r[:, e]| + |lo_e|)")
    assert r < 128 / 4
