"""Pins of the fp64 CPU oracle against facts that do not come from the oracle.

The paper prints no worked numerical example of the layer, so each pin is a
closed form, an invariant, an exhaustive brute force on tiny inputs, an
arbitrary-precision evaluation, or a special case that reduces to a library
routine (torch / numpy / scipy).  Between them a dropped term, a wrong sign or
index, or a transposed operand anywhere in the oracle fails at least one test:

* logits (Eq. 1)                    exact rational sums (``fractions.Fraction``)
* selection + tie rule (Eq. 7)      brute force over all k-subsets, keys at 60 digits
* gates (Eqs. 4-5)                  60-digit evaluation; W_r = 0 gives exactly 1/k
* permutation (Algorithm 1, ph. 1)  numpy stable argsort / bincount / cumsum,
                                    permutation invariants, round trip
* expert FFN (E=1, k=1)             torch fp64 matmul + GELU (erf form)
* combine + gates (Eq. 6)           dense masked sum over all experts (torch einsum)
* k = E with W_r = 0                mean of all experts
* shared expert                     routed weights zero -> lambda * shared expert
* token order                       permuting tokens permutes the outputs
"""
import itertools
import math
from fractions import Fraction

import mpmath
import numpy as np
import pytest
import scipy.special
import torch

import oracle
import workloads
from workloads import bf16_bits_to_f32, f32_to_bf16_bits

mpmath.mp.dps = 60


def _rng(seed):
    return np.random.default_rng(1000 + seed)


def _bf16(a):
    return f32_to_bf16_bits(np.asarray(a, np.float32))


def _exact_logits(x_bits, Wr):
    """Exact rational logits."""
    xf = bf16_bits_to_f32(x_bits).astype(np.float64)
    T, d = xf.shape
    E = Wr.shape[1]
    out = [[sum((Fraction(float(xf[t, i])) * Fraction(float(Wr[i, e])) for i in range(d)), Fraction(0))
             for e in range(E)] for t in range(T)]
    return out


def _brute_topk(keys, k):
    """Lexicographically smallest sorted id tuple among the k-subsets whose every
    key is >= every key left out (the lowest-id tie rule, stated as a set)."""
    E = len(keys)
    best = None
    for S in itertools.combinations(range(E), k):
        inside = min(keys[e] for e in S)
        outside = max((keys[e] for e in range(E) if e not in S), default=None)
        if outside is not None and inside < outside:
            continue
        if best is None or S < best:
            best = S
    return best


def _mp_key(s_frac, b):
    s = mpmath.mpf(s_frac.numerator) / s_frac.denominator
    return 1 / (1 + mpmath.exp(-s)) + mpmath.mpf(float(b))


# ------------------------------------------------------------------ logits

@pytest.mark.parametrize("seed", range(6))
def test_logits_match_exact_rationals(seed):
    rng = _rng(seed)
    T, d, E = 5, 7, 3          # d != E: a transposed W_r index cannot pass
    x = _bf16(rng.standard_normal((T, d)))
    Wr = (rng.standard_normal((d, E)) * 0.3).astype(np.float32)
    s = oracle.logits(x, Wr)
    ex = _exact_logits(x, Wr)
    xf = bf16_bits_to_f32(x).astype(np.float64)
    for t in range(T):
        for e in range(E):
            bound = d * 2.0 ** -53 * float(np.sum(np.abs(xf[t] * Wr[:, e])))
            assert abs(s[t, e] - float(ex[t][e])) <= bound + 1e-300


# --------------------------------------------------------------- selection

@pytest.mark.parametrize("seed", range(40))
def test_select_bias_only_brute_force_with_ties(seed):
    """W_r = 0: s = 0, sigmoid = 1/2 exactly, key = 1/2 + b.  b on a dyadic grid
    makes exact ties common.  Selection must be the brute-force top-k with the
    lowest-id rule, and every gate exactly 1/k."""
    rng = _rng(seed)
    E = int(rng.integers(1, 9))
    k = int(rng.integers(1, min(E, 4) + 1))
    T, d = 4, 3
    x = _bf16(rng.standard_normal((T, d)))
    Wr = np.zeros((d, E), np.float32)
    b = rng.choice(np.array([-0.5, -0.25, 0.0, 0.25, 0.5], np.float32), size=E).astype(np.float32)
    idx, gate, margin = oracle.route(x, Wr, b, k)
    want = _brute_topk([0.5 + float(v) for v in b], k)
    for t in range(T):
        assert tuple(idx[t]) == want
        assert np.all(gate[t] == 1.0 / k)
    assert len(set(want)) == k


@pytest.mark.parametrize("seed", range(25))
def test_select_brute_force_high_precision(seed):
    """General logits: keys evaluated at 60 digits from exact rational logits,
    brute force over all subsets.  Duplicated W_r columns with equal bias make
    exact ties that must go to the lower id."""
    rng = _rng(100 + seed)
    E = int(rng.integers(2, 9))
    k = int(rng.integers(1, min(E, 4) + 1))
    T, d = 6, int(rng.integers(1, 6))
    x = _bf16(rng.standard_normal((T, d)))
    Wr = (rng.standard_normal((d, E)) * 0.8).astype(np.float32)
    b = (rng.uniform(-0.1, 0.1, size=E)).astype(np.float32)
    if E >= 3 and seed % 2 == 0:             # exact tie between experts 0 and E-1 (or a pair)
        a, c = sorted(rng.choice(E, size=2, replace=False))
        Wr[:, c] = Wr[:, a]
        b[c] = b[a]
    idx, gate, margin = oracle.route(x, Wr, b, k)
    ex = _exact_logits(x, Wr)
    for t in range(T):
        keys = [_mp_key(ex[t][e], b[e]) for e in range(E)]
        want = _brute_topk(keys, k)
        assert tuple(idx[t]) == want, (t, keys, idx[t], want)
        sig = [1 / (1 + mpmath.exp(-mpmath.mpf(ex[t][e].numerator) / ex[t][e].denominator)) for e in want]
        tot = sum(sig)
        for j, e in enumerate(want):
            assert abs(gate[t, j] - float(sig[j] / tot)) <= 4e-16
        left = [keys[e] for e in range(E) if e not in want]
        if left:
            m = float(min(keys[e] for e in want) - max(left))
            assert abs(margin[t] - m) <= 1e-15
        else:
            assert margin[t] == math.inf


def test_gates_sum_to_one_and_bias_excluded():
    rng = _rng(7)
    T, d, E, k = 64, 32, 16, 4
    x = _bf16(rng.standard_normal((T, d)))
    Wr = (rng.standard_normal((d, E)) * 0.2).astype(np.float32)
    b = rng.uniform(-0.1, 0.1, size=E).astype(np.float32)
    idx, gate, _ = oracle.route(x, Wr, b, k)
    assert np.all(np.abs(gate.sum(1) - 1.0) <= 1e-15)
    assert np.all((gate > 0) & (gate < 1))
    # changing b may change the selection but never the gate formula: with the same
    # selection forced (b shifted uniformly), gates are unchanged
    idx2, gate2, _ = oracle.route(x, Wr, (b + np.float32(0.0625)).astype(np.float32), k)
    same = np.all(idx == idx2, axis=1)
    assert same.any()
    assert np.array_equal(gate[same], gate2[same])
    # ids ascending and distinct
    assert np.all(np.diff(idx, axis=1) > 0)


# -------------------------------------------------------------- permutation

def _random_routing(rng, T, E, k, empty=()):
    allowed = np.array([e for e in range(E) if e not in set(empty)])
    idx = np.stack([np.sort(rng.choice(allowed, size=k, replace=False)) for _ in range(T)]).astype(np.int32)
    return idx


@pytest.mark.parametrize("T,E,k,empty", [(1, 1, 1, ()), (37, 5, 2, (1,)), (200, 16, 4, (0, 15)),
                                         (129, 8, 8, ()), (0, 4, 2, ())])
def test_permute_against_stable_argsort(T, E, k, empty):
    rng = _rng(T + E + k)
    idx = _random_routing(rng, T, E, k, empty) if T else np.zeros((0, k), np.int32)
    counts, offsets, perm, inv = oracle.permute(idx, E)
    flat = idx.ravel()
    # library routines: bincount / cumsum / stable argsort
    assert np.array_equal(counts, np.bincount(flat, minlength=E))
    assert np.array_equal(offsets, np.concatenate([[0], np.cumsum(np.bincount(flat, minlength=E))]))
    assert np.array_equal(perm, np.argsort(flat, kind="stable"))
    # invariants
    assert counts.sum() == T * k and offsets[-1] == T * k
    assert np.array_equal(np.sort(perm), np.arange(T * k))
    assert np.array_equal(inv[perm], np.arange(T * k))
    for e in range(E):
        seg = perm[offsets[e]:offsets[e + 1]]
        assert np.all(flat[seg] == e)
        assert np.all(np.diff(seg) > 0)
    for e in empty:
        assert counts[e] == 0
    # round trip: unpermute(permute(v)) == v
    v = rng.standard_normal(T * k)
    assert np.array_equal(v[perm][inv], v)


# ------------------------------------------------------------ expert FFN

def _t64(bits):
    return torch.from_numpy(bf16_bits_to_f32(bits).astype(np.float64))


def _gelu_t(u):
    return torch.nn.functional.gelu(u, approximate="none")


@pytest.mark.parametrize("h", [40, 13])
def test_single_expert_is_dense_mlp(h):
    """E = 1, k = 1: the layer is GELU(x W1) W2 (gate 1); d != h so a transposed
    W1 or W2 index cannot pass (h = 13: a width that is not a multiple of 8)."""
    rng = _rng(11)
    T, d = 9, 24
    x = _bf16(rng.standard_normal((T, d)))
    W1 = _bf16(rng.standard_normal((1, d, h)) / np.sqrt(d))
    W2 = _bf16(rng.standard_normal((1, h, d)) / np.sqrt(h))
    Wr = (rng.standard_normal((d, 1)) * 0.02).astype(np.float32)
    b = np.zeros(1, np.float32)
    y, idx, gate, _ = oracle.forward_tokens(x, Wr, b, W1, W2, 1)
    want = _gelu_t(_t64(x) @ _t64(W1[0])) @ _t64(W2[0])
    assert np.all(idx == 0) and np.all(gate == 1.0)
    np.testing.assert_allclose(y, want.numpy(), rtol=1e-12, atol=1e-12)


def test_gelu_against_normal_cdf():
    """GELU(u) = u Phi(u) (scipy ndtr) and GELU(u) - GELU(-u) = u, through a 1x1 expert."""
    us = np.array([-6.0, -2.5, -1.0, -0.375, 0.0, 0.5, 1.0, 3.0, 8.0], np.float32)
    T = us.size
    x = _bf16(us[:, None])
    W1 = _bf16(np.ones((1, 1, 1)))
    W2 = _bf16(np.ones((1, 1, 1)))
    y, *_ = oracle.forward_tokens(x, np.zeros((1, 1), np.float32), np.zeros(1, np.float32), W1, W2, 1)
    u = bf16_bits_to_f32(x)[:, 0].astype(np.float64)
    # the erf form 0.5 u (1 + erf(u / sqrt 2)) loses relative accuracy where 1 + erf
    # cancels (u << 0); its absolute error stays below ~|u| * eps
    err = np.abs(y[:, 0] - u * scipy.special.ndtr(u))
    assert np.all(err <= 1e-14 * np.abs(u * scipy.special.ndtr(u)) + 4 * np.abs(u) * 2.0 ** -53)
    xm = _bf16(-us[:, None])
    ym, *_ = oracle.forward_tokens(xm, np.zeros((1, 1), np.float32), np.zeros(1, np.float32), W1, W2, 1)
    np.testing.assert_allclose(y[:, 0] - ym[:, 0], u, rtol=0, atol=1e-15)


def _layer(rng, T, d, E, k, h, hs=0, wr_scale=0.3):
    x = _bf16(rng.standard_normal((T, d)))
    Wr = (rng.standard_normal((d, E)) * wr_scale).astype(np.float32)
    b = rng.uniform(-0.1, 0.1, size=E).astype(np.float32)
    W1 = _bf16(rng.standard_normal((E, d, h)) / np.sqrt(d))
    W2 = _bf16(rng.standard_normal((E, h, d)) / np.sqrt(h))
    Ws1 = Ws2 = None
    if hs:
        Ws1 = _bf16(rng.standard_normal((d, hs)) / np.sqrt(d))
        Ws2 = _bf16(rng.standard_normal((hs, d)) / np.sqrt(hs))
    return x, Wr, b, W1, W2, Ws1, Ws2


def _all_experts_t(x, W1, W2):
    xt = _t64(x)
    hid = _gelu_t(torch.einsum("td,edh->teh", xt, _t64(W1)))
    return torch.einsum("teh,ehd->ted", hid, _t64(W2))


@pytest.mark.parametrize("hs,lam", [(0, 1.0), (24, 1.0), (24, 0.25)])
def test_dense_masked_formulation(hs, lam):
    """y = sum_e mask_e g_e E_e(x) + lam S(x), with every expert evaluated densely
    (torch einsum), using the oracle's own selection and gates."""
    rng = _rng(21 + hs)
    T, d, E, k, h = 40, 16, 8, 3, 20
    x, Wr, b, W1, W2, Ws1, Ws2 = _layer(rng, T, d, E, k, h, hs)
    y, idx, gate, _ = oracle.forward_tokens(x, Wr, b, W1, W2, k, Ws1, Ws2, lam)
    G = torch.zeros(T, E, dtype=torch.float64)
    G.scatter_(1, torch.from_numpy(idx.astype(np.int64)), torch.from_numpy(gate))
    dense = torch.einsum("te,ted->td", G, _all_experts_t(x, W1, W2))
    if hs:
        dense = dense + lam * (_gelu_t(_t64(x) @ _t64(Ws1)) @ _t64(Ws2))
    np.testing.assert_allclose(y, dense.numpy(), rtol=1e-12, atol=1e-12)


def test_staged_functions_agree_with_whole_layer():
    """permute -> expert_rows -> combine reproduces forward_tokens."""
    rng = _rng(31)
    T, d, E, k, h, hs = 33, 16, 6, 2, 12, 8
    x, Wr, b, W1, W2, Ws1, Ws2 = _layer(rng, T, d, E, k, h, hs)
    y, idx, gate, _, shared = oracle.forward_tokens(x, Wr, b, W1, W2, k, Ws1, Ws2, 0.5, want_shared=True)
    counts, offsets, perm, inv = oracle.permute(idx, E)
    rows = oracle.expert_rows(x, perm, offsets, W1, W2, k, np.arange(T * k, dtype=np.int32))
    y2 = oracle.combine(rows, inv, gate, shared, 0.5)
    np.testing.assert_allclose(y2, y, rtol=1e-13, atol=1e-13)
    hid = oracle.expert_rows(x, perm, offsets, W1, None, k, np.arange(T * k, dtype=np.int32), hidden=True)
    e_of_row = np.repeat(np.arange(E), counts)
    want = _gelu_t(torch.einsum("rd,rdh->rh", _t64(x[perm // k]), _t64(W1[e_of_row])))
    np.testing.assert_allclose(hid, want.numpy(), rtol=1e-12, atol=1e-13)


def test_all_experts_uniform_gates():
    """k = E and W_r = 0: every gate is 1/E and y is the mean of all experts."""
    rng = _rng(41)
    T, d, E, h = 12, 16, 5, 8
    x, _, b, W1, W2, _, _ = _layer(rng, T, d, E, E, h)
    Wr = np.zeros((d, E), np.float32)
    y, idx, gate, margin = oracle.forward_tokens(x, Wr, b, W1, W2, E)
    assert np.all(idx == np.arange(E)) and np.all(gate == 1.0 / E) and np.all(np.isinf(margin))
    want = _all_experts_t(x, W1, W2).mean(1)
    np.testing.assert_allclose(y, want.numpy(), rtol=1e-12, atol=1e-13)


def test_shared_expert_alone():
    """Routed experts all zero: y = lam * GELU(x Ws1) Ws2."""
    rng = _rng(51)
    T, d, E, k, h, hs = 10, 16, 4, 2, 8, 24
    x, Wr, b, W1, W2, Ws1, Ws2 = _layer(rng, T, d, E, k, h, hs)
    W1[:] = 0
    W2[:] = 0
    y, *_ = oracle.forward_tokens(x, Wr, b, W1, W2, k, Ws1, Ws2, 0.75)
    want = 0.75 * (_gelu_t(_t64(x) @ _t64(Ws1)) @ _t64(Ws2))
    np.testing.assert_allclose(y, want.numpy(), rtol=1e-12, atol=1e-13)


def test_token_order_equivariance():
    rng = _rng(61)
    T, d, E, k, h = 30, 16, 8, 2, 12
    x, Wr, b, W1, W2, _, _ = _layer(rng, T, d, E, k, h)
    y, idx, gate, _ = oracle.forward_tokens(x, Wr, b, W1, W2, k)
    p = rng.permutation(T)
    y2, idx2, gate2, _ = oracle.forward_tokens(x[p], Wr, b, W1, W2, k)
    assert np.array_equal(idx2, idx[p])
    np.testing.assert_array_equal(gate2, gate[p])
    np.testing.assert_array_equal(y2, y[p])
    # a token subset gives the same rows
    sub = np.array([3, 0, 29, 7], np.int32)
    y3, idx3, _, _ = oracle.forward_tokens(x, Wr, b, W1, W2, k, tokens=sub)
    np.testing.assert_array_equal(y3, y[sub])


def test_generator_recipe_is_seeded_and_shaped():
    cfg = workloads.small_config(T=16, d=32, E=4, k=2, h=16, h_s=8, seed=3)
    a = workloads.make_layer(cfg)
    b = workloads.make_layer(cfg)
    assert np.array_equal(a.x, b.x) and np.array_equal(a.W1, b.W1) and np.array_equal(a.Ws2, b.Ws2)
    assert a.x.shape == (16, 32) and a.Wr.shape == (32, 4) and a.W1.shape == (4, 32, 16)
    assert a.W2.shape == (4, 16, 32) and a.Ws1.shape == (32, 8) and a.Ws2.shape == (8, 32)
    # bf16 round trip of the generator's rounding
    v = np.array([1.0, -2.5, 3.14159, 1e-3], np.float32)
    back = bf16_bits_to_f32(f32_to_bf16_bits(v))
    assert np.all(np.abs(back - v) <= np.abs(v) * 2.0 ** -8)
    assert np.array_equal(bf16_bits_to_f32(f32_to_bf16_bits(back)), back)


# --------------------------------------------------- loss-free bias update (Eqs. 8-9)

def test_bias_update_zscore_closed_form():
    """Eq. 9 on hand-made loads: counts (2, 4, 6) have mean 4 and population std
    sqrt(8/3), so the z-scores are -sqrt(3/2), 0, +sqrt(3/2) and b moves by -alpha z."""
    alpha = 0.5
    b = np.float32([0.1, -0.2, 0.3])
    out = oracle.update_bias([2, 4, 6], b, alpha)
    z = math.sqrt(1.5)
    want = np.float32([float(b[0]) + alpha * z, float(b[1]), float(b[2]) - alpha * z])
    assert out[1] == b[1]
    np.testing.assert_allclose(out, want, rtol=0, atol=6e-8)   # within one fp32 ulp


def test_bias_update_balanced_loads_leave_b_unchanged():
    """All loads equal: sigma = 0 (z-score, no update) and sign(0) = 0 (sign rule)."""
    b = np.array([0.5, -1.25, 3.0, 0.0], np.float32)
    for rule in ("zscore", "sign"):
        np.testing.assert_array_equal(oracle.update_bias([7, 7, 7, 7], b, 0.01, rule), b)
    np.testing.assert_array_equal(oracle.update_bias([9], [2.5], 0.1), np.float32([2.5]))   # E = 1


def test_bias_update_sign_rule_exact():
    """Eq. 8: each b_e moves by exactly -alpha sign(t_e - mean), mean taken in exact rationals."""
    rng = np.random.default_rng(3)
    counts = rng.integers(0, 400, size=37).astype(np.int32)
    counts[5] = counts[6] = 0
    b = rng.uniform(-0.1, 0.1, size=37).astype(np.float32)
    alpha = 0.001
    out = oracle.update_bias(counts, b, alpha, "sign")
    mean = Fraction(int(counts.sum()), counts.size)
    for e in range(counts.size):
        sgn = (counts[e] > mean) - (counts[e] < mean)
        assert out[e] == np.float32(float(b[e]) - alpha * sgn)


def test_bias_update_zscore_invariants():
    """z-scores of a population sum to 0 and their squares to E; scaling every load by
    the same factor leaves them unchanged."""
    rng = np.random.default_rng(4)
    counts = rng.integers(0, 5000, size=256).astype(np.int32)
    b0 = np.zeros(256, np.float32)
    alpha = 1.0
    z = -oracle.update_bias(counts, b0, alpha).astype(np.float64)
    assert abs(z.sum()) < 1e-4 and abs((z * z).sum() - 256) < 1e-3
    cf = counts.astype(np.float64)
    want = (cf - cf.mean()) / cf.std()                    # numpy population std
    np.testing.assert_allclose(z, want, rtol=0, atol=2e-7)
    z3 = -oracle.update_bias(counts * 3, b0, alpha).astype(np.float64)
    np.testing.assert_allclose(z3, z, rtol=0, atol=2e-7)


# ------------------------------------------------------ SwiGLU experts (App. B)

@pytest.mark.parametrize("h", [40, 13])
def test_single_swiglu_expert_is_dense_swiglu_mlp(h):
    """E = 1, k = 1 with W3: the layer is (SiLU(x W1) * (x W3)) W2, checked against torch
    fp64 (torch.nn.functional.silu); swapping W1 and W3 changes the result."""
    rng = _rng(61)
    T, d = 9, 24
    x = _bf16(rng.standard_normal((T, d)))
    W1 = _bf16(rng.standard_normal((1, d, h)) / np.sqrt(d))
    W3 = _bf16(rng.standard_normal((1, d, h)) / np.sqrt(d))
    W2 = _bf16(rng.standard_normal((1, h, d)) / np.sqrt(h))
    Wr = (rng.standard_normal((d, 1)) * 0.02).astype(np.float32)
    b = np.zeros(1, np.float32)
    y, idx, gate, _ = oracle.forward_tokens(x, Wr, b, W1, W2, 1, W3=W3)
    xt = _t64(x)
    want = (torch.nn.functional.silu(xt @ _t64(W1[0])) * (xt @ _t64(W3[0]))) @ _t64(W2[0])
    assert np.all(idx == 0) and np.all(gate == 1.0)
    np.testing.assert_allclose(y, want.numpy(), rtol=1e-12, atol=1e-12)
    y_sw, *_ = oracle.forward_tokens(x, Wr, b, W3, W2, 1, W3=W1)
    assert np.abs(y_sw - y).max() > 1e-3


def test_swiglu_all_experts_uniform_gates():
    """k = E and W_r = 0 with SwiGLU experts: y is the mean of all E SwiGLU experts
    (a dense einsum over experts in torch fp64)."""
    rng = _rng(62)
    T, d, E, h = 12, 16, 5, 8
    x, _, b, W1, W2, _, _ = _layer(rng, T, d, E, E, h)
    W3 = _bf16(rng.standard_normal((E, d, h)) / np.sqrt(d))
    Wr = np.zeros((d, E), np.float32)
    y, idx, gate, _ = oracle.forward_tokens(x, Wr, b, W1, W2, E, W3=W3)
    xt = _t64(x)
    g = torch.einsum("td,edh->teh", xt, _t64(W1))
    u = torch.einsum("td,edh->teh", xt, _t64(W3))
    want = torch.einsum("teh,ehd->ted", torch.nn.functional.silu(g) * u, _t64(W2)).mean(1)
    np.testing.assert_allclose(y, want.numpy(), rtol=1e-12, atol=1e-13)


def test_swiglu_shared_expert_alone():
    """Routed experts all zero, SwiGLU shared expert: y = lam (SiLU(x Ws1) * (x Ws3)) Ws2."""
    rng = _rng(63)
    T, d, E, k, h, hs = 10, 16, 4, 2, 8, 24
    x, Wr, b, W1, W2, Ws1, Ws2 = _layer(rng, T, d, E, k, h, hs)
    W3 = _bf16(rng.standard_normal((E, d, h)) / np.sqrt(d))
    Ws3 = _bf16(rng.standard_normal((d, hs)) / np.sqrt(d))
    W1[:] = 0
    W2[:] = 0
    y, *_ = oracle.forward_tokens(x, Wr, b, W1, W2, k, Ws1, Ws2, 0.75, W3=W3, Ws3=Ws3)
    xt = _t64(x)
    want = 0.75 * ((torch.nn.functional.silu(xt @ _t64(Ws1)) * (xt @ _t64(Ws3))) @ _t64(Ws2))
    np.testing.assert_allclose(y, want.numpy(), rtol=1e-12, atol=1e-13)


@pytest.mark.parametrize("act", ["gelu", "swiglu"])
def test_shared_expert_splits_into_chunks(act):
    """The activation acts on each hidden unit separately, so a shared expert of width
    2h equals the sum of two shared experts of width h holding its first and second h
    hidden units (columns of Ws1 and Ws3, rows of Ws2): Eq. 6 with m = 2 shared experts
    at the routed width, the form in which the kernels run it.  Checked on the oracle
    with the routed experts zeroed."""
    rng = _rng(71)
    T, d, E, k, h = 11, 16, 4, 2, 12
    x, Wr, b, W1, W2, Ws1, Ws2 = _layer(rng, T, d, E, k, h, 2 * h)
    W1[:] = 0
    W2[:] = 0
    W3 = Ws3 = None
    if act == "swiglu":
        W3 = _bf16(rng.standard_normal((E, d, h)) / np.sqrt(d))
        Ws3 = _bf16(rng.standard_normal((d, 2 * h)) / np.sqrt(d))
    y, *_ = oracle.forward_tokens(x, Wr, b, W1, W2, k, Ws1, Ws2, 0.5, W3=W3, Ws3=Ws3)
    parts = []
    for c in range(2):
        cols = slice(c * h, (c + 1) * h)
        yc, *_ = oracle.forward_tokens(x, Wr, b, W1, W2, k, np.ascontiguousarray(Ws1[:, cols]),
                                       np.ascontiguousarray(Ws2[cols]), 0.5, W3=W3,
                                       Ws3=None if Ws3 is None else np.ascontiguousarray(Ws3[:, cols]))
        parts.append(yc)
    np.testing.assert_allclose(y, parts[0] + parts[1], rtol=1e-12, atol=1e-13)
    assert np.abs(parts[0]).max() > 1e-3 and np.abs(parts[1]).max() > 1e-3


# ------------------------------------------ backward (training path, App. B)

def _torch_layer_from_oracle_routing(x, Wr, W1, W2, idx, lam, Ws1=None, Ws2=None, W3=None, Ws3=None):
    """The layer in torch fp64 autograd with the selection idx held fixed: gates are
    sigmoid(s) renormalised over the selected experts (Eqs. 4-5), experts GELU or
    SwiGLU, plus lam times the shared expert (Eq. 6).  Inputs are torch leaves."""
    s = x @ Wr
    it = torch.from_numpy(idx.astype(np.int64))
    sg = torch.sigmoid(torch.gather(s, 1, it))
    g = sg / sg.sum(1, keepdim=True)

    def ffn(xx, A, B, C):   # A, B: [T, d, h] per token (or [d, h]); C: [T, h, d] (or [h, d])
        if A.dim() == 2:
            u = xx @ A
            a = torch.nn.functional.silu(u) * (xx @ B) if B is not None else _gelu_t(u)
            return a @ C
        u = torch.einsum("td,tdh->th", xx, A)
        a = (torch.nn.functional.silu(u) * torch.einsum("td,tdh->th", xx, B) if B is not None
             else _gelu_t(u))
        return torch.einsum("th,thd->td", a, C)

    y = 0.0
    for j in range(idx.shape[1]):
        e = it[:, j]
        y = y + g[:, j:j + 1] * ffn(x, W1[e], None if W3 is None else W3[e], W2[e])
    if Ws1 is not None:
        y = y + lam * ffn(x, Ws1, Ws3, Ws2)
    return y


def _backward_case(seed, T, d, E, k, h, hs=0, swiglu=False, lam=0.5):
    rng = _rng(seed)
    x, Wr, b, W1, W2, Ws1, Ws2 = _layer(rng, T, d, E, k, h, hs)
    W3 = _bf16(rng.standard_normal((E, d, h)) / np.sqrt(d)) if swiglu else None
    Ws3 = _bf16(rng.standard_normal((d, hs)) / np.sqrt(d)) if (swiglu and hs) else None
    dy = rng.standard_normal((T, d))
    return x, Wr, b, W1, W2, W3, Ws1, Ws2, Ws3, dy, lam


@pytest.mark.parametrize("T,d,E,k,h,hs,swiglu", [
    (7, 16, 1, 1, 12, 0, False), (9, 24, 6, 2, 13, 0, False), (8, 16, 5, 3, 8, 20, False),
    (9, 24, 6, 2, 13, 0, True), (8, 16, 5, 3, 8, 20, True), (6, 8, 4, 4, 6, 6, True),
])
def test_backward_matches_autograd(T, d, E, k, h, hs, swiglu):
    """Every gradient of the oracle's backward against torch fp64 autograd of the layer
    written with torch primitives, the selection held at the oracle's."""
    x, Wr, b, W1, W2, W3, Ws1, Ws2, Ws3, dy, lam = _backward_case(T + E + h, T, d, E, k, h, hs, swiglu)
    got = oracle.backward(x, Wr, b, W1, W2, k, dy, Ws1 if hs else None, Ws2 if hs else None, lam,
                          W3=W3, Ws3=Ws3)
    idx, _, _ = oracle.route(x, Wr, b, k)
    leaves = {"dx": _t64(x), "dWr": torch.from_numpy(Wr.astype(np.float64)), "dW1": _t64(W1),
              "dW2": _t64(W2)}
    if swiglu:
        leaves["dW3"] = _t64(W3)
    if hs:
        leaves["dWs1"], leaves["dWs2"] = _t64(Ws1), _t64(Ws2)
        if swiglu:
            leaves["dWs3"] = _t64(Ws3)
    for v in leaves.values():
        v.requires_grad_(True)
    y = _torch_layer_from_oracle_routing(leaves["dx"], leaves["dWr"], leaves["dW1"], leaves["dW2"], idx,
                                         lam, leaves.get("dWs1"), leaves.get("dWs2"), leaves.get("dW3"),
                                         leaves.get("dWs3"))
    (torch.from_numpy(dy) * y).sum().backward()
    assert set(got) == set(leaves)
    for name, leaf in leaves.items():
        want = leaf.grad.numpy()
        scale = max(np.abs(want).max(), 1e-300)
        np.testing.assert_allclose(got[name], want, rtol=0, atol=1e-12 * scale, err_msg=name)
        if not (name == "dWr" and E == 1):
            assert np.abs(want).max() > 1e-6, name


@pytest.mark.parametrize("swiglu", [False, True])
def test_backward_linear_weight_identities(swiglu):
    """y is linear in W2 (and, with SwiGLU, in W3) and the shared term in Ws2 (Ws3), so
    <dW2, W2> = <dy, y_routed> and <dWs2, Ws2> = lam <dy, S(x)> (the same for W3, Ws3):
    Euler's identity, checked against the pinned forward oracle."""
    T, d, E, k, h, hs = 10, 16, 6, 2, 12, 24
    x, Wr, b, W1, W2, W3, Ws1, Ws2, Ws3, dy, lam = _backward_case(81, T, d, E, k, h, hs, swiglu, 0.75)
    y, _, _, _, S = oracle.forward_tokens(x, Wr, b, W1, W2, k, Ws1, Ws2, lam, want_shared=True,
                                          W3=W3, Ws3=Ws3)
    gr = oracle.backward(x, Wr, b, W1, W2, k, dy, Ws1, Ws2, lam, W3=W3, Ws3=Ws3)
    routed = float(np.sum(dy * (y - lam * S)))
    shared = float(lam * np.sum(dy * S))
    f = lambda a: a.astype(np.float64)  # noqa: E731
    w2 = lambda a: workloads.bf16_bits_to_f32(a).astype(np.float64)  # noqa: E731
    assert abs(np.sum(gr["dW2"] * w2(W2)) - routed) <= 1e-11 * abs(routed) + 1e-12
    assert abs(np.sum(gr["dWs2"] * w2(Ws2)) - shared) <= 1e-11 * abs(shared) + 1e-12
    if swiglu:
        assert abs(np.sum(gr["dW3"] * w2(W3)) - routed) <= 1e-11 * abs(routed) + 1e-12
        assert abs(np.sum(gr["dWs3"] * w2(Ws3)) - shared) <= 1e-11 * abs(shared) + 1e-12
    assert abs(routed) > 1e-3 and abs(shared) > 1e-3 and f(dy).std() > 0


def test_backward_router_gets_no_gradient_when_gates_cannot_matter():
    """Identical experts (every expert output equal) make sum_j g_j o = o whatever the
    gates, so W_r gets no gradient; with one expert (E = k = 1) the gate is always 1."""
    T, d, E, k, h = 8, 16, 5, 3, 8
    x, Wr, b, W1, W2, W3, Ws1, Ws2, Ws3, dy, lam = _backward_case(82, T, d, E, k, h)
    W1[:] = W1[0]
    W2[:] = W2[0]
    gr = oracle.backward(x, Wr, b, W1, W2, k, dy)
    assert np.abs(gr["dWr"]).max() <= 1e-13 * np.abs(gr["dW1"]).max()
    x1, Wr1, b1, W11, W21, *_ , dy1, _ = _backward_case(83, T, d, 1, 1, h)
    gr1 = oracle.backward(x1, Wr1, b1, W11, W21, 1, dy1)
    assert np.all(gr1["dWr"] == 0.0)


@pytest.mark.parametrize("swiglu", [False, True])
def test_backward_router_finite_differences(swiglu):
    """Central differences of the pinned forward oracle along a direction V of W_r,
    against <dWr, V>.  W_r and V are dyadic, so W_r +- V are exact fp32 inputs; only
    tokens whose selection margin is far above the key change carry dy, so no
    selection changes between the two evaluations."""
    rng = _rng(84)
    T, d, E, k, h = 24, 32, 8, 3, 12
    x, _, b, W1, W2, _, _ = _layer(rng, T, d, E, k, h)
    W3 = _bf16(rng.standard_normal((E, d, h)) / np.sqrt(d)) if swiglu else None
    Wr = (np.round(rng.standard_normal((d, E)) * 0.3 * 2 ** 12) / 2 ** 12).astype(np.float32)
    V = (rng.integers(-8, 9, (d, E)) * 2.0 ** -20).astype(np.float32)
    assert np.array_equal((Wr + V) - V, Wr) and np.array_equal((Wr - V) + V, Wr)
    _, _, margin = oracle.route(x, Wr, b, k)
    dy = rng.standard_normal((T, d))
    dy[margin < 1e-2] = 0.0
    assert (margin >= 1e-2).sum() >= T // 2
    L = lambda W: float(np.sum(dy * oracle.forward_tokens(x, W, b, W1, W2, k, W3=W3)[0]))  # noqa: E731
    fd = (L(Wr + V) - L(Wr - V)) / 2.0
    gr = oracle.backward(x, Wr, b, W1, W2, k, dy, W3=W3)
    an = float(np.sum(gr["dWr"] * V.astype(np.float64)))
    assert abs(an) > 1e-9
    assert abs(fd - an) <= 1e-7 * abs(an), (fd, an)


@pytest.mark.parametrize("swiglu", [False, True])
def test_backward_rows_reassemble_the_layer_gradients(swiglu):
    """The staged per-row gradients put back together: sum over the rows of expert e of
    x_t^T du_r is the whole backward's dW1[e] (dW3[e] from dv), and
    sum_r g_r dg_r + lam sum_t dy_t . S(x_t) is sum_t dy_t . y_t of the forward oracle."""
    T, d, E, k, h, hs = 12, 16, 6, 2, 10, 20
    x, Wr, b, W1, W2, W3, Ws1, Ws2, Ws3, dy, lam = _backward_case(91, T, d, E, k, h, hs, swiglu, 0.5)
    idx, gate, _ = oracle.route(x, Wr, b, k)
    counts, offsets, perm, inv = oracle.permute(idx, E)
    gate_rows = gate.reshape(-1)[perm]
    st = oracle.backward_rows(x, perm, offsets, gate_rows, W1, W2, k, dy,
                              np.arange(T * k, dtype=np.int32), W3=W3)
    whole = oracle.backward(x, Wr, b, W1, W2, k, dy, Ws1, Ws2, lam, W3=W3, Ws3=Ws3)
    xf = workloads.bf16_bits_to_f32(x).astype(np.float64)
    tok = perm // k
    for name, g in (("dW1", st["du"]),) + ((("dW3", st.get("dv")),) if swiglu else ()):
        got = np.zeros((E, d, h))
        for e in range(E):
            r = slice(offsets[e], offsets[e + 1])
            got[e] = xf[tok[r]].T @ g[r]
        np.testing.assert_allclose(got, whole[name], rtol=0, atol=1e-12 * np.abs(whole[name]).max(),
                                   err_msg=name)
    y, _, _, _, S = oracle.forward_tokens(x, Wr, b, W1, W2, k, Ws1, Ws2, lam, want_shared=True,
                                          W3=W3, Ws3=Ws3)
    lhs = float(np.sum(gate_rows * st["dg"]) + lam * np.sum(dy * S))
    rhs = float(np.sum(dy * y))
    assert abs(lhs - rhs) <= 1e-12 * max(abs(rhs), 1.0)


def test_backward_skips_tokens_without_dy_exactly():
    """A token whose dy row is zero contributes nothing: with dy on 3 of 8192 tokens the
    backward equals, bit for bit, the backward of the 3-token layer holding those tokens
    (same weights), and dx is zero elsewhere."""
    lay = workloads.make_layer(workloads.small_config(8192, 128, 16, 4, 64, h_s=64, lam=0.5, seed=3))
    c = lay.cfg
    toks = np.array([5, 4000, 8191])
    rng = _rng(92)
    dy = np.zeros((c.T, c.d))
    dy[toks] = rng.standard_normal((toks.size, c.d))
    full = oracle.backward(lay.x, lay.Wr, lay.b, lay.W1, lay.W2, c.k, dy, lay.Ws1, lay.Ws2, c.lam)
    part = oracle.backward(lay.x[toks], lay.Wr, lay.b, lay.W1, lay.W2, c.k, dy[toks], lay.Ws1, lay.Ws2,
                           c.lam)
    for name in part:
        if name == "dx":
            assert np.array_equal(full["dx"][toks], part["dx"])
            assert not np.any(np.delete(full["dx"], toks, axis=0))
        else:
            assert np.array_equal(full[name], part[name]), name


def test_backward_zero_dy_token_with_nonfinite_weight_is_not_skipped():
    """A token with dy_t = 0 adds exact zeros only when the factors its terms multiply
    are finite.  With an infinite entry in W2 of an expert the token uses, the
    gradient through that expert is 0 * inf = NaN, as in torch autograd of the layer;
    the skip of zero-cotangent tokens must not hide it."""
    x, Wr, b, W1, W2, W3, Ws1, Ws2, Ws3, dy, lam = _backward_case(5, 4, 8, 4, 2, 6)
    idx, _, _ = oracle.route(x, Wr, b, 2)
    dy[0] = 0.0
    W2 = W2.copy()
    W2[idx[0, 0], 0, 0] = 0x7F80   # bf16 +inf
    got = oracle.backward(x, Wr, b, W1, W2, 2, dy)
    xt, Wt = _t64(x), _t64(W2)
    xt.requires_grad_(True)
    y = _torch_layer_from_oracle_routing(xt, torch.from_numpy(Wr.astype(np.float64)), _t64(W1), Wt,
                                         idx, lam)
    (torch.from_numpy(dy) * y).sum().backward()
    want = xt.grad.numpy()
    assert np.isnan(want[0]).any()
    assert np.array_equal(np.isnan(got["dx"][0]), np.isnan(want[0]))
