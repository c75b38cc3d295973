"""Grouped GEMM parity (App. B, Algorithm 1, Kernels 1-2): the tcgen05 up-projection
with GELU, the expert FFN rows, the shared expert and the stand-alone combine,
each against the oracle on the same seeded inputs."""
import numpy as np
import pytest
import torch

import oracle
import workloads
from paper_2608_17402_gb300 import moevie
from tests._gpu import assert_close, check_status, dev, dev_bf16, dev_rows, to_np_f64

pytestmark = pytest.mark.gpu


def _bf(rng, shape, std=1.0):
    return workloads.f32_to_bf16_bits((rng.standard_normal(shape) * std).astype(np.float32))


def _case(seed, T, d, E, k, h, sizes=None):
    rng = np.random.default_rng(seed)
    x = _bf(rng, (T, d))
    W1 = _bf(rng, (E, d, h), 1 / np.sqrt(d))
    W2 = _bf(rng, (E, h, d), 1 / np.sqrt(h))
    if sizes is not None:   # an explicit expert load (k == 1)
        ids = np.concatenate([np.full(n, e, np.int32) for e, n in enumerate(sizes)])
        rng.shuffle(ids)
        idx = ids.reshape(T, 1)
    else:
        idx = np.stack([np.sort(rng.choice(E, size=k, replace=False)) for _ in range(T)]).astype(np.int32)
    counts, offsets, perm, inv = oracle.permute(idx, E)
    return x, W1, W2, idx, counts, offsets, perm, inv


SHAPES = [
    # seed, T, d, E, k, h, sizes
    (1, 64, 64, 4, 2, 64, None),          # one k-block, tiny N
    (2, 300, 128, 8, 2, 416, None),       # N tail of the up GEMM (416 = 2 x 208), K tail of the down GEMM
    (3, 515, 256, 6, 1, 96, [0, 1, 127, 128, 129, 130]),   # segment-length edges incl. an empty expert
    (4, 257, 1024, 3, 3, 512, None),      # k = E, long K loop
    (5, 40, 776, 2, 1, 48, None),         # d % 16 != 0 (8-column output tail), K tail in the up GEMM
    (6, 899, 192, 6, 1, 64, [0, 1, 255, 256, 257, 130]),   # segments around the 256-row m-tile
    # hidden widths that are not multiples of 8 or 16 (rows of W1 and H padded to 8)
    (7, 333, 256, 5, 2, 684, None),       # the paper's L width: N and K tails of 44
    (8, 200, 128, 4, 2, 854, None),       # the paper's H width: 6 columns past a multiple of 8
    (9, 150, 64, 3, 1, 13, [50, 0, 100]), # odd h below one output group
    (10, 90, 96, 2, 2, 1, None),          # h = 1
]


@pytest.mark.parametrize("seed,T,d,E,k,h,sizes", SHAPES)
def test_expert_hidden_matches_oracle(seed, T, d, E, k, h, sizes):
    x, W1, W2, idx, counts, offsets, perm, inv = _case(seed, T, d, E, k, h, sizes)
    ws = moevie.Workspace(T, d, E, k, h)
    hid = moevie.moevie_test_expert_hidden(dev_bf16(x), dev(perm), dev(offsets), dev_rows(W1), k, ws)
    check_status(ws)
    want = oracle.expert_rows(x, perm, offsets, W1, None, k, np.arange(T * k, dtype=np.int32), hidden=True)
    assert_close(to_np_f64(hid), want, "hidden")


@pytest.mark.parametrize("seed,T,d,E,k,h,sizes", SHAPES)
def test_expert_ffn_matches_oracle(seed, T, d, E, k, h, sizes):
    x, W1, W2, idx, counts, offsets, perm, inv = _case(seed, T, d, E, k, h, sizes)
    ws = moevie.Workspace(T, d, E, k, h)
    rows = moevie.moevie_expert_ffn(dev_bf16(x), dev(perm), dev(offsets), dev_rows(W1), dev_bf16(W2), k, ws)
    check_status(ws)
    want = oracle.expert_rows(x, perm, offsets, W1, W2, k, np.arange(T * k, dtype=np.int32))
    assert_close(to_np_f64(rows), want, "out_rows")


@pytest.mark.parametrize("hs", [1024, 684])
def test_shared_expert_matches_oracle(hs):
    rng = np.random.default_rng(9)
    T, d = 300, 256
    x = _bf(rng, (T, d))
    Ws1 = _bf(rng, (d, hs), 1 / np.sqrt(d))
    Ws2 = _bf(rng, (hs, d), 1 / np.sqrt(hs))
    ws = moevie.Workspace(T, d, 1, 1, 16, hs)
    out = moevie.moevie_shared_expert(dev_bf16(x), dev_rows(Ws1), dev_bf16(Ws2), ws)
    check_status(ws)
    # the shared expert is the single-expert layer E = 1, k = 1
    want, *_ = oracle.forward_tokens(x, np.zeros((d, 1), np.float32), np.zeros(1, np.float32),
                                     Ws1[None], Ws2[None], 1)
    assert_close(to_np_f64(out), want, "shared")


@pytest.mark.parametrize("with_shared", [False, True])
def test_combine_matches_oracle(with_shared):
    rng = np.random.default_rng(11)
    T, d, E, k = 333, 136, 8, 3
    idx = np.stack([np.sort(rng.choice(E, size=k, replace=False)) for _ in range(T)]).astype(np.int32)
    _, _, perm, inv = oracle.permute(idx, E)
    rows = _bf(rng, (T * k, d))
    gate = rng.dirichlet(np.ones(k), size=T).astype(np.float32)
    shared = _bf(rng, (T, d)) if with_shared else None
    y = moevie.moevie_combine(dev_bf16(rows), dev(inv), dev(gate), k,
                              dev_bf16(shared) if with_shared else None, 0.5)
    want = oracle.combine(workloads.bf16_bits_to_f32(rows).astype(np.float64), inv,
                          gate.astype(np.float64),
                          workloads.bf16_bits_to_f32(shared).astype(np.float64) if with_shared else None,
                          0.5)
    assert_close(to_np_f64(y), want, "combine")
