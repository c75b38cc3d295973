"""moevie_permute_static (the permute with a fixed device scratch instead of a
caller workspace) against moevie_permute, through the C ABI: identical outputs on
two calls in a row, and oversized inputs rejected before anything is enqueued.
This file is collected last so that it also runs after every other GPU test."""
import gc

import numpy as np
import pytest
import torch

import workloads
from paper_2608_17402_gb300 import moevie
from tests._gpu import check_status

pytestmark = pytest.mark.gpu

MAX_SLOTS = 1 << 20


def _ids(T, E, k, seed):
    """Distinct ascending ids per token, as the router emits them."""
    rng = np.random.default_rng(seed)
    keys = rng.random((T, E))
    return np.sort(np.argsort(-keys, axis=1)[:, :k], axis=1).astype(np.int32)


@pytest.mark.parametrize("T,E,k", [(1, 4, 1), (1000, 64, 8), (4099, 33, 5),
                                   (65536, 256, 8), (MAX_SLOTS // 8, 1024, 8)])
def test_static_permute_matches_workspace_permute(T, E, k):
    idx = torch.from_numpy(_ids(T, E, k, T + E)).cuda()
    ws = moevie.Workspace(T, 8, E, k, 16)
    want = moevie.moevie_permute(idx, E, ws)
    check_status(ws)
    want = [t.cpu() for t in want]
    for _ in range(2):   # a second call must not depend on what the first left behind
        got = moevie.moevie_permute_static(idx, E)
        torch.cuda.synchronize()
        for name, a, b in zip(("counts", "offsets", "perm", "inv"), got, want):
            assert torch.equal(a.cpu(), b), name


def test_static_permute_skewed_and_empty_experts():
    """Most slots on a few experts, many experts empty (the skewed routing case)."""
    cfg = workloads.CONFIGS["c4"]
    rng = np.random.default_rng(11)
    T, E, k = 20000, cfg.E, cfg.k
    p = rng.pareto(1.2, E) + 1e-3
    p[rng.random(E) < 0.3] = 0.0
    ids = np.stack([np.sort(rng.choice(E, k, replace=False, p=p / p.sum())) for _ in range(T)])
    idx = torch.from_numpy(ids.astype(np.int32)).cuda()
    ws = moevie.Workspace(T, 8, E, k, 16)
    want = [t.cpu() for t in moevie.moevie_permute(idx, E, ws)]
    check_status(ws)
    for _ in range(2):
        got = moevie.moevie_permute_static(idx, E)
        for a, b in zip(got, want):
            assert torch.equal(a.cpu(), b)


def test_static_permute_rejects_oversize_and_accepts_empty():
    idx = torch.zeros((MAX_SLOTS // 8 + 1, 8), dtype=torch.int32, device="cuda")
    with pytest.raises(moevie.MoevieError) as e:
        moevie.moevie_permute_static(idx, 16)
    assert e.value.code == 2   # MOEVIE_ERR_UNSUPPORTED
    counts, offsets, _, _ = moevie.moevie_permute_static(
        torch.zeros((0, 4), dtype=torch.int32, device="cuda"), 16)
    assert int(counts.abs().sum()) == 0 and int(offsets.abs().sum()) == 0


def test_static_permute_allocates_nothing():
    """With its outputs preallocated, neither a second nor a third call changes the
    device's free memory (cudaMemGetInfo) or torch's allocated bytes: the scratch is
    the library's fixed device array.  The first call may load the library's device
    code (set-up), so it runs before the measurement."""
    T, E, k = 4096, 64, 8
    idx = torch.from_numpy(_ids(T, E, k, 3)).cuda()
    out = (torch.empty(E, dtype=torch.int32, device="cuda"),
           torch.empty(E + 1, dtype=torch.int32, device="cuda"),
           torch.empty(T * k, dtype=torch.int32, device="cuda"),
           torch.empty(T * k, dtype=torch.int32, device="cuda"))
    moevie.moevie_permute_static(idx, E, out=out)
    torch.cuda.synchronize()
    gc.collect()   # tensors left by earlier tests are freed now, not during the measurement
    gc.disable()
    try:
        for _ in range(2):
            free0, _ = torch.cuda.mem_get_info()
            alloc0 = torch.cuda.memory_allocated()
            moevie.moevie_permute_static(idx, E, out=out)
            torch.cuda.synchronize()
            free1, _ = torch.cuda.mem_get_info()
            assert free1 == free0, (free0, free1)
            assert torch.cuda.memory_allocated() == alloc0
    finally:
        gc.enable()


def test_static_permute_drops_out_of_range_ids():
    """Ids -1 and E are device errors that drop their slot: inv = -1 there, counts and
    offsets leave them out, and every valid slot keeps the stable expert-major row
    that moevie_permute gives it (the workspace entry point, same rule)."""
    T, E, k = 300, 16, 4
    ids = _ids(T, E, k, 21)
    bad = [(3, 0, -1), (77, 2, E), (299, 3, E), (150, 1, -1)]
    for t, j, v in bad:
        ids[t, j] = v
    idx = torch.from_numpy(ids).cuda()
    ws = moevie.Workspace(T, 8, E, k, 16)
    want = [t.cpu() for t in moevie.moevie_permute(idx, E, ws)]
    for _ in range(2):
        counts, offsets, perm, inv = (t.cpu() for t in moevie.moevie_permute_static(idx, E))
        for t, j, _v in bad:
            assert int(inv[t * k + j]) == -1
        valid = (ids >= 0) & (ids < E)
        assert torch.equal(counts, torch.from_numpy(np.bincount(ids[valid], minlength=E).astype(np.int32)))
        assert int(offsets[E]) == int(valid.sum())
        assert torch.equal(counts, want[0]) and torch.equal(offsets, want[1]) and torch.equal(inv, want[3])
        n = int(valid.sum())
        assert torch.equal(perm[:n], want[2][:n])
