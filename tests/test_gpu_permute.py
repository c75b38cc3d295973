"""Expert-major order parity (App. B, Algorithm 1, phase 1): counts, offsets, perm
and inv from the GPU are bit-exact against the oracle's stable counting sort."""
import numpy as np
import pytest

import oracle
from paper_2608_17402_gb300 import moevie
from tests._gpu import check_status, dev

pytestmark = pytest.mark.gpu


def _routing(rng, T, E, k, empty=(), hot=None):
    allowed = np.array([e for e in range(E) if e not in set(empty)])
    rows = []
    for _ in range(T):
        if hot is not None:
            rest = rng.choice(allowed[allowed != hot], size=k - 1, replace=False)
            rows.append(np.sort(np.concatenate([[hot], rest])))
        else:
            rows.append(np.sort(rng.choice(allowed, size=k, replace=False)))
    return np.stack(rows).astype(np.int32) if T else np.zeros((0, k), np.int32)


@pytest.mark.parametrize("T,E,k,empty,hot", [
    (1, 1, 1, (), None), (3, 4, 2, (0,), None), (127, 16, 2, (3, 7), None),
    (128, 16, 4, (), None), (129, 64, 8, (0, 63), None), (1000, 256, 8, (5,), 17),
    (4097, 128, 1, (), None), (3000, 1024, 8, (), None), (2048, 8, 8, (), None),
])
def test_permute_matches_oracle(T, E, k, empty, hot):
    rng = np.random.default_rng(T + 31 * E + k)
    idx = _routing(rng, T, E, k, empty, hot)
    ws = moevie.Workspace(max(T, 1), 8, E, k, 16)
    counts, offsets, perm, inv = moevie.moevie_permute(dev(idx), E, ws)
    check_status(ws)
    oc, oo, op, oi = oracle.permute(idx, E)
    assert np.array_equal(counts.cpu().numpy(), oc)
    assert np.array_equal(offsets.cpu().numpy(), oo)
    assert np.array_equal(perm.cpu().numpy(), op)
    assert np.array_equal(inv.cpu().numpy(), oi)


@pytest.mark.parametrize("sizes", [[0, 1, 127, 128, 129, 255], [0, 1, 255, 256, 257, 511, 512, 513]])
def test_permute_segment_length_edges(sizes):
    """Segments around the 128-row CTA half and the 256-row m-tile of the GEMMs."""
    E, k = len(sizes), 1
    ids = np.concatenate([np.full(n, e, np.int32) for e, n in enumerate(sizes)])
    rng = np.random.default_rng(3)
    rng.shuffle(ids)
    idx = ids.reshape(-1, 1)
    ws = moevie.Workspace(idx.shape[0], 8, E, k, 16)
    counts, offsets, perm, inv = moevie.moevie_permute(dev(idx), E, ws)
    check_status(ws)
    assert counts.cpu().numpy().tolist() == sizes
    oc, oo, op, oi = oracle.permute(idx, E)
    assert np.array_equal(perm.cpu().numpy(), op) and np.array_equal(inv.cpu().numpy(), oi)


def test_permute_reports_bad_ids():
    """An id outside [0, E) is a device error in the status block, not a fault."""
    E, k = 8, 2
    idx = np.array([[0, 3], [1, 9], [2, 5]], np.int32)
    ws = moevie.Workspace(3, 8, E, k, 16)
    moevie.moevie_permute(dev(idx), E, ws)
    code, detail = moevie.moevie_get_device_status(ws)
    assert code == 6 and detail[2] == 3 and detail[3] == 9
