"""Loss-free balancing bias update (Sec. 2.2.2, Eqs. 8-9) through moevie_update_bias
against the oracle: the sign rule bit for bit; the z-score rule within one fp32 ulp
(both sides compute in fp64 and round the new b_e to fp32, but the standard
deviation's sum of squares runs in a different order)."""
import numpy as np
import pytest
import torch

import oracle
import workloads
from paper_2608_17402_gb300 import moevie
from tests._gpu import check_status, dev, layer_to_device, workspace_for

pytestmark = pytest.mark.gpu


def _gpu_update(counts, b, alpha, rule):
    ws = moevie.Workspace(16, 16, 4, 2, 16)
    bt = dev(np.asarray(b, np.float32)).clone()
    moevie.moevie_update_bias(dev(np.asarray(counts, np.int32)), bt, alpha, ws, rule)
    check_status(ws)
    return bt.cpu().numpy()


@pytest.mark.parametrize("E", [1, 16, 64, 255, 256, 1024])
@pytest.mark.parametrize("rule", ["zscore", "sign"])
def test_bias_update_matches_oracle(E, rule):
    rng = np.random.default_rng(E)
    counts = rng.integers(0, 3000, size=E).astype(np.int32)
    if E > 4:
        counts[:3] = 0                                  # empty experts
        counts[3] = int(counts.mean())                  # a load near the mean
    b = rng.uniform(-0.1, 0.1, size=E).astype(np.float32)
    alpha = 1e-3
    got = _gpu_update(counts, b, alpha, rule)
    want = oracle.update_bias(counts, b, alpha, rule)
    if rule == "sign":
        np.testing.assert_array_equal(got, want)
    else:
        np.testing.assert_allclose(got, want, rtol=0, atol=np.spacing(np.abs(want)).max())


def test_bias_update_balanced_and_exact_mean():
    """Equal loads: nothing moves.  Loads symmetric about an integer mean: the expert at
    the mean keeps its bias under both rules."""
    b = np.linspace(-0.05, 0.05, 64).astype(np.float32)
    for rule in ("zscore", "sign"):
        np.testing.assert_array_equal(_gpu_update(np.full(64, 128, np.int32), b, 0.01, rule), b)
    counts = np.array([10, 20, 30], np.int32)
    for rule in ("zscore", "sign"):
        got = _gpu_update(counts, [0.5, 0.25, -0.5], 0.1, rule)
        assert got[1] == np.float32(0.25)
        np.testing.assert_allclose(got, oracle.update_bias(counts, [0.5, 0.25, -0.5], 0.1, rule),
                                   rtol=0, atol=6e-8)


def test_bias_update_from_forward_counts():
    """One balancing step driven by the counts a forward returns (c0 layer)."""
    lay = workloads.make_layer(workloads.CONFIGS["c0"])
    x, W = layer_to_device(lay)
    ws = workspace_for(lay)
    _, rt = moevie.moevie_moe_forward(W, x, ws, routing=True)
    counts = rt["counts"]
    b = W.b.clone()
    moevie.moevie_update_bias(counts, b, 1e-3, ws, "zscore")
    check_status(ws)
    want = oracle.update_bias(counts.cpu().numpy(), lay.b, 1e-3, "zscore")
    np.testing.assert_allclose(b.cpu().numpy(), want, rtol=0, atol=np.spacing(np.abs(want)).max())


def test_bias_update_negative_load_is_a_device_error():
    ws = moevie.Workspace(16, 16, 4, 2, 16)
    b = torch.zeros(8, dtype=torch.float32, device="cuda")
    counts = torch.tensor([1, 2, -3, 4, 5, 6, 7, 8], dtype=torch.int32, device="cuda")
    moevie.moevie_update_bias(counts, b, 0.1, ws)
    code, detail = moevie.moevie_get_device_status(ws)
    assert code == 6 and detail[1] == 21
    assert float(b.abs().sum()) == 0.0
