"""Device error path: a bounded wait that nobody satisfies gives up, records
MOEVIE_ERR_TIMEOUT in the workspace status block, and the context stays usable.
Nothing here faults, traps or hangs the GPU."""
import pytest
import torch

from paper_2608_17402_gb300 import moevie

pytestmark = pytest.mark.gpu


def test_bounded_wait_reports_timeout_and_context_survives():
    ws = moevie.Workspace(16, 16, 4, 2, 16)
    code, _ = moevie.moevie_get_device_status(ws)
    assert code == 0
    moevie.moevie_test_wait_timeout(ws, 1_000_000)     # 1 ms
    code, detail = moevie.moevie_get_device_status(ws)
    assert code == 5 and detail[1] == 30
    # the status is sticky until the workspace is set up again
    moevie.moevie_workspace_init(ws)
    assert moevie.moevie_get_device_status(ws)[0] == 0
    # the CUDA context still works
    a = torch.arange(1024, device="cuda", dtype=torch.float32)
    assert float(a.sum()) == 1023 * 1024 / 2
