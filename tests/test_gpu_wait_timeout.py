"""Failure detection without a GPU fault: a device wait that nothing
satisfies gives up after its limit, reports HPD_DEVERR_TIMEOUT through the
error word, and leaves the context usable (the next attention call matches
the oracle)."""
import time

import numpy as np
import pytest

pytestmark = pytest.mark.gpu

HPD_DEVERR_TIMEOUT = 0x40


def test_wait_runs_out_and_context_stays_usable():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2607_18839_gb300 import hpd as H
    from paper_2607_18839_gb300 import workloads as W
    import oracle

    ws = torch.zeros(256, dtype=torch.uint8, device="cuda")
    H.hpd_workspace_init(ws.data_ptr(), 256, None)
    t0 = time.perf_counter()
    H.hpd_wait_selftest(ws.data_ptr(), 2000, None)  # 2 ms per wait
    flags = H.hpd_read_errors(ws.data_ptr(), None)
    el = time.perf_counter() - t0
    assert flags == HPD_DEVERR_TIMEOUT | (HPD_DEVERR_TIMEOUT << 8)
    assert el < 5.0
    with pytest.raises(H.HpdError):
        H.hpd_wait_selftest(ws.data_ptr(), 0, None)
    # the context still works
    inp = W.make_config("c1")
    d = H.DeviceInputs.from_host(inp)
    out, lse = H.branch_attn(d)
    torch.cuda.synchronize()
    ref_out, ref_lse = oracle.branch_attn(inp)
    got = out.float().cpu().numpy().reshape(ref_out.shape)
    assert np.nanmax(np.abs(got - ref_out)) <= 1e-2
    assert np.nanmax(np.abs(lse.cpu().numpy().reshape(ref_lse.shape) - ref_lse)) <= 1e-3
