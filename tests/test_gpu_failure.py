"""Failure detection on the GPU without a fault: the bounded wait every
kernel uses runs out on a barrier that nothing signals, reports
PF_DEVERR_TIMEOUT through the error word, and leaves the context usable
(a verify step afterwards still matches the oracle)."""
import time

import pytest
import torch

from paper_2609_32166_gb300 import binding as pb
from paper_2609_32166_gb300 import inputs as I
from tests.parity import Case

pytestmark = pytest.mark.gpu


def _run(limit_ns, signal):
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    ok = torch.full((1,), -1, dtype=torch.int32, device="cuda")
    t0 = time.perf_counter()
    pb.pf_selftest_wait(err.data_ptr(), limit_ns, signal, ok.data_ptr(),
                        torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    return int(err.item()), int(ok.item()), time.perf_counter() - t0


def test_unsignalled_wait_times_out_and_reports():
    err, ok, dt = _run(2_000_000, signal=False)     # 2 ms limit
    assert err & pb.PF_DEVERR_TIMEOUT
    assert ok == 0
    assert dt < 5.0


def test_signalled_wait_completes():
    err, ok, _ = _run(2_000_000, signal=True)
    assert err == 0 and ok == 1


def test_context_usable_after_a_timeout():
    _run(1_000_000, signal=False)
    c = Case(I.WORKLOADS["tiny-f32-chain8"], seed=2)
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    c.check_attention(0, 0)
    c.check_lmhead(res)
    c.check_commit(res)


def test_selftest_rejects_bad_limits():
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    with pytest.raises(pb.PfError):
        pb.pf_selftest_wait(err.data_ptr(), 10, False, err.data_ptr())
