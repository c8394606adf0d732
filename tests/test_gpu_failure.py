"""Failure detection on the GPU without a fault: a bounded device wait that
runs out (an mbarrier nothing arrives on, through the kernels' own wait
routine with a short budget) must come back as ACID_ERR_TIMEOUT through
acid_check_device_error, clear itself, and leave the context usable."""

import numpy as np
import pytest

import acid_synth as S
import oracle as O

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def acid():
    import __graft_entry__ as g

    g.build()
    from paper_2607_12358_gb300 import acid as a

    return a


def test_bounded_wait_reports_timeout_and_context_survives(acid):
    from paper_2607_12358_gb300 import _capi as A

    acid.check_device_error()  # nothing pending
    acid.selftest_wait_timeout(2_000_000)  # about a millisecond of SM clocks
    with pytest.raises(A.AcidError) as e:
        acid.check_device_error()
    assert e.value.status == A.ACID_ERR_TIMEOUT
    acid.check_device_error()  # the flag was cleared by the read
    # the context still computes correctly afterwards
    prev, cur = S.micro_pair(4096, 0.01, seed=3, d=256)
    p = torch.from_numpy(prev).cuda().to(torch.bfloat16)
    c = torch.from_numpy(cur).cuda().to(torch.bfloat16)
    rel = torch.empty(1, dtype=torch.float64, device="cuda")
    acid.acid_drift_signal(p, c, out_rel=rel)
    ref = O.rel_l1(S.round_to_bf16(prev).astype(np.float64), S.round_to_bf16(cur).astype(np.float64))
    assert abs(rel.item() - ref) <= 1e-3 * ref
    acid.check_device_error()
