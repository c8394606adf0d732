"""acid_drift_signal_noalloc: the drift reduction for callers that cannot
allocate device memory (not even a workspace), checked through the C ABI
against acid_drift_signal, the entry point that takes a caller-provided
workspace, and against the fp64 CPU oracle.  Two calls in a row, so a stale
scratch array would show.

This file is collected last so that a run stopping at the first failure has
already run every other test; it also passes on its own in a fresh process.
"""

import ctypes

import numpy as np
import pytest

import acid_synth as S
import oracle as O

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")
DEV = "cuda"
DRIFT_RTOL = 1e-3  # the drift tolerance used by the other parity tests


@pytest.fixture(scope="module")
def lib():
    import __graft_entry__ as g

    g.build()
    from paper_2607_12358_gb300 import _capi

    return _capi


def _workspace_call(A, tp, tc, dtype):
    from paper_2607_12358_gb300 import acid

    rel, sums = acid.acid_drift_signal(tp, tc)
    return rel.item(), sums.cpu().numpy()


def _noalloc_call(A, tp, tc, dtype, host=False):
    stream = torch.cuda.current_stream().cuda_stream
    if host:
        rel = ctypes.c_double(-1.0)
        sums = (ctypes.c_double * 2)()
        A.check(A.load().acid_drift_signal_noalloc(tp.data_ptr(), tc.data_ptr(), tp.numel(), dtype,
                                                   ctypes.addressof(rel), ctypes.addressof(sums), stream))
        return rel.value, np.array([sums[0], sums[1]])
    rel = torch.full((1,), -1.0, dtype=torch.float64, device=DEV)
    sums = torch.full((2,), -1.0, dtype=torch.float64, device=DEV)
    A.check(A.load().acid_drift_signal_noalloc(tp.data_ptr(), tc.data_ptr(), tp.numel(), dtype, rel.data_ptr(),
                                               sums.data_ptr(), stream))
    torch.cuda.synchronize()
    return rel.item(), sums.cpu().numpy()


def _pair(rows, sigma, seed, bf16=True):
    prev, cur = S.micro_pair(rows, sigma, seed=seed, d=S.MICRO_D, bf16=bf16)
    dt = torch.bfloat16 if bf16 else torch.float32
    return torch.from_numpy(prev).to(DEV, dt), torch.from_numpy(cur).to(DEV, dt)


def test_noalloc_matches_workspace_entry_point_twice(lib):
    A = lib
    # first call: large bf16 pair; second call: a smaller, ragged fp32 pair (fewer
    # thread blocks than the first call, so stale partials would be summed)
    cases = [(_pair(4096, 1e-2, 1), A.ACID_BF16), (_pair(37, 1e-1, 2, bf16=False), A.ACID_FP32)]
    for (tp, tc), dt in cases:
        ref_rel, ref_sums = _workspace_call(A, tp, tc, dt)
        rel, sums = _noalloc_call(A, tp, tc, dt)
        assert abs(rel - ref_rel) <= DRIFT_RTOL * ref_rel
        np.testing.assert_allclose(sums, ref_sums, rtol=DRIFT_RTOL)
        # the same inputs in the fp64 oracle (the device values, upcast)
        p64, c64 = tp.double().cpu().numpy(), tc.double().cpu().numpy()
        orel = O.rel_l1(p64, c64)
        assert abs(rel - orel) <= DRIFT_RTOL * orel, (rel, orel)
        np.testing.assert_allclose(sums, [np.abs(c64 - p64).sum(), np.abs(p64).sum()], rtol=DRIFT_RTOL)
        hrel, hsums = _noalloc_call(A, tp, tc, dt, host=True)
        assert abs(hrel - ref_rel) <= DRIFT_RTOL * ref_rel
        np.testing.assert_allclose(hsums, ref_sums, rtol=DRIFT_RTOL)


def test_noalloc_rejects_sizes_beyond_maximum(lib):
    A = lib
    out = torch.zeros(1, dtype=torch.float64, device=DEV)
    x = torch.zeros(16, dtype=torch.bfloat16, device=DEV)
    st = A.load().acid_drift_signal_noalloc(x.data_ptr(), x.data_ptr(), (1 << 31) + 1, A.ACID_BF16,
                                            out.data_ptr(), None, None)
    assert st == A.ACID_ERR_UNSUPPORTED
    assert b"maximum" in A.load().acid_last_error()
