"""GPU parity of the drift signal and cache apply (through the C ABI) against
the oracle, on the drift micro-benchmark workload ([T, 3072] bf16 pairs,
T in {4096, 32760, 67320, 118800}, sigma in {1e-3, 1e-2, 1e-1}) and edge
cases."""

import math

import numpy as np
import pytest

import acid_synth as S
import oracle as O

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")
DEV = "cuda"

DRIFT_RTOL = 1e-3  # drift values within 1e-3 relative of the oracle


@pytest.fixture(scope="module")
def acid():
    import __graft_entry__ as g

    g.build()
    from paper_2607_12358_gb300 import acid as a

    return a


def _bf(a):
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(DEV, torch.bfloat16)


@pytest.mark.parametrize("T", S.MICRO_T)
def test_microbench_drift_apply_and_decisions(acid, T):
    """Full-size micro-benchmark: each sigma's drift value matches the oracle
    within 1e-3, the fused drift + apply gives the same drift and
    out = cur + residual to one bf16 rounding, and the dual-threshold decisions
    on the resulting signal sequence match the oracle's."""
    r = S.micro_residual(T, seed=5)
    tr = _bf(r)
    gpu_s, ref_s = [], []
    for sigma in S.MICRO_SIGMA:
        prev, cur = S.micro_pair(T, sigma, seed=5)
        tp, tc = _bf(prev), _bf(cur)
        rel, sums = acid.acid_drift_signal(tp, tc)
        ref = O.rel_l1(prev, cur)
        num, den = O.drift_sums(prev, cur)
        assert abs(rel.item() - ref) <= DRIFT_RTOL * ref
        s = sums.cpu().numpy()
        assert abs(s[0] - num) <= 1e-4 * num and abs(s[1] - den) <= 1e-4 * den
        out, rel2, _ = acid.acid_drift_apply(tp, tc, tr)
        assert abs(rel2.item() - ref) <= DRIFT_RTOL * ref
        # one rounding of an exact fp32 sum: at most half a bf16 ulp from the rounded fp64 sum
        ref_out = S.round_to_bf16((cur.astype(np.float64) + r).astype(np.float32))
        got = out.float().cpu().numpy()
        ulp = np.abs(ref_out) * 2.0 ** -7 + 1e-30
        assert np.all(np.abs(got - ref_out) <= ulp)
        assert np.mean(got == ref_out) > 0.999
        gpu_s.append(rel.item())
        ref_s.append(ref)
        del tp, tc, out
    # decisions: sigma sweep as a signal sequence under the workload thresholds
    seq_g = gpu_s * 4
    seq_r = ref_s * 4
    d_g = O.controller_decisions(seq_g, 0, 0.05, 0.2, 0.01)
    d_r = O.controller_decisions(seq_r, 0, 0.05, 0.2, 0.01)
    assert d_g == d_r


def test_drift_identical_is_zero(acid):
    a = _bf(np.random.default_rng(0).normal(size=12345))
    rel, sums = acid.acid_drift_signal(a, a)
    assert rel.item() == 0.0 and sums[0].item() == 0.0


def test_drift_zero_denominator(acid):
    z = torch.zeros(100, device=DEV, dtype=torch.bfloat16)
    rel, _ = acid.acid_drift_signal(z, z)
    assert rel.item() == 0.0
    rel, _ = acid.acid_drift_signal(z, torch.ones_like(z))
    assert math.isinf(rel.item())


@pytest.mark.parametrize("n", [1, 7, 8, 9, 1000, 4097, 3 * 2 ** 20 + 5])
@pytest.mark.parametrize("dtype", ["bf16", "fp32"])
def test_drift_ragged_lengths(acid, n, dtype):
    rng = np.random.default_rng(n)
    prev = rng.normal(size=n).astype(np.float32)
    cur = (prev + 0.05 * rng.normal(size=n)).astype(np.float32)
    if dtype == "bf16":
        prev, cur = S.round_to_bf16(prev), S.round_to_bf16(cur)
        tp, tc = _bf(prev), _bf(cur)
    else:
        tp, tc = torch.from_numpy(prev).to(DEV), torch.from_numpy(cur).to(DEV)
    rel, _ = acid.acid_drift_signal(tp, tc)
    ref = O.rel_l1(prev, cur)
    assert abs(rel.item() - ref) <= DRIFT_RTOL * ref
    out = acid.acid_cache_apply(tp, tc)
    ref_out = (prev.astype(np.float64) + cur).astype(np.float32)
    if dtype == "bf16":
        ref_out = S.round_to_bf16(ref_out)
    np.testing.assert_array_equal(out.float().cpu().numpy(), ref_out)


def test_drift_host_output_pointer(acid):
    """A host output pointer makes the call synchronous and fills host memory."""
    import ctypes
    from paper_2607_12358_gb300 import _capi as A

    prev, cur = S.micro_pair(64, 1e-1, seed=9)
    tp, tc = _bf(prev), _bf(cur)
    out = ctypes.c_double(-1.0)
    sums = (ctypes.c_double * 2)()
    ws = torch.empty(acid.drift_workspace_size(tp.numel()), dtype=torch.uint8, device=DEV)
    A.check(A.load().acid_drift_signal(tp.data_ptr(), tc.data_ptr(), tp.numel(), A.ACID_BF16, ctypes.addressof(out),
                                       ctypes.addressof(sums), ws.data_ptr(), ws.numel(),
                                       torch.cuda.current_stream().cuda_stream))
    ref = O.rel_l1(prev, cur)
    assert abs(out.value - ref) <= DRIFT_RTOL * ref
    assert sums[1] == pytest.approx(O.drift_sums(prev, cur)[1], rel=1e-5)


def test_drift_empty_input(acid):
    e = torch.empty(0, device=DEV, dtype=torch.bfloat16)
    rel, sums = acid.acid_drift_signal(e, e)
    assert rel.item() == 0.0


def test_drift_rejects_small_workspace(acid):
    from paper_2607_12358_gb300._capi import AcidError
    a = torch.zeros(64, device=DEV, dtype=torch.bfloat16)
    with pytest.raises(AcidError):
        acid.acid_drift_signal(a, a, workspace=torch.empty(16, dtype=torch.uint8, device=DEV))


def test_drift_and_apply_past_32_bit_offsets(acid):
    """2^31 + 13 bf16 elements (4.3 GB per tensor): element offsets past 2^31,
    byte offsets past 4 GiB and a ragged tail of 5 after the last 8-wide vector.

    prev_i = 1 + (i mod 7), cur = 1.25 prev and residual_i = (i mod 5)/2 - 1.
    Every value, difference and per-thread fp32 partial sum is a multiple of
    1/4 far below 2^22, so all of them are exact in bf16 and fp32.
    Hence rel_l1 = 1/4 exactly, Σ|prev| = 28 q + r(r+1)/2 with n = 7q + r,
    and out = cur + residual holds element for element, by the plain cache
    apply and by the fused drift + apply alike."""
    n = 2 ** 31 + 13
    chunk = 2 ** 28
    prev = torch.empty(n, dtype=torch.bfloat16, device=DEV)
    cur = torch.empty_like(prev)
    res = torch.empty_like(prev)
    for s in range(0, n, chunk):
        i = torch.arange(s, min(n, s + chunk), device=DEV, dtype=torch.int64)
        p = (1 + i % 7).to(torch.float32)
        prev[s:s + i.numel()] = p.to(torch.bfloat16)
        cur[s:s + i.numel()] = (1.25 * p).to(torch.bfloat16)
        res[s:s + i.numel()] = ((i % 5).to(torch.float32) * 0.5 - 1.0).to(torch.bfloat16)
        del i, p
    q, r = divmod(n, 7)
    den = 28 * q + r * (r + 1) // 2

    rel, sums = acid.acid_drift_signal(prev, cur)
    assert rel.item() == 0.25
    assert sums.cpu().tolist() == [den / 4, float(den)]

    def check_out(out):
        for s in range(0, n, chunk):
            i = torch.arange(s, min(n, s + chunk), device=DEV, dtype=torch.int64)
            want = (1.25 * (1 + i % 7).to(torch.float32) + (i % 5).to(torch.float32) * 0.5 - 1.0).to(torch.bfloat16)
            assert torch.equal(out[s:s + i.numel()], want), f"chunk at {s}"
            del i, want

    out = acid.acid_cache_apply(cur, res)
    check_out(out)
    out.zero_()
    out, rel2, sums2 = acid.acid_drift_apply(prev, cur, res, out=out)
    assert rel2.item() == 0.25 and sums2.cpu().tolist() == [den / 4, float(den)]
    check_out(out)
    del prev, cur, res, out
    torch.cuda.empty_cache()


@pytest.mark.parametrize("rows,d", [(32760, 1536), (2049, 256), (777, 3072), (5, 1920), (1, 8)])
def test_temni_drift_matches_oracle(acid, rows, d):
    """acid_temni_drift: the TeaCache signal formed from two consecutive steps'
    fp32 patch embeddings and block-0 modulations, against the oracle's
    LayerNorm-modulate and relative L1 (Sec. 2, "TeaCache").  Shapes: the
    Wan step's 32760 x 1536, row counts that leave partial groups of rows per
    CTA, the widest rows (3072), a width that is not a multiple of 256, and
    a single 8-wide row."""
    rng = np.random.default_rng(rows + d)
    h_prev = rng.normal(size=(rows, d)).astype(np.float32)
    h_cur = (h_prev + 0.05 * rng.normal(size=(rows, d))).astype(np.float32)
    mod_prev = (0.3 * rng.normal(size=2 * d)).astype(np.float32)
    mod_cur = (mod_prev + 0.01 * rng.normal(size=2 * d)).astype(np.float32)
    t = {k: torch.from_numpy(v).to(DEV) for k, v in (("hp", h_prev), ("hc", h_cur), ("mp", mod_prev), ("mc", mod_cur))}
    rel, sums = acid.acid_temni_drift(t["hp"], t["hc"], t["mp"], t["mc"], eps=1e-6)
    torch.cuda.synchronize()
    acid.check_device_error()
    up = O.modulate(O.layer_norm(h_prev, 1e-6), mod_prev[:d], mod_prev[d:])
    uc = O.modulate(O.layer_norm(h_cur, 1e-6), mod_cur[:d], mod_cur[d:])
    ref = O.rel_l1(up, uc)
    assert abs(rel.item() - ref) <= DRIFT_RTOL * ref, (rel.item(), ref)
    np.testing.assert_allclose(sums.cpu().numpy(), [np.abs(uc - up).sum(), np.abs(up).sum()], rtol=DRIFT_RTOL)


def test_temni_drift_identical_steps_and_empty(acid):
    """The same h and modulation on both steps give exactly 0; zero rows give 0."""
    rng = np.random.default_rng(5)
    h = torch.from_numpy(rng.normal(size=(300, 1536)).astype(np.float32)).to(DEV)
    m = torch.from_numpy((0.2 * rng.normal(size=3072)).astype(np.float32)).to(DEV)
    rel, sums = acid.acid_temni_drift(h, h, m, m)
    assert rel.item() == 0.0 and sums[0].item() == 0.0 and sums[1].item() > 0
    e = torch.empty((0, 1536), dtype=torch.float32, device=DEV)
    rel, sums = acid.acid_temni_drift(e, e, m, m)
    assert rel.item() == 0.0 and sums.cpu().tolist() == [0.0, 0.0]
