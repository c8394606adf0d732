"""GPU parity of the kernel-level entry points (through the C ABI) against
the CPU oracle's definitions of the same operations."""

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


DEV = "cuda"


def _bf(a):
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(DEV, torch.bfloat16)


def _f32(a):
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(DEV)


def _rel_l2(got, ref):
    return float(np.linalg.norm(got - ref) / max(np.linalg.norm(ref), 1e-30))


# ---------------------------------------------------------------------------
# Linear layers (tcgen05 GEMM, bf16 in / fp32 accumulate)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("M,K,N", [(128, 64, 64), (200, 128, 256), (333, 192, 128), (1000, 1536, 768),
                                   (64, 4096, 3072), (257, 64, 96)])
def test_linear_bf16_bias(acid, M, K, N):
    rng = np.random.default_rng(M + K + N)
    a = S.round_to_bf16(rng.normal(size=(M, K)).astype(np.float32))
    w = S.round_to_bf16((0.05 * rng.normal(size=(N, K))).astype(np.float32))
    b = rng.normal(size=N).astype(np.float32)
    out = acid.acid_linear_forward(_bf(a), _bf(w), _f32(b), out_fp32=True)
    ref = O.linear(a, w, b)
    got = out.cpu().numpy()
    # fp32 accumulation of bf16 products: error ~ sqrt(K) * 2^-24 * |terms|
    assert np.abs(got - ref).max() <= 1e-4 * (1 + np.abs(ref).max()), np.abs(got - ref).max()


@pytest.mark.parametrize("epi", ["bias", "gelu", "gated_res", "res"])
def test_linear_bf16_epilogues(acid, epi):
    M, K, N = 300, 256, 512
    rng = np.random.default_rng(7)
    a = S.round_to_bf16(rng.normal(size=(M, K)).astype(np.float32))
    w = S.round_to_bf16((0.1 * rng.normal(size=(N, K))).astype(np.float32))
    b = rng.normal(size=N).astype(np.float32)
    g = rng.normal(size=N).astype(np.float32)
    r = S.round_to_bf16(rng.normal(size=(M, N)).astype(np.float32))
    res = _bf(r)
    out = acid.acid_linear_forward(_bf(a), _bf(w), _f32(b), epilogue=epi, gate=_f32(g),
                                   residual=res if epi in ("gated_res", "res") else None,
                                   out=res if epi in ("gated_res", "res") else None)
    acc = O.linear(a, w, b)
    ref = {"bias": acc, "gelu": O.gelu_tanh(acc), "gated_res": r + g * acc, "res": r + acc}[epi]
    got = out.float().cpu().numpy()
    # bf16 output: one rounding (2^-9 relative) plus the tanh approximation for GELU
    assert np.abs(got - ref).max() <= 2 ** -8 * (np.abs(ref).max() + 1), np.abs(got - ref).max()
    assert _rel_l2(got, ref) <= 4e-3


@pytest.mark.parametrize("M,K,N", [(891, 320, 512), (1000, 64, 768), (2500, 1096, 1024)])
@pytest.mark.parametrize("epi,fp32", [("bias", True), ("gelu", False), ("gated_res", False), ("gated_res", True),
                                      ("res", True)])
def test_linear_bf16_many_row_blocks(acid, M, K, N, epi, fp32):
    """The 256-wide tile path over several row blocks, including an odd count
    and a ragged last block (891 rows), fewer k-blocks than pipeline stages, a
    K that wraps the stage ring several times with a partial last k-block
    (1096), and every epilogue with bf16 and fp32 output/residual."""
    rng = np.random.default_rng(M + 7 * K + N)
    a = S.round_to_bf16(rng.normal(size=(M, K)).astype(np.float32))
    w = S.round_to_bf16((0.1 * rng.normal(size=(N, K))).astype(np.float32))
    b = rng.normal(size=N).astype(np.float32)
    g = rng.normal(size=N).astype(np.float32)
    r = rng.normal(size=(M, N)).astype(np.float32)
    if not fp32:
        r = S.round_to_bf16(r)
    has_res = epi in ("gated_res", "res")
    res = (_f32(r) if fp32 else _bf(r)) if has_res else None
    out = acid.acid_linear_forward(_bf(a), _bf(w), _f32(b), epilogue=epi, gate=_f32(g), residual=res, out=res,
                                   out_fp32=fp32)
    acc = O.linear(a, w, b)
    ref = {"bias": acc, "gelu": O.gelu_tanh(acc), "gated_res": r + g * acc, "res": r + acc}[epi]
    got = out.float().cpu().numpy()
    tol = 1e-4 if (fp32 and epi != "gelu") else 2 ** -8
    assert np.abs(got - ref).max() <= tol * (np.abs(ref).max() + 1), np.abs(got - ref).max()


@pytest.mark.parametrize("M,K,N", [(700, 192, 640), (300, 128, 1920), (513, 64, 5760), (129, 96, 160)])
@pytest.mark.parametrize("epi", ["bias", "gelu", "gated_res", "res"])
def test_linear_bf16_partial_last_column_tile(acid, M, K, N, epi):
    """N not a multiple of the 256-wide tile: the last column tile reads
    zero-filled weight rows and stores only its valid columns (CogVideoX
    widths 1920 and 5760 among them)."""
    rng = np.random.default_rng(M * 7 + N)
    a = S.round_to_bf16(rng.normal(size=(M, K)).astype(np.float32))
    w = S.round_to_bf16((0.1 * rng.normal(size=(N, K))).astype(np.float32))
    b = rng.normal(size=N).astype(np.float32)
    g = rng.normal(size=N).astype(np.float32)
    r = rng.normal(size=(M, N)).astype(np.float32)
    has_res = epi in ("gated_res", "res")
    res = _f32(r) if has_res else None
    out = acid.acid_linear_forward(_bf(a), _bf(w), _f32(b), epilogue=epi, gate=_f32(g), residual=res, out=res,
                                   out_fp32=True)
    acc = O.linear(a, w, b)
    ref = {"bias": acc, "gelu": O.gelu_tanh(acc), "gated_res": r + g * acc, "res": r + acc}[epi]
    got = out.cpu().numpy()
    tol = 2 ** -9 if epi == "gelu" else 1e-4
    assert np.abs(got - ref).max() <= tol * (np.abs(ref).max() + 1), np.abs(got - ref).max()


@pytest.mark.parametrize("M,K,N", [(891, 2112, 1024), (130, 4160, 2304), (1000, 64, 4096), (257, 2176, 160)])
@pytest.mark.parametrize("epi,fp32", [("bias", True), ("gelu", False), ("gated_res", True), ("res", False)])
def test_linear_bf16_pair_tiles(acid, M, K, N, epi, fp32):
    """Shapes that run on SM pairs (N or K above 2048): 256-row pair tiles
    whose second CTA holds a ragged (123, 2) or a full last row block, a K
    that is a multiple of 64 with many stage-ring wraps, N a multiple of 256,
    and a 160-wide output whose second CTA's weight rows lie beyond N."""
    rng = np.random.default_rng(M + 3 * K + 5 * N)
    a = S.round_to_bf16(rng.normal(size=(M, K)).astype(np.float32))
    w = S.round_to_bf16((0.05 * rng.normal(size=(N, K))).astype(np.float32))
    b = rng.normal(size=N).astype(np.float32)
    g = rng.normal(size=N).astype(np.float32)
    r = rng.normal(size=(M, N)).astype(np.float32)
    if not fp32:
        r = S.round_to_bf16(r)
    has_res = epi in ("gated_res", "res")
    res = (_f32(r) if fp32 else _bf(r)) if has_res else None
    out = acid.acid_linear_forward(_bf(a), _bf(w), _f32(b), epilogue=epi, gate=_f32(g), residual=res, out=res,
                                   out_fp32=fp32)
    acc = O.linear(a, w, b)
    ref = {"bias": acc, "gelu": O.gelu_tanh(acc), "gated_res": r + g * acc, "res": r + acc}[epi]
    got = out.float().cpu().numpy()
    tol = 1e-4 if (fp32 and epi != "gelu") else 2 ** -8
    assert np.abs(got - ref).max() <= tol * (np.abs(ref).max() + 1), np.abs(got - ref).max()


@pytest.mark.parametrize("K,epi,fp32", [(1536, "gated_res", True), (1536, "res", True), (1536, "bias", False),
                                        (1536, "gelu", True), (8960, "gated_res", False)])
def test_linear_bf16_wan_shapes_last_rows(acid, K, epi, fp32):
    """The Wan-1.3B projections with N = 1536 over 32760 rows (output
    projections, cross-attention query, FFN2) and a GELU output, at full size:
    the persistent launch's last, partly filled round of tiles and the ragged
    last row tile (32760 = 255 x 128 + 120).  Every one of the last 640 rows,
    and rows spread over the rest, are compared with the oracle."""
    M, N = 32760, 1536
    rng = np.random.default_rng(K + N)
    a = S.round_to_bf16(rng.normal(size=(M, K)).astype(np.float32))
    w = S.round_to_bf16((0.03 * rng.normal(size=(N, K))).astype(np.float32))
    b = rng.normal(size=N).astype(np.float32)
    g = rng.normal(size=N).astype(np.float32)
    r = rng.normal(size=(M, N)).astype(np.float32)
    if not fp32:
        r = S.round_to_bf16(r)
    # the residual has the output's dtype and is updated in place
    out = _f32(r) if fp32 else _bf(r)
    acid.acid_linear_forward(_bf(a), _bf(w), _f32(b), epilogue=epi, gate=_f32(g),
                             residual=out if epi in ("gated_res", "res") else None, out=out, out_fp32=fp32)
    rows = np.array(sorted(set(range(M - 640, M)) | set(rng.integers(0, M - 640, size=64).tolist()) | {0, 1}))
    acc = O.linear(a[rows], w, b)
    ref = {"bias": acc, "gelu": O.gelu_tanh(acc), "gated_res": r[rows] + g * acc, "res": r[rows] + acc}[epi]
    got = out[torch.from_numpy(rows).to(DEV)].float().cpu().numpy()
    tol = 1e-4 if (fp32 and epi != "gelu") else 2 ** -8
    assert np.abs(got - ref).max() <= tol * (np.abs(ref).max() + 1), np.abs(got - ref).max()


def test_linear_bf16_offsets_past_32_bits(acid):
    """An output of 262181 x 8960 fp32 values (2.35e9 elements, 9.4 GB),
    updated in place by the gated-residual epilogue.  Rows from 239675 on
    start past element 2^31, so the residual reads and the stores there need
    64-bit offsets; the last row tile holds 37 rows.  Sampled rows, at both
    ends and around the 2^31 boundary, are compared with the oracle."""
    M, K, N = 262144 + 37, 64, 8960
    rng = np.random.default_rng(31)
    a = S.round_to_bf16(rng.normal(size=(M, K)).astype(np.float32))
    w = S.round_to_bf16((0.1 * rng.normal(size=(N, K))).astype(np.float32))
    b = rng.normal(size=N).astype(np.float32)
    g = rng.normal(size=N).astype(np.float32)

    def resid(rows):  # a closed-form residual, cheap to build on the device and on the host
        return ((rows[:, None] * 7 + np.arange(N)[None, :]) % 13).astype(np.float32) / 4 - 1.5

    res = torch.empty((M, N), dtype=torch.float32, device=DEV)
    cols = torch.arange(N, device=DEV, dtype=torch.int64)
    for r0 in range(0, M, 16384):
        rows = torch.arange(r0, min(M, r0 + 16384), device=DEV, dtype=torch.int64)
        res[r0:r0 + rows.numel()] = ((rows[:, None] * 7 + cols[None, :]) % 13).float() / 4 - 1.5
        del rows
    out = acid.acid_linear_forward(_bf(a), _bf(w), _f32(b), epilogue="gated_res", gate=_f32(g), residual=res,
                                   out=res, out_fp32=True)
    rows = np.array([0, 1, 127, 128, 239674, 239675, 239676, 262015, 262143, 262144, 262180])
    got = out[torch.from_numpy(rows).to(DEV)].cpu().numpy()
    ref = resid(rows) + g * O.linear(a[rows], w, b)
    assert np.abs(got - ref).max() <= 1e-4 * (np.abs(ref).max() + 1), np.abs(got - ref).max()
    del res, out
    torch.cuda.empty_cache()


@pytest.mark.parametrize("M,K,N", [(1, 64, 64), (7, 8, 32), (127, 72, 96), (129, 200, 256), (3, 4104, 128)])
def test_linear_bf16_edge_shapes(acid, M, K, N):
    """Single rows, K below / not a multiple of the 64-wide k-block (zero-filled
    by TMA), N a multiple of 32 only, and a ragged long K."""
    rng = np.random.default_rng(M * 1000 + K)
    a = S.round_to_bf16(rng.normal(size=(M, K)).astype(np.float32))
    w = S.round_to_bf16((0.1 * rng.normal(size=(N, K))).astype(np.float32))
    b = rng.normal(size=N).astype(np.float32)
    got = acid.acid_linear_forward(_bf(a), _bf(w), _f32(b), out_fp32=True).cpu().numpy()
    ref = O.linear(a, w, b)
    assert np.abs(got - ref).max() <= 1e-4 * (1 + np.abs(ref).max())


def test_linear_fp32(acid):
    M, K, N = 77, 96, 130
    rng = np.random.default_rng(8)
    a, w, b = rng.normal(size=(M, K)), rng.normal(size=(N, K)), rng.normal(size=N)
    out = acid.acid_linear_forward(_f32(a), _f32(w), _f32(b), epilogue="gelu")
    ref = O.gelu_tanh(O.linear(a.astype(np.float32), w.astype(np.float32), b.astype(np.float32)))
    assert _rel_l2(out.cpu().numpy(), ref) <= 1e-5


def test_linear_rejects_bad_shapes(acid):
    from paper_2607_12358_gb300._capi import AcidError
    a = torch.zeros(10, 64, device=DEV, dtype=torch.bfloat16)
    w = torch.zeros(40, 64, device=DEV, dtype=torch.bfloat16)  # N % 32 != 0
    with pytest.raises(AcidError):
        acid.acid_linear_forward(a, w)


# ---------------------------------------------------------------------------
# Attention (tcgen05 flash attention)
# ---------------------------------------------------------------------------

def _attn_case(nq, nk, H, D, seed, qscale=1.0):
    rng = np.random.default_rng(seed)
    q = S.round_to_bf16((qscale * rng.normal(size=(nq, H * D))).astype(np.float32))
    k = S.round_to_bf16(rng.normal(size=(nk, H * D)).astype(np.float32))
    v = S.round_to_bf16(rng.normal(size=(nk, H * D)).astype(np.float32))
    ref = O.attention(q.reshape(nq, H, D), k.reshape(nk, H, D), v.reshape(nk, H, D)).reshape(nq, H * D)
    return q, k, v, ref


@pytest.mark.parametrize("nq,nk,H,D,qscale", [(128, 128, 1, 128, 1.0), (300, 300, 2, 128, 1.0),
                                              (300, 257, 2, 64, 2.0), (1000, 512, 3, 128, 3.0),
                                              (129, 1000, 2, 64, 4.0), (2048, 2048, 2, 128, 1.0),
                                              (1000, 2000, 3, 64, 3.0)])
def test_attention_bf16(acid, nq, nk, H, D, qscale):
    q, k, v, ref = _attn_case(nq, nk, H, D, nq + nk, qscale)
    out = acid.acid_attention_forward(_bf(q), _bf(k), _bf(v), H)
    got = out.float().cpu().numpy()
    assert _rel_l2(got, ref) <= 1e-2, _rel_l2(got, ref)
    assert np.abs(got - ref).max() <= 5e-2


@pytest.mark.parametrize("nq,H,D", [(2560, 16, 128), (2048, 19, 64), (32760, 12, 128)])
def test_attention_split_last_wave(acid, nq, H, D):
    """With a workspace, the work items of a partial last wave are split along
    the key range and merged; the result matches the oracle and the unsplit
    launch (the largest case is the Wan self-attention shape, checked on
    sampled rows)."""
    rng = np.random.default_rng(nq + H)
    q = S.round_to_bf16((2.0 * rng.normal(size=(nq, H * D))).astype(np.float32))
    k = S.round_to_bf16(rng.normal(size=(nq, H * D)).astype(np.float32))
    v = S.round_to_bf16(rng.normal(size=(nq, H * D)).astype(np.float32))
    ws = torch.empty(acid.attention_workspace_size(D), dtype=torch.uint8, device=DEV)
    split = acid.acid_attention_forward(_bf(q), _bf(k), _bf(v), H, workspace=ws).float().cpu().numpy()
    plain = acid.acid_attention_forward(_bf(q), _bf(k), _bf(v), H).float().cpu().numpy()
    rows = np.unique(np.concatenate([np.arange(0, nq, max(1, nq // 40)), np.arange(nq - 300, nq)]))
    ref = O.attention(q[rows].reshape(-1, H, D), k.reshape(nq, H, D), v.reshape(nq, H, D)).reshape(len(rows), H * D)
    assert _rel_l2(split[rows], ref) <= 1e-2
    assert np.abs(split[rows] - ref).max() <= 5e-2
    assert _rel_l2(split, plain) <= 5e-3


@pytest.mark.parametrize("nq,nk,H,D", [(8192, 100, 12, 128), (8192, 500, 24, 64), (8192, 512, 12, 128)])
def test_attention_persistent_items(acid, nq, nk, H, D):
    """Persistent CTAs walk several (query-tile pair, head) items: 384 or 768
    items over one CTA per SM (head dim 128) or two (64).  The query scale
    differs per head (logit spreads from about 1 to about 8), so a running max
    or sum carried from one item into the next would show; with nk = 100
    every step is an item boundary and the only key tile is masked.  Every
    row is checked against the oracle, with and without a workspace (short
    key ranges leave it unused)."""
    rng = np.random.default_rng(nq + nk + H)
    scale = np.repeat(1.0 + 7.0 * (np.arange(H) % 3 == 0), D)[None, :]
    q = S.round_to_bf16((scale * rng.normal(size=(nq, H * D))).astype(np.float32))
    k = S.round_to_bf16(rng.normal(size=(nk, H * D)).astype(np.float32))
    v = S.round_to_bf16(rng.normal(size=(nk, H * D)).astype(np.float32))
    ref = O.attention(q.reshape(nq, H, D), k.reshape(nk, H, D), v.reshape(nk, H, D)).reshape(nq, H * D)
    ws = torch.empty(acid.attention_workspace_size(D), dtype=torch.uint8, device=DEV)
    for w in (None, ws):
        got = acid.acid_attention_forward(_bf(q), _bf(k), _bf(v), H, workspace=w).float().cpu().numpy()
        assert _rel_l2(got, ref) <= 1e-2, (w is None, _rel_l2(got, ref))
        assert np.abs(got - ref).max() <= 5e-2, (w is None, np.abs(got - ref).max())


@pytest.mark.parametrize("nq,nk,H,D", [(131072, 512, 12, 128), (65536, 500, 24, 64)])
def test_attention_persistent_many_items(acid, nq, nk, H, D):
    """Long runs of items per persistent CTA: 6144 items over 152 CTAs (about
    40 each, 160 key-tile steps whose barrier phases and ring slots carry
    across items) at head dim 128, and over 304 CTAs (about 20 each, masked
    last tile) at head dim 64.  Sampled rows, the first and last items among
    them, against the oracle."""
    rng = np.random.default_rng(nq + nk)
    q = S.round_to_bf16((2.0 * rng.standard_normal(size=(nq, H * D), dtype=np.float32)))
    k = S.round_to_bf16(rng.standard_normal(size=(nk, H * D), dtype=np.float32))
    v = S.round_to_bf16(rng.standard_normal(size=(nk, H * D), dtype=np.float32))
    got = acid.acid_attention_forward(_bf(q), _bf(k), _bf(v), H).float().cpu().numpy()
    acid.check_device_error()
    rows = np.unique(np.concatenate([np.arange(0, 300), np.arange(0, nq, nq // 97), np.arange(nq - 300, nq)]))
    ref = O.attention(q[rows].reshape(-1, H, D), k.reshape(nk, H, D), v.reshape(nk, H, D)).reshape(len(rows), H * D)
    assert _rel_l2(got[rows], ref) <= 1e-2, _rel_l2(got[rows], ref)
    assert np.abs(got[rows] - ref).max() <= 5e-2


def test_attention_one_key_returns_value(acid):
    q, k, v, ref = _attn_case(200, 1, 2, 128, 3)
    got = acid.acid_attention_forward(_bf(q), _bf(k), _bf(v), 2).float().cpu().numpy()
    np.testing.assert_array_equal(got, np.broadcast_to(v, got.shape))


def test_attention_peaky_rescaling(acid):
    """Logits spanning far more than 2^8 across key tiles exercise the
    deferred rescaling of the output accumulator."""
    q, k, v, ref = _attn_case(256, 1024, 1, 128, 5, qscale=1.0)
    k = k.copy()
    k[900:] *= 12.0  # late keys dominate: the running max jumps in the last tiles
    k = S.round_to_bf16(k)
    ref = O.attention(q.reshape(256, 1, 128), k.reshape(1024, 1, 128), v.reshape(1024, 1, 128)).reshape(256, 128)
    got = acid.acid_attention_forward(_bf(q), _bf(k), _bf(v), 1).float().cpu().numpy()
    assert _rel_l2(got, ref) <= 1e-2


@pytest.mark.parametrize("D", [64, 128])
def test_attention_rescale_diverging_rows(acid, D):
    """Key tiles whose logits grow tile by tile (scale 1 + 0.6 j on tile j)
    and query rows of seven different norms: rows cross the 2^8 rescale
    threshold at different tiles, so within a warp some rows keep the
    one-pass softmax while others reload S and move their reference.  The
    last key tile is partial (masked)."""
    nq, nk, H = 300, 1000, 2
    bkv = 64 if D == 64 else 128
    rng = np.random.default_rng(70 + D)
    q = rng.normal(size=(nq, H * D)) * (0.5 + 0.5 * (np.arange(nq) % 7))[:, None]
    k = rng.normal(size=(nk, H * D)) * (1.0 + 0.6 * (np.arange(nk) // bkv))[:, None]
    v = rng.normal(size=(nk, H * D))
    q, k, v = (S.round_to_bf16(x.astype(np.float32)) for x in (q, k, v))
    ref = O.attention(q.reshape(nq, H, D), k.reshape(nk, H, D), v.reshape(nk, H, D)).reshape(nq, H * D)
    got = acid.acid_attention_forward(_bf(q), _bf(k), _bf(v), H).float().cpu().numpy()
    assert _rel_l2(got, ref) <= 1e-2, _rel_l2(got, ref)
    assert np.abs(got - ref).max() <= 5e-2


def test_attention_fp32(acid):
    rng = np.random.default_rng(11)
    q, k, v = (rng.normal(size=(70, 128)) for _ in range(3))
    ref = O.attention(q.reshape(70, 2, 64), k.reshape(70, 2, 64), v.reshape(70, 2, 64)).reshape(70, 128)
    got = acid.acid_attention_forward(_f32(q), _f32(k), _f32(v), 2).cpu().numpy()
    assert _rel_l2(got, ref) <= 1e-5


# ---------------------------------------------------------------------------
# adaLN LayerNorm
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("d", [256, 1536, 1920, 3072])
def test_layernorm_mod(acid, d):
    rng = np.random.default_rng(d)
    x = S.round_to_bf16((2.0 + 3.0 * rng.normal(size=(333, d))).astype(np.float32))
    sh, sc = rng.normal(size=d).astype(np.float32), rng.normal(size=d).astype(np.float32)
    ref = O.modulate(O.layer_norm(x), sh, sc)
    got = acid.acid_layernorm_mod(_bf(x), _f32(sh), _f32(sc), out_dtype=torch.float32).cpu().numpy()
    assert np.abs(got - ref).max() <= 1e-4 * (1 + np.abs(ref).max())
    got16 = acid.acid_layernorm_mod(_bf(x), _f32(sh), _f32(sc)).float().cpu().numpy()
    assert np.abs(got16 - ref).max() <= 2 ** -8 * (1 + np.abs(ref).max())


@pytest.mark.parametrize("d", [1536, 3072])
def test_layernorm_mod_fp32_input_into_bf16_buffer(acid, d):
    """The block's case: the fp32 residual stream normalised into a bf16 GEMM
    operand, written into a caller-given buffer (one bf16 rounding of the
    fp64 reference)."""
    rng = np.random.default_rng(d + 1)
    x = (0.5 + 4.0 * rng.normal(size=(1001, d))).astype(np.float32)
    sh, sc = rng.normal(size=d).astype(np.float32), rng.normal(size=d).astype(np.float32)
    ref = O.modulate(O.layer_norm(x), sh, sc)
    y = torch.full((1001, d), float("nan"), dtype=torch.bfloat16, device=DEV)
    got = acid.acid_layernorm_mod(_f32(x), _f32(sh), _f32(sc), out_dtype=torch.bfloat16, out=y)
    assert got.data_ptr() == y.data_ptr()
    got = got.float().cpu().numpy()
    assert np.abs(got - ref).max() <= 2 ** -8 * (1 + np.abs(ref).max())


def test_empty_inputs_return_without_launching(acid):
    """Zero rows: the linear layer, attention, LayerNorm-mod and cache apply
    return OK and launch nothing."""
    n0 = acid.launch_count()
    a = torch.empty(0, 128, dtype=torch.bfloat16, device=DEV)
    w = torch.zeros(256, 128, dtype=torch.bfloat16, device=DEV)
    assert acid.acid_linear_forward(a, w).shape == (0, 256)
    q = torch.empty(0, 256, dtype=torch.bfloat16, device=DEV)
    kv = torch.zeros(64, 256, dtype=torch.bfloat16, device=DEV)
    assert acid.acid_attention_forward(q, kv, kv, 2).shape == (0, 256)
    x = torch.empty(0, 256, dtype=torch.bfloat16, device=DEV)
    assert acid.acid_layernorm_mod(x).shape[0] == 0
    e = torch.empty(0, dtype=torch.bfloat16, device=DEV)
    acid.acid_cache_apply(e, e, out=e)
    torch.cuda.synchronize()
    acid.check_device_error()
    assert acid.launch_count() == n0
