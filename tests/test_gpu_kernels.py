"""Kernel-level parity on the GPU: every hot-path kernel of libsgd, called through
the C ABI (include/sgd_kernels.h), against the CPU oracle's definition of the same
operation, on seeded inputs with ragged tails (M, N, K, keys not tile multiples).

Operands and stored activations are fp16 (fp32 accumulation).  Tolerances: an
fp16 output may differ from the fp32 oracle by the rounding of the result
(relative 2^-11) plus fp32 accumulation-order noise; fp32 outputs (the residual
update) by accumulation order only."""
import math

import numpy as np
import pytest
import torch

from oracle import denoiser as odn
from paper_2609_29505_gb300 import synth

pytestmark = pytest.mark.gpu

F16_REL = 2.0 ** -11


@pytest.fixture(scope="module")
def B():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    from paper_2609_29505_gb300 import binding, build
    build.build()
    binding.lib()
    return binding


def _rand(rng, shape, scale=1.0, dtype=torch.float16):
    return torch.from_numpy((rng.standard_normal(shape) * scale).astype(np.float32)).to(dtype)


def _f(t):
    return t.float().cpu().numpy()


def _check_f16(got, want, extra_abs=0.0):
    got = _f(got)
    scale = float(np.sqrt(np.mean(want.astype(np.float64) ** 2))) + 1e-30
    bound = F16_REL * np.abs(want) + 2e-5 * scale + extra_abs
    bad = np.abs(got - want) > bound
    assert not bad.any(), (f"{bad.sum()} of {bad.size} outside fp16 rounding; max err "
                           f"{np.max(np.abs(got - want)):.3e}, rms(want) {scale:.3e}")


# sgd_kernel_gemm variant codes (include/sgd_kernels.h)
VARIANTS = [0, 3, 5, 6, 7, 8, 9, 10, 11, 12, 1]
VARIANT_IDS = ["tcgen05", "tcgen05_bk32", "tcgen05_epi4",
               "tcgen05_epi8", "tcgen05_bn128", "tcgen05_dp", "tcgen05_streamk", "tcgen05_bn224",
               "tcgen05_mfast", "tcgen05_grouped", "simt"]

GEMM_SHAPES = [(64, 256, 256), (300, 520, 688), (129, 264, 72), (1000, 1376, 512), (4128, 1024, 2048)]


@pytest.mark.parametrize("simt", VARIANTS, ids=VARIANT_IDS)
@pytest.mark.parametrize("M,N,K", GEMM_SHAPES)
def test_gemm_bf16(B, M, N, K, simt):
    rng = np.random.default_rng(M + N + K)
    A = _rand(rng, (M, K)).cuda()
    W = _rand(rng, (N, K), 1 / math.sqrt(K)).cuda()
    out = torch.empty(M, N, dtype=torch.float16, device="cuda")
    epi = B.sgd_epilogue_args(kind=B.EPI_F16, out=out.data_ptr(), ldo=N)
    B.sgd_kernel_gemm(A, W, M, N, K, epi, use_simt=simt)
    torch.cuda.synchronize()
    assert B.sgd_kernel_status() == 0
    _check_f16(out, odn.linear(_f(A), _f(W)))


@pytest.mark.parametrize("simt", VARIANTS, ids=VARIANT_IDS)
@pytest.mark.parametrize("gated", [False, True])
def test_gemm_delta_residual_and_cache(B, simt, gated):
    rng = np.random.default_rng(5)
    M, N, K, rpb = 520, 264, 688, 130
    A = _rand(rng, (M, K)).cuda()
    W = _rand(rng, (N, K), 1 / math.sqrt(K)).cuda()
    h0 = torch.from_numpy(rng.standard_normal((M, N)).astype(np.float32)).cuda()
    h = h0.clone()
    cache = torch.zeros(M, N, dtype=torch.float16, device="cuda")
    gate = torch.from_numpy(rng.standard_normal((M // rpb, N)).astype(np.float32)).cuda()
    epi = B.sgd_epilogue_args(kind=B.EPI_DELTA, h=h.data_ptr(), ldh=N, cache=cache.data_ptr(),
                              ld_cache=N, gate=gate.data_ptr() if gated else None, ld_gate=N,
                              rows_per_batch=rpb)
    B.sgd_kernel_gemm(A, W, M, N, K, epi, use_simt=simt)
    torch.cuda.synchronize()
    delta = odn.linear(_f(A), _f(W))
    if gated:
        delta = delta * np.repeat(gate.cpu().numpy(), rpb, axis=0)
    want_h = h0.cpu().numpy() + delta
    np.testing.assert_allclose(h.cpu().numpy(), want_h, rtol=2e-5, atol=2e-5)
    _check_f16(cache, delta)


@pytest.mark.parametrize("simt", VARIANTS, ids=VARIANT_IDS)
@pytest.mark.parametrize("act", [0, 1])
def test_gemm_gated_activation(B, simt, act):
    rng = np.random.default_rng(6)
    M, f, K = 300, 688, 256
    A = _rand(rng, (M, K)).cuda()
    W = _rand(rng, (2 * f, K), 1 / math.sqrt(K)).cuda()
    out = torch.empty(M, f, dtype=torch.float16, device="cuda")
    epi = B.sgd_epilogue_args(kind=B.EPI_GATED, out=out.data_ptr(), ldo=f, act=act)
    B.sgd_kernel_gemm(A, W, M, f, K, epi, use_simt=simt)
    torch.cuda.synchronize()
    u = odn.linear(_f(A), _f(W))
    want = odn.silu(u[:, :f]) * u[:, f:] if act == 0 else u[:, :f] * odn.gelu_erf(u[:, f:])
    _check_f16(out, want, extra_abs=1e-4 * float(np.abs(want).max()))


@pytest.mark.parametrize("simt", VARIANTS, ids=VARIANT_IDS)
@pytest.mark.parametrize("act", [0, 1])
def test_gemm_gelu(B, simt, act):
    rng = np.random.default_rng(7)
    M, N, K = 200, 1152, 288
    A = _rand(rng, (M, K)).cuda()
    W = _rand(rng, (N, K), 1 / math.sqrt(K)).cuda()
    out = torch.empty(M, N, dtype=torch.float16, device="cuda")
    epi = B.sgd_epilogue_args(kind=B.EPI_GELU, out=out.data_ptr(), ldo=N, act=act)
    B.sgd_kernel_gemm(A, W, M, N, K, epi, use_simt=simt)
    torch.cuda.synchronize()
    u = odn.linear(_f(A), _f(W))
    want = odn.gelu_erf(u) if act else odn.gelu_tanh(u)
    _check_f16(out, want, extra_abs=1e-4 * float(np.abs(want).max()))


@pytest.mark.parametrize("simt", VARIANTS, ids=VARIANT_IDS)
@pytest.mark.parametrize("dh", [64, 128])
def test_gemm_rope_epilogue(B, simt, dh):
    rng = np.random.default_rng(8)
    H, n_tok, bsz = 4, 96, 3
    d = H * dh
    M, N, K = bsz * n_tok, 3 * d, d
    A = _rand(rng, (M, K)).cuda()
    W = _rand(rng, (N, K), 1 / math.sqrt(K)).cuda()
    half = dh // 2
    pos = np.arange(n_tok, dtype=np.float64)[:, None]
    freq = 10000.0 ** (-np.arange(half) * 2.0 / dh)
    cos = torch.from_numpy(np.cos(pos * freq).astype(np.float32)).cuda()
    sin = torch.from_numpy(np.sin(pos * freq).astype(np.float32)).cuda()
    out = torch.empty(M, N, dtype=torch.float16, device="cuda")
    epi = B.sgd_epilogue_args(kind=B.EPI_ROPE, out=out.data_ptr(), ldo=N, rope_cos=cos.data_ptr(),
                              rope_sin=sin.data_ptr(), rope_tokens=n_tok, d_head=dh, rope_cols=2 * d)
    B.sgd_kernel_gemm(A, W, M, N, K, epi, use_simt=simt)
    torch.cuda.synchronize()
    qkv = odn.linear(_f(A), _f(W)).reshape(bsz, n_tok, 3, H, dh)
    want = qkv.copy()
    for j in range(2):  # q and k rotate, v does not
        x = qkv[:, :, j].transpose(0, 2, 1, 3)  # [b, H, n, dh]
        want[:, :, j] = odn.rope(x, np.arange(n_tok), 10000.0).transpose(0, 2, 1, 3)
    _check_f16(out, want.reshape(M, N), extra_abs=1e-4)


@pytest.mark.parametrize("impl", [0, 1, 2, 3], ids=["tcgen05", "mma_sync", "tcgen05_1tile", "tcgen05_2tile"])
@pytest.mark.parametrize("dh,H,nq,nkv,bsz", [(64, 4, 64, 64, 1), (72, 3, 136, 136, 2),
                                              (128, 2, 192, 192, 2), (64, 5, 200, 77, 2),
                                              (64, 4, 258, 258, 2), (128, 2, 33, 5, 3),
                                              (128, 3, 1024, 1024, 1), (64, 2, 300, 700, 2),
                                              (128, 2, 600, 333, 2), (64, 3, 512, 1024, 1)])
def test_attention(B, dh, H, nq, nkv, bsz, impl):
    rng = np.random.default_rng(dh + nq + nkv)
    d = H * dh
    q = _rand(rng, (bsz * nq, d), 1.5).cuda()
    k = _rand(rng, (bsz * nkv, d), 1.5).cuda()
    v = _rand(rng, (bsz * nkv, d)).cuda()
    o = torch.empty(bsz * nq, d, dtype=torch.float16, device="cuda")
    B.sgd_kernel_attention(q, d, k, v, d, o, d, bsz, nq, nkv, H, dh, impl=impl)
    torch.cuda.synchronize()
    want = odn.attention(_f(q).reshape(bsz, nq, d), _f(k).reshape(bsz, nkv, d),
                         _f(v).reshape(bsz, nkv, d), H).reshape(bsz * nq, d)
    got = _f(o)
    # P and O are rounded to fp16: relative error of a few fp16 ulps on O
    err = np.linalg.norm(got - want) / np.linalg.norm(want)
    assert err < 1.5e-3, err
    assert np.max(np.abs(got - want)) < 5e-3 * float(np.abs(want).max())
    assert B.sgd_kernel_status() == 0


@pytest.mark.parametrize("impl", [0, 2, 3], ids=["tcgen05", "tcgen05_1tile", "tcgen05_2tile"])
@pytest.mark.parametrize("dh", [64, 128])
def test_attention_growing_row_maxima(B, dh, impl):
    """Later key tiles carry larger scores, so row maxima grow by more than 2^8 from tile to
    tile and the accumulated O is rescaled in TMEM (the lazy-rescale path)."""
    rng = np.random.default_rng(dh + impl)
    H, nq, nkv, bsz = 2, 640, 640, 1
    d = H * dh
    q = _rand(rng, (bsz * nq, d), 1.0).cuda()
    kk = rng.standard_normal((bsz * nkv, d)).astype(np.float32)
    kk *= (1.0 + 1.5 * (np.arange(bsz * nkv) // 128))[:, None]  # tile j scaled by 1 + 1.5 j
    k = torch.from_numpy(kk).half().cuda()
    v = _rand(rng, (bsz * nkv, d)).cuda()
    o = torch.empty(bsz * nq, d, dtype=torch.float16, device="cuda")
    B.sgd_kernel_attention(q, d, k, v, d, o, d, bsz, nq, nkv, H, dh, impl=impl)
    torch.cuda.synchronize()
    want = odn.attention(_f(q).reshape(bsz, nq, d), _f(k).reshape(bsz, nkv, d),
                         _f(v).reshape(bsz, nkv, d), H).reshape(bsz * nq, d)
    got = _f(o)
    err = np.linalg.norm(got - want) / np.linalg.norm(want)
    assert err < 1.5e-3, err
    assert B.sgd_kernel_status() == 0


@pytest.mark.parametrize("kind,d", [(0, 256), (0, 4096), (1, 1280), (2, 1152), (1, 1024), (0, 2048),
                                    (1, 2056), (2, 12)])
def test_norm(B, kind, d):
    rng = np.random.default_rng(kind * 10000 + d)
    rows, rpb = 260, 130
    h = torch.from_numpy((rng.standard_normal((rows, d)) * 3 + 0.5).astype(np.float32)).cuda()
    g = _rand(rng, (d,), 0.1).float().add(1.0).to(torch.bfloat16).cuda() if kind != 2 else None
    b = _rand(rng, (d,), 0.1, torch.bfloat16).cuda() if kind == 1 else None
    out = torch.empty(rows, d, dtype=torch.float16, device="cuda")
    shift = scale = None
    if kind == 2:
        mod = torch.from_numpy(rng.standard_normal((rows // rpb, 2 * d)).astype(np.float32) * 0.3).cuda()
        shift, scale = mod[:, :d], mod[:, d:]
        B.sgd_kernel_norm(h, out, rows, d, kind, shift=mod, scale=mod[:, d:], ld_mod=2 * d,
                          rows_per_batch=rpb, eps=1e-6)
    else:
        B.sgd_kernel_norm(h, out, rows, d, kind, g=g, b=b, eps=1e-6)
    torch.cuda.synchronize()
    hn = h.cpu().numpy()
    if kind == 0:
        want = odn.rms_norm(hn, _f(g), 1e-6)
    elif kind == 1:
        want = odn.layer_norm(hn, _f(g), _f(b), 1e-6)
    else:
        x = odn.layer_norm(hn, None, None, 1e-6).reshape(rows // rpb, rpb, d)
        want = odn.modulate(x, shift.cpu().numpy(), scale.cpu().numpy()).reshape(rows, d)
    _check_f16(out, want, extra_abs=1e-5)


@pytest.mark.parametrize("n_caches", [1, 3, 17])
def test_frozen_run_sums_in_unit_order(B, n_caches):
    rng = np.random.default_rng(n_caches)
    n = 4128 * 64
    h0 = rng.standard_normal(n).astype(np.float32)
    caches = [_rand(rng, (n,)).cuda() for _ in range(n_caches)]
    h = torch.from_numpy(h0).cuda()
    B.sgd_kernel_frozen_run(h, caches)
    torch.cuda.synchronize()
    want = h0.copy()
    for c in caches:  # Algorithm 2: each frozen unit adds its cached Delta in graph order
        want = (want + _f(c)).astype(np.float32)
    np.testing.assert_array_equal(h.cpu().numpy(), want)


def test_gemm_large_sampled_rows_tcgen05(B):
    """LLaDA-sized projection (M = N = K = 4096) on tcgen05; 96 sampled rows checked."""
    rng = np.random.default_rng(9)
    M = N = K = 4096
    A = torch.randn(M, K, generator=torch.Generator().manual_seed(1)).to(torch.float16).cuda()
    W = (torch.randn(N, K, generator=torch.Generator().manual_seed(2)) / 64).to(torch.float16).cuda()
    out = torch.empty(M, N, dtype=torch.float16, device="cuda")
    epi = B.sgd_epilogue_args(kind=B.EPI_F16, out=out.data_ptr(), ldo=N)
    B.sgd_kernel_gemm(A, W, M, N, K, epi)
    torch.cuda.synchronize()
    rows = np.sort(rng.choice(M, 96, replace=False))
    want = odn.linear(_f(A[rows]), _f(W))
    _check_f16(out[rows], want)


@pytest.mark.parametrize("M,N,K,epi", [(4096, 4096, 4096, "f16"), (2048, 1152, 1152, "delta"),
                                       (1000, 1376, 512, "gelu"), (4096, 4096, 1024, "gated")])
def test_gemm_streamk_repeatable(B, M, N, K, epi):
    """Stream-K (leftover tiles split along K over all SMs, partial sums in a workspace):
    two launches in a row give identical bits (the partials are summed in a fixed order and
    the tile tickets are back at zero after each launch), and agree with the
    data-parallel schedule to fp16 rounding and with the oracle on sampled rows."""
    rng = np.random.default_rng(M + N + K + 1)
    gated = epi == "gated"
    A = _rand(rng, (M, K)).cuda()
    W = _rand(rng, (2 * N if gated else N, K), 1 / math.sqrt(K)).cuda()
    kind = {"f16": B.EPI_F16, "delta": B.EPI_DELTA, "gelu": B.EPI_GELU, "gated": B.EPI_GATED}[epi]

    def run(variant):
        if epi == "delta":
            h = torch.zeros(M, N, device="cuda")
            e = B.sgd_epilogue_args(kind=kind, h=h.data_ptr(), ldh=N)
            B.sgd_kernel_gemm(A, W, M, N, K, e, use_simt=variant)
            return h
        out = torch.empty(M, N, dtype=torch.float16, device="cuda")
        e = B.sgd_epilogue_args(kind=kind, out=out.data_ptr(), ldo=N)
        B.sgd_kernel_gemm(A, W, M, N, K, e, use_simt=variant)
        return out

    first, second, dp = run(9), run(9), run(8)
    torch.cuda.synchronize()
    assert B.sgd_kernel_status() == 0
    assert torch.equal(first, second)
    rows = np.sort(rng.choice(M, 64, replace=False))
    u = odn.linear(_f(A[rows]), _f(W))
    want = {"f16": u, "delta": u, "gelu": odn.gelu_tanh(u),
            "gated": odn.silu(u[:, :N]) * u[:, N:] if gated else None}[epi]
    if epi == "delta":
        np.testing.assert_allclose(_f(first[rows]), want, rtol=2e-5, atol=2e-5)
        np.testing.assert_allclose(_f(first), _f(dp), rtol=2e-5, atol=2e-5)
    else:
        extra = 1e-4 * float(np.abs(want).max())
        _check_f16(first[rows], want, extra_abs=extra)
        a, b = _f(first), _f(dp)  # two fp16 roundings of nearly equal sums: 1 ulp apart at most
        assert np.all(np.abs(a - b) <= 2.0 ** -10 * np.abs(b) + extra)


def test_f16_clamp_is_reported(B):
    """An fp16 store that has to clamp (|x| > 65504) raises the clamp flag, which
    sgd_kernel_f16_clamped reports once and clears; an in-range GEMM leaves it down."""
    M = N = K = 64
    A = torch.full((M, K), 300.0, dtype=torch.float16, device="cuda")
    W = torch.full((N, K), 300.0, dtype=torch.float16, device="cuda")
    out = torch.empty(M, N, dtype=torch.float16, device="cuda")
    B.sgd_kernel_f16_clamped()
    e = B.sgd_epilogue_args(kind=B.EPI_F16, out=out.data_ptr(), ldo=N)
    B.sgd_kernel_gemm(A, W, M, N, K, e)
    torch.cuda.synchronize()
    assert torch.all(out == 65504.0)
    assert B.sgd_kernel_f16_clamped() == 1
    assert B.sgd_kernel_f16_clamped() == 0
    A.fill_(0.5)
    W.fill_(0.25)
    B.sgd_kernel_gemm(A, W, M, N, K, e)
    torch.cuda.synchronize()
    assert torch.all(out == 8.0)
    assert B.sgd_kernel_f16_clamped() == 0
    assert B.sgd_kernel_status() == 0


def test_check_device_reports_clamped_activations(B):
    """A model whose projections overflow fp16 (tiny with W_QKV scaled by 2^17) still runs,
    and sgd_check_device reports SGD_ERR_RANGE instead of returning silently clamped
    results; the unscaled model reports nothing."""
    cfg = synth.get_config("tiny")
    w = {k: v.cuda() for k, v in synth.make_weights(cfg, "cpu").items()}
    inp = synth.make_inputs(cfg, "cpu")
    out = torch.empty(cfg.batch, cfg.n_out_tokens, cfg.out_channels, device="cuda")
    S = [cfg.T] * cfg.n_units
    for scale, want in ((1.0, None), (2.0 ** 17, B.SGD_ERR_RANGE)):
        ws = dict(w)
        ws["blocks.0.w_qkv"] = (w["blocks.0.w_qkv"].float() * scale).to(torch.bfloat16)
        B.sgd_kernel_f16_clamped()
        m = B.Denoiser(cfg, ws)
        m.set_schedule(cfg.T, S, synth.block_groups(cfg))
        m.step(inp.z0.cuda(), out, 1000.0, 1)
        if want is None:
            m.check_device()
        else:
            with pytest.raises(B.SgdError) as err:
                m.check_device()
            assert err.value.code == want
            m.check_device()  # reported once
        m.close()


# ---------------------------------------------------------------------------
# pre-norm folded into the GEMM (the north-star's fused norm + projection)
# ---------------------------------------------------------------------------

FOLD_VARIANTS = [0, 3, 5, 6, 7, 9]
FOLD_IDS = ["tcgen05", "tcgen05_bk32", "tcgen05_epi4", "tcgen05_epi8", "tcgen05_bn128",
            "tcgen05_streamk"]


def _row_stats(x, slots):
    """Partial row sums of x^2 and x over `slots` column blocks (test input: any partition
    is valid), in the kernel layout [2 * 64, M]."""
    M, K = x.shape
    st = np.zeros((128, M), np.float32)
    edges = np.linspace(0, K, slots + 1).astype(int)
    for p in range(slots):
        blk = x[:, edges[p]:edges[p + 1]].astype(np.float64)
        st[p] = np.sum(blk * blk, axis=1)
        st[64 + p] = np.sum(blk, axis=1)
    return st


@pytest.mark.parametrize("variant", FOLD_VARIANTS, ids=FOLD_IDS)
@pytest.mark.parametrize("norm", ["rms", "ln"])
@pytest.mark.parametrize("epi", ["f16", "rope", "gated", "gelu", "f32"])
def test_gemm_folded_norm(B, norm, epi, variant):
    """norm(x) W^T with the norm's gain folded into B and rstd (and the LayerNorm mean /
    shift) applied in the epilogue, against the oracle's norm followed by its linear map
    and epilogue function, on ragged shapes."""
    rng = np.random.default_rng(31 + variant)
    H, dh, n_tok, bsz = 3, 64, 70, 3
    K = H * dh
    M = bsz * n_tok
    N = {"rope": 3 * K, "gated": 328, "gelu": 520, "f16": 264, "f32": 264}[epi]
    b_rows = 2 * N if epi == "gated" else N
    x = (rng.standard_normal((M, K)) * 2.0 + rng.standard_normal((M, 1)) * 0.7).astype(np.float32)
    g = torch.from_numpy(1.0 + 0.1 * rng.standard_normal(K).astype(np.float32)).to(torch.bfloat16)
    bsh = torch.from_numpy(0.1 * rng.standard_normal(K).astype(np.float32)).to(torch.bfloat16)
    W = _rand(rng, (b_rows, K), 1 / math.sqrt(K), torch.bfloat16)
    Wg = (W.float() * g.float()).half()                      # gain folded, one fp16 rounding
    colsum = np.zeros(b_rows + 512, np.float32)
    colsum[:b_rows] = Wg.double().sum(dim=1).numpy()
    colbias = np.zeros(b_rows + 512, np.float32)
    colbias[:b_rows] = (W.double() @ bsh.double()).numpy()
    slots = 3
    st = torch.from_numpy(_row_stats(x, slots)).cuda()
    A = torch.from_numpy(x).half().cuda()
    out = torch.empty(M, N, dtype=torch.float32 if epi == "f32" else torch.float16, device="cuda")
    kind = {"f16": B.EPI_F16, "rope": B.EPI_ROPE, "gated": B.EPI_GATED, "gelu": B.EPI_GELU,
            "f32": B.EPI_F32}[epi]
    cs, cb = torch.from_numpy(colsum).cuda(), torch.from_numpy(colbias).cuda()
    e = B.sgd_epilogue_args(kind=kind, out=out.data_ptr(), ldo=N, norm=1 if norm == "rms" else 2,
                            rstat=st.data_ptr(), stat_slots=slots, stat_ld=M, norm_eps=1e-6,
                            colsum=cs.data_ptr(), colbias=cb.data_ptr(), act=1 if epi == "gelu" else 0)
    if epi == "rope":
        half = dh // 2
        pos = np.arange(n_tok, dtype=np.float64)[:, None]
        freq = 10000.0 ** (-np.arange(half) * 2.0 / dh)
        cos = torch.from_numpy(np.cos(pos * freq).astype(np.float32)).cuda()
        sin = torch.from_numpy(np.sin(pos * freq).astype(np.float32)).cuda()
        e.rope_cos, e.rope_sin = cos.data_ptr(), sin.data_ptr()
        e.rope_tokens, e.d_head, e.rope_cols = n_tok, dh, 2 * K
    if norm == "ln" and epi == "rope":  # not a model combination (RoPE models use RMSNorm)
        with pytest.raises(B.SgdError) as err:
            B.sgd_kernel_gemm(A, Wg.cuda(), M, N, K, e, use_simt=variant)
        assert err.value.code == B.SGD_ERR_SHAPE
        return
    B.sgd_kernel_gemm(A, Wg.cuda(), M, N, K, e, use_simt=variant)
    torch.cuda.synchronize()
    assert B.sgd_kernel_status() == 0

    def finish(u):
        if epi == "gated":
            return odn.silu(u[:, :N]) * u[:, N:]
        if epi == "gelu":
            return odn.gelu_erf(u)
        if epi == "rope":
            qkv = u.reshape(bsz, n_tok, 3, H, dh)
            r = qkv.copy()
            for j in range(2):
                t = qkv[:, :, j].transpose(0, 2, 1, 3)
                r[:, :, j] = odn.rope(t, np.arange(n_tok), 10000.0).transpose(0, 2, 1, 3)
            return r.reshape(M, N)
        return u

    # (1) the oracle: norm, then the linear map and the epilogue function, unrounded operands
    if norm == "rms":
        xn = odn.rms_norm(x, g.float().numpy(), 1e-6)
    else:
        xn = odn.layer_norm(x, g.float().numpy(), bsh.float().numpy(), 1e-6)
    want = finish(odn.linear(xn, W.float().numpy()))
    got = _f(out).astype(np.float64)
    err = np.linalg.norm(got - want) / np.linalg.norm(want)
    assert err < 2e-3, err  # fp16 rounding of x and of W g (2^-11 each) and of the output
    # (2) element-wise: the same algebra on the operands the kernel multiplies (fp16 x, fp16
    # W g), so that only accumulation order and the output rounding remain
    xr = A.double().cpu().numpy()
    acc = xr @ Wg.double().numpy().T
    ss, s1 = np.sum(x.astype(np.float64) ** 2, axis=1), np.sum(x.astype(np.float64), axis=1)
    if norm == "rms":
        u = acc / np.sqrt(ss / K + 1e-6)[:, None]
    else:
        mean = s1 / K
        rstd = 1.0 / np.sqrt(ss / K - mean ** 2 + 1e-6)
        u = rstd[:, None] * (acc - mean[:, None] * colsum[None, :b_rows]) + colbias[None, :b_rows]
    tight = finish(u.astype(np.float32))
    _check_f16(out, tight, extra_abs=2e-4 * float(np.sqrt(np.mean(tight.astype(np.float64) ** 2))))


@pytest.mark.parametrize("finalise", [False, True], ids=["slots", "finalised"])
@pytest.mark.parametrize("variant", [0, 5, 7, 9, 10], ids=["tcgen05", "epi4", "bn128", "streamk", "bn224"])
@pytest.mark.parametrize("kind", ["delta", "f32"])
def test_gemm_residual_writer_emits_h16_and_row_sums(B, kind, variant, finalise):
    """A writer of the residual stream also stores fp16(h_new) (bit-exact against torch's
    rounding of the same fp32 values) and, per row, partial sums of h_new^2 and h_new whose
    slot sums equal the full row sums.  Finalised: the CTA completing each 128-row block
    stores the slot-order fp32 sum of its slots (bit-exact against that sum on the host) in
    slot 0 of the final buffer and leaves the tickets at zero."""
    rng = np.random.default_rng(41 + variant)
    M, N, K = 300, 1032 if variant != 10 else 4096, 512
    if variant == 9:
        M, N, K = 4096, 4096, 4096
    A = _rand(rng, (M, K)).cuda()
    W = _rand(rng, (N, K), 1 / math.sqrt(K)).cuda()
    h = torch.from_numpy(rng.standard_normal((M, N)).astype(np.float32)).cuda()
    h16 = torch.empty(M, N, dtype=torch.float16, device="cuda")
    st = torch.full((128, M), float("nan"), device="cuda")
    fin = torch.full((128, M), float("nan"), device="cuda")
    cnt = torch.zeros((M + 127) // 128, dtype=torch.int32, device="cuda")
    if kind == "delta":
        e = B.sgd_epilogue_args(kind=B.EPI_DELTA, h=h.data_ptr(), ldh=N, h16=h16.data_ptr(),
                                stat_out=st.data_ptr(), stat_out_ld=M)
    else:
        e = B.sgd_epilogue_args(kind=B.EPI_F32, out=h.data_ptr(), ldo=N, h16=h16.data_ptr(),
                                stat_out=st.data_ptr(), stat_out_ld=M)
    if finalise:
        e.stat_cnt, e.stat_final = cnt.data_ptr(), fin.data_ptr()
    slots = B.sgd_kernel_gemm_stat_slots(M, N, K, e, variant)
    assert 2 <= slots <= 64 and slots % 2 == 0
    h0 = h.clone()
    B.sgd_kernel_gemm(A, W, M, N, K, e, use_simt=variant)
    torch.cuda.synchronize()
    assert B.sgd_kernel_status() == 0
    rows = np.sort(rng.choice(M, 48, replace=False))
    u = odn.linear(_f(A[rows]), _f(W))
    want = (_f(h0[rows]) if kind == "delta" else 0.0) + u
    np.testing.assert_allclose(_f(h[rows]), want, rtol=2e-5, atol=2e-5)
    assert torch.equal(h16, h.half())
    hv = h.double()
    ss = st[:slots].double().sum(dim=0)
    s1 = st[64:64 + slots].double().sum(dim=0)
    torch.testing.assert_close(ss, (hv * hv).sum(dim=1), rtol=2e-5, atol=1e-3)
    torch.testing.assert_close(s1, hv.sum(dim=1), rtol=2e-5, atol=1e-2)
    if finalise:
        slots_h = st[:slots].cpu().numpy()
        sums_h = st[64:64 + slots].cpu().numpy()
        want_ss = np.zeros(M, np.float32)
        want_s1 = np.zeros(M, np.float32)
        for p in range(slots):  # slot order, fp32
            want_ss = (want_ss + slots_h[p]).astype(np.float32)
            want_s1 = (want_s1 + sums_h[p]).astype(np.float32)
        np.testing.assert_array_equal(fin[0].cpu().numpy(), want_ss)
        np.testing.assert_array_equal(fin[64].cpu().numpy(), want_s1)
        assert int(cnt.abs().sum()) == 0


def _padded_heads(x, H, dh, hs, rng=None):
    """[rows, H dh] -> [rows, H hs]: head h at columns [h hs, h hs + dh); the gap columns
    hold zeros (rng None) or random finite values."""
    rows = x.shape[0]
    out = np.zeros((rows, H * hs), np.float32) if rng is None else \
        rng.standard_normal((rows, H * hs)).astype(np.float32) * 3.0
    for h in range(H):
        out[:, h * hs:h * hs + dh] = x[:, h * dh:(h + 1) * dh]
    return out


@pytest.mark.parametrize("impl", [0, 3, 1], ids=["tcgen05", "tcgen05_2tile", "mma_sync"])
@pytest.mark.parametrize("H,nq,nkv,bsz", [(16, 256, 256, 2), (3, 136, 136, 2), (2, 300, 77, 3),
                                          (4, 640, 640, 1)])
def test_attention_dh72_head_padded(B, H, nq, nkv, bsz, impl):
    """d_h = 72 (DiT-XL/2) from a head-padded layout (80 columns per head): the tcgen05
    kernel reads each head as a 64- and a 16-column block, with zeros after every Q head and
    arbitrary finite values after K and V heads, against the oracle's attention; O is
    written with 72 columns per head."""
    rng = np.random.default_rng(H + nq + nkv)
    dh, hs = 72, 80
    d = H * dh
    q = (rng.standard_normal((bsz * nq, d)) * 1.5).astype(np.float32)
    k = (rng.standard_normal((bsz * nkv, d)) * 1.5).astype(np.float32)
    v = rng.standard_normal((bsz * nkv, d)).astype(np.float32)
    q, k, v = (torch.from_numpy(t).half().float().numpy() for t in (q, k, v))
    qp = torch.from_numpy(_padded_heads(q, H, dh, hs)).half().cuda()
    kp = torch.from_numpy(_padded_heads(k, H, dh, hs, rng)).half().cuda()
    vp = torch.from_numpy(_padded_heads(v, H, dh, hs, rng)).half().cuda()
    o = torch.full((bsz * nq, d), float("nan"), dtype=torch.float16, device="cuda")
    B.sgd_kernel_attention_hs(qp, H * hs, kp, vp, H * hs, hs, o, d, bsz, nq, nkv, H, dh, impl=impl)
    torch.cuda.synchronize()
    want = odn.attention(q.reshape(bsz, nq, d), k.reshape(bsz, nkv, d), v.reshape(bsz, nkv, d),
                         H).reshape(bsz * nq, d)
    got = _f(o)
    err = np.linalg.norm(got - want) / np.linalg.norm(want)
    assert err < 1.5e-3, err
    assert np.max(np.abs(got - want)) < 5e-3 * float(np.abs(want).max())
    assert B.sgd_kernel_status() == 0
