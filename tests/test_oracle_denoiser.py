"""Pins for the oracle's scheduled forward (Sec. 3.1, Algorithm 2) and block math.

The paper fixes the residual-unit semantics; the block architectures are
textbook definitions, pinned here by textbook special cases and by independent
restatements (complex-number RoPE, x * Phi(x) GELU, brute-force loops).
"""
import itertools
import math

import numpy as np
import pytest
import torch
from scipy.special import expit, softmax as sp_softmax
from scipy.stats import norm as sp_norm

from oracle import denoiser as dn
from oracle import spectral as sp
from oracle import trajectory as tj
from paper_2609_29505_gb300 import synth

F32 = np.float32


def _weights(cfg):
    return dn.to_numpy_weights(synth.make_weights(cfg, "cpu"))


def _inputs(cfg):
    inp = synth.make_inputs(cfg, "cpu")
    z0 = None if inp.z0 is None else inp.z0.numpy()
    cls = None if inp.class_ids is None else inp.class_ids.numpy()
    ctx = None if inp.ctx is None else inp.ctx.float().numpy()
    ids_at = None
    if cfg.stem == "embed":
        ids_at = lambda s: synth.token_ids_at(cfg, inp, s).numpy()
    return z0, cls, ctx, ids_at


def _micro(block="prenorm", **kw):
    base = dict(name="micro", stem="time_add", block=block, norm="rms", mlp="swiglu",
                head="linear", n_blocks=2, d=32, n_heads=2, d_head=16, d_ff=48, batch=1,
                n_tokens=5, d_in=32, d_out=32, out_channels=32, T=4, seed=99, horizons=[4])
    if block == "adaln":
        base.update(stem="patch", norm="ln_plain", mlp="gelu_tanh", head="adaln_linear",
                    d_in=8, d_out=16, out_channels=8, n_classes=5, t_freq=16)
    if block == "xattn":
        base.update(stem="identity", norm="ln", mlp="geglu", head="identity",
                    ctx_len=3, d_ctx=24)
    base.update(kw)
    return synth.ModelConfig(**base)


# ---------------------------------------------------------------------------
# elementwise and layer pins
# ---------------------------------------------------------------------------

def test_linear_brute_force():
    rng = np.random.default_rng(0)
    x = rng.standard_normal((3, 4)).astype(F32)
    W = rng.standard_normal((5, 4)).astype(F32)
    y = dn.linear(x, W)
    for i in range(3):
        for o in range(5):
            acc = sum(float(x[i, k]) * float(W[o, k]) for k in range(4))
            assert y[i, o] == pytest.approx(acc, rel=1e-5, abs=1e-6)


def test_activation_pins():
    x = np.linspace(-6, 6, 1001).astype(F32)
    np.testing.assert_allclose(dn.gelu_erf(x), x * sp_norm.cdf(x), rtol=2e-6, atol=1e-6)
    np.testing.assert_allclose(dn.silu(x), x * expit(x), rtol=2e-6, atol=1e-6)
    assert np.max(np.abs(dn.gelu_tanh(x) - dn.gelu_erf(x))) < 1e-3
    assert dn.gelu_tanh(np.array([0.0], F32))[0] == 0.0
    assert dn.silu(np.array([0.0], F32))[0] == 0.0


def test_norm_pins():
    rng = np.random.default_rng(1)
    x = (rng.standard_normal((7, 96)) * 3 + 1.5).astype(F32)
    y = dn.rms_norm(x, np.ones(96, F32), 1e-6)
    np.testing.assert_allclose(np.mean(y.astype(np.float64) ** 2, axis=-1), 1.0, rtol=1e-5)
    y = dn.layer_norm(x, None, None, 1e-6)
    np.testing.assert_allclose(np.mean(y, axis=-1), 0.0, atol=1e-5)
    np.testing.assert_allclose(np.var(y.astype(np.float64), axis=-1), 1.0, rtol=1e-5)
    g = rng.standard_normal(96).astype(F32)
    b = rng.standard_normal(96).astype(F32)
    np.testing.assert_allclose(dn.layer_norm(x, g, b, 1e-6), y * g + b, rtol=1e-6, atol=1e-6)
    # RMSNorm is scale invariant, LayerNorm is shift invariant
    np.testing.assert_allclose(dn.rms_norm(5 * x, g, 1e-12), dn.rms_norm(x, g, 1e-12), rtol=2e-6,
                               atol=2e-6)
    np.testing.assert_allclose(dn.layer_norm(x + 4, g, b, 1e-12), dn.layer_norm(x, g, b, 1e-12),
                               rtol=2e-5, atol=2e-5)


def test_sinusoid_pins():
    e = dn.sinusoid(0.0, 16)
    np.testing.assert_array_equal(e, np.concatenate([np.ones(8), np.zeros(8)]).astype(F32))
    t = 37.5
    e = dn.sinusoid(t, 16)
    assert e[0] == pytest.approx(math.cos(t), abs=1e-6)
    assert e[8] == pytest.approx(math.sin(t), abs=1e-6)
    w7 = 10000.0 ** (-7 / 8)
    assert e[7] == pytest.approx(math.cos(t * w7), abs=1e-6)
    assert e[15] == pytest.approx(math.sin(t * w7), abs=1e-6)


def test_rope_pins():
    rng = np.random.default_rng(2)
    dh = 16
    x = rng.standard_normal((6, dh)).astype(F32)
    pos = np.arange(6)
    y = dn.rope(x, pos, 10000.0)
    np.testing.assert_array_equal(y[0], x[0])               # position 0 is the identity
    np.testing.assert_allclose(np.linalg.norm(y, axis=-1), np.linalg.norm(x, axis=-1), rtol=1e-5)
    # complex-number restatement: pairs (x_i, x_{i+half}) rotate by pos * theta^(-2i/dh)
    half = dh // 2
    zc = x[:, :half].astype(np.complex128) + 1j * x[:, half:]
    ang = pos[:, None] * 10000.0 ** (-2.0 * np.arange(half) / dh)[None, :]
    zr = zc * np.exp(1j * ang)
    np.testing.assert_allclose(y[:, :half], zr.real, rtol=1e-5, atol=1e-5)
    np.testing.assert_allclose(y[:, half:], zr.imag, rtol=1e-5, atol=1e-5)
    # relative-position property of the scores
    q, k = x[1], x[2]
    a = dn.rope(np.stack([q, k]), np.array([4, 1]), 10000.0)
    b = dn.rope(np.stack([q, k]), np.array([9, 6]), 10000.0)
    assert float(a[0] @ a[1]) == pytest.approx(float(b[0] @ b[1]), rel=1e-4, abs=1e-4)


def test_attention_pins():
    rng = np.random.default_rng(3)
    B, Nq, Nk, H, dh = 2, 5, 7, 3, 8
    d = H * dh
    q = rng.standard_normal((B, Nq, d)).astype(F32)
    v = rng.standard_normal((B, Nk, d)).astype(F32)
    # identical keys -> uniform weights -> mean of V
    k = np.repeat(rng.standard_normal((B, 1, d)).astype(F32), Nk, axis=1)
    o = dn.attention(q, k, v, H)
    np.testing.assert_allclose(o, np.broadcast_to(v.mean(axis=1, keepdims=True), o.shape),
                               rtol=1e-5, atol=1e-5)
    # one key -> V itself
    o = dn.attention(q, k[:, :1], v[:, :1], H)
    np.testing.assert_allclose(o, np.broadcast_to(v[:, :1], o.shape), rtol=1e-6, atol=1e-6)
    # general case against a float64 restatement with the library softmax, head by head
    k = rng.standard_normal((B, Nk, d)).astype(F32)
    o = dn.attention(q, k, v, H)
    for b in range(B):
        for h in range(H):
            sl = slice(h * dh, (h + 1) * dh)
            p = sp_softmax(q[b, :, sl].astype(np.float64) @ k[b, :, sl].T / math.sqrt(dh), axis=1)
            np.testing.assert_allclose(o[b, :, sl], p @ v[b, :, sl], rtol=1e-4, atol=1e-5)
    p = dn.softmax_rows(rng.standard_normal((4, 9)).astype(F32) * 20)
    np.testing.assert_allclose(p.sum(axis=1), 1.0, rtol=1e-6)


# ---------------------------------------------------------------------------
# model-level special cases
# ---------------------------------------------------------------------------

def _zero_branch_outputs(cfg, W):
    W = dict(W)
    for b in range(cfg.n_blocks):
        for name in ("w_o", "w_2", "wx_o"):
            key = f"blocks.{b}.{name}"
            if key in W:
                W[key] = np.zeros_like(W[key])
    return W


@pytest.mark.parametrize("name", ["tiny", "dit_small", "sdxl_small", "llada_small"])
def test_zero_branches_give_head_of_stem(name):
    cfg = synth.get_config(name)
    W = _zero_branch_outputs(cfg, _weights(cfg))
    z0, cls, ctx, ids_at = _inputs(cfg)
    x = ids_at(3) if ids_at else z0
    t = 421.0
    got = dn.denoise_full(cfg, W, x, t, cls, ctx)
    want = dn.head(cfg, W, dn.stem(cfg, W, x, t, cls), dn.conditioning(cfg, W, t, cls))
    np.testing.assert_array_equal(got, want)


def test_uvit_skips_composition_by_hand():
    """With zero branch outputs only the long skips act: in-blocks push h0 unchanged,
    the mid block passes it, out-block j applies W_skip_j [h; h0]."""
    cfg = synth.get_config("uvit_small")
    W = _zero_branch_outputs(cfg, _weights(cfg))
    z0, cls, _, _ = _inputs(cfg)
    t = 250.0
    h0 = dn.stem(cfg, W, z0, t, cls)
    h = h0
    for j in range(cfg.n_skips):
        h = (np.concatenate([h, h0], axis=-1) @ W[f"skips.{j}.w"].T).astype(F32)
    want = dn.head(cfg, W, h, None)
    np.testing.assert_allclose(dn.denoise_full(cfg, W, z0, t, cls), want, rtol=1e-6, atol=1e-6)


def test_dit_zero_gates_make_every_delta_zero():
    cfg = synth.get_config("dit_small")
    W = _weights(cfg)
    d = cfg.d
    for b in range(cfg.n_blocks):
        wm = W[f"blocks.{b}.w_mod"].copy()
        wm[2 * d:3 * d] = 0.0
        wm[5 * d:6 * d] = 0.0
        W[f"blocks.{b}.w_mod"] = wm
    z0, cls, _, _ = _inputs(cfg)
    t = 600.0
    c = dn.conditioning(cfg, W, t, cls)
    want = dn.head(cfg, W, dn.stem(cfg, W, z0, t, cls), c)
    np.testing.assert_array_equal(dn.denoise_full(cfg, W, z0, t, cls), want)


def test_xattn_single_context_token_is_projected_value():
    """softmax over one key is 1: Delta_xattn = (ctx W_V^T) W_O^T for every query."""
    cfg = _micro("xattn", ctx_len=1)
    W = _weights(cfg)
    rng = np.random.default_rng(4)
    h = rng.standard_normal((1, cfg.n_tokens, cfg.d)).astype(F32)
    ctx = rng.standard_normal((1, 1, cfg.d_ctx)).astype(F32)
    delta = dn.branch(cfg, W, 0, "xattn", h, None, ctx)
    v = ctx[0, 0] @ W["blocks.0.wx_kv"][cfg.d:].T
    np.testing.assert_allclose(delta[0], np.broadcast_to(v @ W["blocks.0.wx_o"].T, delta[0].shape),
                               rtol=1e-5, atol=1e-5)


def test_embed_stem_and_logits_head():
    cfg = synth.get_config("llada_small")
    W = _weights(cfg)
    ids = np.array([[0, 5, 999, 5]])
    h = dn.stem(cfg, W, ids, 0.0, None)
    np.testing.assert_array_equal(h[0], W["embed"][[0, 5, 999, 5]])
    logits = dn.head(cfg, W, h, None)
    x = dn.rms_norm(h, W["normf_w"], cfg.eps)
    np.testing.assert_allclose(logits, x @ W["w_head"].T, rtol=1e-5, atol=1e-5)


# ---------------------------------------------------------------------------
# executor semantics (Sec. 3.1, Algorithm 2)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("name", ["tiny", "dit_small", "uvit_small", "sdxl_small", "llada_small"])
def test_full_budget_equals_unscheduled_forward_exactly(name):
    cfg = synth.get_config(name)
    W = _weights(cfg)
    z0, cls, ctx, ids_at = _inputs(cfg)
    T = 3
    S = [T] * cfg.n_units
    cache = {}
    z = z0
    for s in range(1, T + 1):
        x = ids_at(s) if ids_at else z
        t = tj.timestep(T, s)
        a = dn.denoise(cfg, W, x, t, s, S, cache, cls, ctx)
        b = dn.denoise_full(cfg, W, x, t, cls, ctx)
        np.testing.assert_array_equal(a, b)
        if not ids_at:
            z = (x - a / F32(T)).astype(F32)


@pytest.mark.parametrize("name", ["tiny", "dit_small", "uvit_small", "sdxl_small"])
def test_frozen_unit_output_is_input_plus_cache(name):
    cfg = synth.get_config(name)
    W = _weights(cfg)
    z0, cls, ctx, _ = _inputs(cfg)
    T = 4
    S = [(u % T) + 1 for u in range(cfg.n_units)]
    cache = {}
    for s in range(1, T + 1):
        tr = dn.Trace()
        dn.denoise(cfg, W, z0, tj.timestep(T, s), s, S, cache, cls, ctx, trace=tr)
        for u, active, h_in, h_out in tr.units:
            assert active == (s <= S[u])
            if not active:
                np.testing.assert_array_equal(h_out, (h_in + cache[u]).astype(F32))


def _definition_trajectory(cfg, W, S, T, z0, cls, ctx):
    """Sec. 3.1 written as a recursion, without a cache: h(-1, s) is the stem of step s,
    h(u, s) = h(u-1, s) + F_u(h(u-1, s)) for s <= S_u and h(u-1, s) + F_u(h(u-1, S_u))
    afterwards.  Conditioning c_r of the refresh step enters F_u.  States integrate
    z_{s+1} = z_s - eps_s / T."""
    zs = [np.asarray(z0, F32)]
    units = [(b, kind) for b in range(cfg.n_blocks) for kind in cfg.branches]
    outs = []

    def h(u, s):
        t = tj.timestep(T, s)
        if u < 0:
            return dn.stem(cfg, W, zs[s - 1], t, cls)
        b, kind = units[u]
        r = s if s <= S[u] else S[u]
        prev = h(u - 1, s)
        c_r = dn.conditioning(cfg, W, tj.timestep(T, r), cls)
        upd = dn.branch(cfg, W, b, kind, h(u - 1, r) if r != s else prev, c_r, ctx)
        return (prev + upd).astype(F32)

    for s in range(1, T + 1):
        eps = dn.head(cfg, W, h(len(units) - 1, s), dn.conditioning(cfg, W, tj.timestep(T, s), cls))
        outs.append(eps)
        zs.append((zs[-1] - eps / F32(T)).astype(F32))
    return zs, outs


@pytest.mark.parametrize("block", ["prenorm", "adaln", "xattn"])
def test_brute_force_all_block_schedules_two_layers(block):
    """Every block-lifetime vector in {1..T}^2 (T = 4): the cached executor equals the
    cache-free recursion of Sec. 3.1 bit for bit."""
    cfg = _micro(block)
    W = _weights(cfg)
    z0, cls, ctx, _ = _inputs(cfg)
    T = cfg.T
    nb = len(cfg.branches)
    for Sb in itertools.product(range(1, T + 1), repeat=cfg.n_blocks):
        S = [Sb[u // nb] for u in range(cfg.n_units)]
        got = tj.run(cfg, W, S, T, z0=z0, class_ids=cls, ctx=ctx)
        zs, outs = _definition_trajectory(cfg, W, S, T, z0, cls, ctx)
        for a, b in zip(got["outputs"], outs):
            np.testing.assert_array_equal(a, b)
        np.testing.assert_array_equal(got["states"][-1], zs[-1])


def test_brute_force_all_branch_schedules_two_layers():
    """Branch granularity: every per-branch lifetime vector in {1..T}^4 (T = 4)."""
    cfg = _micro("prenorm")
    W = _weights(cfg)
    z0, cls, ctx, _ = _inputs(cfg)
    T = cfg.T
    for S in itertools.product(range(1, T + 1), repeat=cfg.n_units):
        got = tj.run(cfg, W, list(S), T, z0=z0)
        zs, outs = _definition_trajectory(cfg, W, list(S), T, z0, cls, ctx)
        np.testing.assert_array_equal(got["states"][-1], zs[-1])
        np.testing.assert_array_equal(got["outputs"][-1], outs[-1])


def test_uvit_brute_force_skip_model():
    """U-ViT structure (3 blocks, one long skip): the cached executor against a cache-free
    recursion that re-runs every frozen branch on its input at step S_u, with the skip
    combine and push applied on current values at every step."""
    cfg = synth.get_config("uvit_small").with_(n_blocks=3, n_skips=1, d=32, n_heads=2,
                                                d_head=16, d_ff=64, batch=1, n_tokens=6,
                                                T=3, n_classes=4)
    W = _weights(cfg)
    z0, cls, _, _ = _inputs(cfg)
    T = cfg.T
    units = [(b, kind) for b in range(cfg.n_blocks) for kind in cfg.branches]

    def forward(zs, s, S):
        t = tj.timestep(T, s)

        def run_to(s_eval):
            # evaluate the network at step s_eval, frozen branches replayed recursively
            h = dn.stem(cfg, W, zs[s_eval - 1], tj.timestep(T, s_eval), cls)
            skips, u = [], 0
            for b in range(cfg.n_blocks):
                if b > cfg.n_skips:
                    h = dn.skip_combine(W, b - cfg.n_skips - 1, h, skips.pop())
                for kind in cfg.branches:
                    if s_eval <= S[u]:
                        h = (h + dn.branch(cfg, W, b, kind, h)).astype(F32)
                    else:
                        h = (h + branch_input_delta(u, S[u])).astype(F32)
                    u += 1
                if b < cfg.n_skips:
                    skips.append(h)
            return h

        memo = {}

        def branch_input_delta(u, r):
            # Delta_{u, r}: re-run the network at step r up to unit u and apply F_u there
            if (u, r) in memo:
                return memo[(u, r)]
            h = dn.stem(cfg, W, zs[r - 1], tj.timestep(T, r), cls)
            skips, v = [], 0
            for b in range(cfg.n_blocks):
                if b > cfg.n_skips:
                    h = dn.skip_combine(W, b - cfg.n_skips - 1, h, skips.pop())
                for kind in cfg.branches:
                    dlt = dn.branch(cfg, W, b, kind, h) if r <= S[v] else branch_input_delta(v, S[v])
                    if v == u:
                        memo[(u, r)] = dlt
                        return dlt
                    h = (h + dlt).astype(F32)
                    v += 1
                if b < cfg.n_skips:
                    skips.append(h)
            raise AssertionError

        return dn.head(cfg, W, run_to(s), None)

    for S in [(3, 3, 1, 1, 2, 2), (1, 1, 3, 3, 2, 2), (2, 2, 2, 2, 1, 1), (1, 1, 1, 1, 1, 1)]:
        got = tj.run(cfg, W, list(S), T, z0=z0, class_ids=cls)
        zs = [z0]
        for s in range(1, T + 1):
            eps = forward(zs, s, S)
            np.testing.assert_array_equal(got["outputs"][s - 1], eps)
            zs.append((zs[-1] - eps / F32(T)).astype(F32))


def test_scheduled_active_sets_keep_groups_atomic():
    cfg = synth.get_config("dit_small")
    W = _weights(cfg)
    groups = synth.block_groups(cfg)
    res = sp.schedule(cfg, W, T=8, budget=0.5, group_of_unit=groups)
    A = sp.active_sets(res["lifetimes"], 8)
    nb = len(cfg.branches)
    for b in range(cfg.n_blocks):
        assert np.all(A[:, b * nb:(b + 1) * nb] == A[:, b * nb:b * nb + 1])
    assert res["ratio"] <= 0.5


# ---------------------------------------------------------------------------
# AdaLN conditioning pins (DiT family): hand-computed cases whose weights are scaled
# identities / selections, so that each quantity has a closed form and a dropped "1 +",
# a SiLU at the wrong stage, a class embedding added before W_t2 or a permuted chunk
# order each change the result.
# ---------------------------------------------------------------------------

def _silu(v):
    return v / (1.0 + math.exp(-v))


def test_modulate_hand_case():
    """x (1 + scale_b) + shift_b, the sample's shift and scale broadcast over its tokens."""
    x = np.array([[[1.0, -2.0], [0.5, 4.0]], [[3.0, 1.0], [-1.0, 0.0]]], F32)   # [B=2, N=2, d=2]
    shift = np.array([[10.0, 20.0], [-5.0, 7.0]], F32)
    scale = np.array([[0.5, -1.0], [2.0, 0.25]], F32)
    got = dn.modulate(x, shift, scale)
    for b in range(2):
        for n in range(2):
            for j in range(2):
                want = float(x[b, n, j]) * (1.0 + float(scale[b, j])) + float(shift[b, j])
                assert got[b, n, j] == pytest.approx(want, rel=1e-6, abs=1e-6)


def _dit_micro_weights(cfg, rng):
    """W_t1 = 3 x (selection of the first t_freq of d rows), W_t2 = 2 I, one-hot-ish class
    rows, W_mod chunks = (j + 1) I, W_modf = [I; 2 I] (the rest random)."""
    W = _weights(cfg)
    d, tf = cfg.d, cfg.t_freq
    W["w_t1"] = np.zeros((d, tf), F32)
    for i in range(min(d, tf)):
        W["w_t1"][i, i] = 3.0
    W["w_t2"] = 2.0 * np.eye(d, dtype=F32)
    W["class_emb"] = np.zeros((cfg.n_classes, d), F32)
    for y in range(cfg.n_classes):
        W["class_emb"][y, y % d] = 5.0 + y
    for b in range(cfg.n_blocks):
        W[f"blocks.{b}.w_mod"] = np.concatenate([(j + 1.0) * np.eye(d, dtype=F32) for j in range(6)])
    W["w_modf"] = np.concatenate([np.eye(d, dtype=F32), 2.0 * np.eye(d, dtype=F32)])
    return W


def _hand_conditioning(cfg, t, y):
    """c = W_t2 silu(W_t1 sinusoid(t)) + class_emb[y] for the weights above, by hand."""
    d, tf = cfg.d, cfg.t_freq
    half = tf // 2
    emb = [math.cos(t * 10000.0 ** (-i / half)) for i in range(half)]
    emb += [math.sin(t * 10000.0 ** (-i / half)) for i in range(half)]
    c = []
    for i in range(d):
        hidden = _silu(3.0 * emb[i]) if i < tf else _silu(0.0)
        c.append(2.0 * hidden + (5.0 + y if i == y % d else 0.0))
    return np.array(c)


def test_conditioning_hand_case():
    cfg = _micro("adaln")
    W = _dit_micro_weights(cfg, np.random.default_rng(5))
    for t, y in ((0.0, 0), (137.25, 3), (999.0, 4)):
        got = dn.conditioning(cfg, W, t, np.array([y]))
        np.testing.assert_allclose(got[0], _hand_conditioning(cfg, t, y), rtol=1e-5, atol=1e-5)


def test_block_modulation_chunk_order():
    """shift1, scale1, gate1, shift2, scale2, gate2 = chunks 0..5 of W_mod silu(c)."""
    cfg = _micro("adaln")
    W = _dit_micro_weights(cfg, np.random.default_rng(6))
    c = np.array([[0.3, -1.2] + [0.1 * i for i in range(cfg.d - 2)]], F32)
    mods = dn.block_modulation(W, 0, c)
    assert len(mods) == 6
    for j, m in enumerate(mods):
        want = [(j + 1.0) * _silu(float(v)) for v in c[0]]
        np.testing.assert_allclose(m[0], want, rtol=1e-5, atol=1e-6)


def test_adaln_branches_use_their_own_chunks():
    """attn: LN(h)(1 + scale1) + shift1 -> attention -> gate1 * (o W_O^T); mlp: LN(h)(1 +
    scale2) + shift2 -> GELU-tanh MLP -> gate2 * (.), with the chunks of the case above."""
    cfg = _micro("adaln")
    W = _dit_micro_weights(cfg, np.random.default_rng(7))
    rng = np.random.default_rng(8)
    h = rng.standard_normal((1, cfg.n_tokens, cfg.d)).astype(F32)
    c = rng.standard_normal((1, cfg.d)).astype(F32)
    sc = np.array([_silu(float(v)) for v in c[0]], np.float64)
    chunk = [(j + 1.0) * sc for j in range(6)]
    x = dn.layer_norm(h, None, None, cfg.eps).astype(np.float64)[0]
    d = cfg.d
    # attention branch
    xm = x * (1.0 + chunk[1]) + chunk[0]
    qkv = xm @ W["blocks.0.w_qkv"].T.astype(np.float64)
    o = dn.attention(qkv[None, :, :d].astype(F32), qkv[None, :, d:2 * d].astype(F32),
                     qkv[None, :, 2 * d:].astype(F32), cfg.n_heads)[0].astype(np.float64)
    want = chunk[2] * (o @ W["blocks.0.w_o"].T.astype(np.float64))
    np.testing.assert_allclose(dn.branch(cfg, W, 0, "attn", h, c)[0], want, rtol=2e-4, atol=2e-4)
    # MLP branch
    xm = x * (1.0 + chunk[4]) + chunk[3]
    u = xm @ W["blocks.0.w_1"].T.astype(np.float64)
    a = 0.5 * u * (1.0 + np.tanh(math.sqrt(2.0 / math.pi) * (u + 0.044715 * u ** 3)))
    want = chunk[5] * (a @ W["blocks.0.w_2"].T.astype(np.float64))
    np.testing.assert_allclose(dn.branch(cfg, W, 0, "mlp", h, c)[0], want, rtol=2e-4, atol=2e-4)


def test_adaln_linear_head_hand_case():
    """shift, scale = chunks of W_modf silu(c) (here silu(c) and 2 silu(c)); out =
    (LN(h)(1 + scale) + shift) W_head^T, first out_channels columns."""
    cfg = _micro("adaln")
    W = _dit_micro_weights(cfg, np.random.default_rng(9))
    rng = np.random.default_rng(10)
    h = rng.standard_normal((1, cfg.n_tokens, cfg.d)).astype(F32)
    c = rng.standard_normal((1, cfg.d)).astype(F32)
    got = dn.head(cfg, W, h, c)
    assert got.shape == (1, cfg.n_tokens, cfg.out_channels)
    sc = [_silu(float(v)) for v in c[0]]
    for n in range(cfg.n_tokens):
        row = [float(v) for v in h[0, n]]
        mu = sum(row) / cfg.d
        var = sum((v - mu) ** 2 for v in row) / cfg.d
        xn = [(v - mu) / math.sqrt(var + cfg.eps) for v in row]
        xm = [xn[i] * (1.0 + 2.0 * sc[i]) + sc[i] for i in range(cfg.d)]
        for o in range(cfg.out_channels):
            want = sum(xm[i] * float(W["w_head"][o, i]) for i in range(cfg.d))
            assert got[0, n, o] == pytest.approx(want, rel=1e-4, abs=1e-4)
