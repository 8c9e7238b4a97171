"""Scheduled denoiser forward, FP32 NumPy (oracle; test infrastructure only).

Residual-unit semantics (Sec. 3.1): a unit maps h_{l-1,s} to
h_{l,s} = h_{l-1,s} + F_l(h_{l-1,s}; c_s).  At steps s <= S_l the branch update
Delta_{l,s} = F_l(h_{l-1,s}; c_s) is computed and stored; at s > S_l the stored
Delta_{l, r_l(s)} is added to the *current* residual stream instead, with
r_l(s) = S_l (Algorithm 2 refreshes the cache on every active step, so the
last refresh happens at s = S_l).  Conditioning, skip features, stem and head
are evaluated at every step (Sec. 4.2).

Block architectures are not spelled out in the paper; they follow the textbook
definitions of the four families it evaluates (LLaDA: RMSNorm + RoPE + SwiGLU;
DiT: AdaLN-Zero + GELU-tanh; U-ViT: LayerNorm + long skips + GELU; SDXL
transformer: LayerNorm + self/cross attention + GEGLU):

* RMSNorm  x * rsqrt(mean(x^2) + eps) * g
* LayerNorm (x - mu) * rsqrt(var + eps) * g + b; AdaLN: LayerNorm without affine,
  then * (1 + scale_b) + shift_b
* attention softmax(q k^T / sqrt(d_h)) v per head, non-causal
* SwiGLU  W_2 (silu(W_gate x) * W_up x); GEGLU W_2 (a * gelu_erf(b)), [a; b] = W_1 x
* DiT gates: Delta_attn = gate1 * Attn(...), Delta_mlp = gate2 * MLP(...)

Arithmetic is float32 on the bf16-rounded weights the GPU also receives; the
only library primitives are matrix products and ``erf``.
"""
from __future__ import annotations

import math
from typing import Dict, List, Optional, Sequence

import numpy as np
from scipy.special import erf as _erf

F32 = np.float32


# ---------------------------------------------------------------------------
# elementwise functions
# ---------------------------------------------------------------------------

def silu(x):
    return (x / (F32(1.0) + np.exp(-x))).astype(F32)


def gelu_tanh(x):
    c = F32(math.sqrt(2.0 / math.pi))
    return (F32(0.5) * x * (F32(1.0) + np.tanh(c * (x + F32(0.044715) * x * x * x)))).astype(F32)


def gelu_erf(x):
    return (F32(0.5) * x * (F32(1.0) + _erf(x / F32(math.sqrt(2.0))).astype(F32))).astype(F32)


# ---------------------------------------------------------------------------
# layers
# ---------------------------------------------------------------------------

def linear(x, W):
    """y = x W^T for W stored [out, in]."""
    return (x @ W.T).astype(F32)


def rms_norm(x, g, eps):
    r = F32(1.0) / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + F32(eps))
    y = x * r
    return (y * g).astype(F32) if g is not None else y.astype(F32)


def layer_norm(x, g, b, eps):
    mu = np.mean(x, axis=-1, keepdims=True)
    xc = x - mu
    var = np.mean(xc * xc, axis=-1, keepdims=True)
    y = xc / np.sqrt(var + F32(eps))
    if g is not None:
        y = y * g
    if b is not None:
        y = y + b
    return y.astype(F32)


def sinusoid(t: float, dim: int) -> np.ndarray:
    """[cos(t w_i), sin(t w_i)], w_i = 10000^(-i/half), i = 0..half-1 (float64 -> fp32)."""
    half = dim // 2
    w = np.exp(-math.log(10000.0) * np.arange(half, dtype=np.float64) / half)
    a = t * w
    return np.concatenate([np.cos(a), np.sin(a)]).astype(F32)


def rope(x, positions, theta):
    """Rotate-half rotary embedding on the last axis of x [..., n, d_h]."""
    dh = x.shape[-1]
    half = dh // 2
    freq = theta ** (-np.arange(half, dtype=np.float64) * 2.0 / dh)
    ang = np.asarray(positions, dtype=np.float64)[:, None] * freq[None, :]
    cos = np.cos(ang).astype(F32)
    sin = np.sin(ang).astype(F32)
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * cos - x2 * sin, x2 * cos + x1 * sin], axis=-1).astype(F32)


def softmax_rows(s):
    s = s - np.max(s, axis=-1, keepdims=True)
    e = np.exp(s)
    return (e / np.sum(e, axis=-1, keepdims=True)).astype(F32)


def attention(q, k, v, n_heads, rope_theta=None):
    """Multi-head attention, non-causal.  q [B, Nq, d], k and v [B, Nk, d]."""
    B, Nq, d = q.shape
    Nk = k.shape[1]
    dh = d // n_heads
    qh = q.reshape(B, Nq, n_heads, dh).transpose(0, 2, 1, 3)
    kh = k.reshape(B, Nk, n_heads, dh).transpose(0, 2, 1, 3)
    vh = v.reshape(B, Nk, n_heads, dh).transpose(0, 2, 1, 3)
    if rope_theta is not None:
        qh = rope(qh, np.arange(Nq), rope_theta)
        kh = rope(kh, np.arange(Nk), rope_theta)
    s = (qh @ kh.transpose(0, 1, 3, 2)) / F32(math.sqrt(dh))
    p = softmax_rows(s.astype(F32))
    o = (p @ vh).astype(F32)
    return o.transpose(0, 2, 1, 3).reshape(B, Nq, d)


# ---------------------------------------------------------------------------
# model pieces
# ---------------------------------------------------------------------------

def _w(weights, name):
    return weights.get(name)


def norm(cfg, x, weights, name):
    if cfg.norm == "rms":
        return rms_norm(x, _w(weights, name + "_w"), cfg.eps)
    if cfg.norm == "ln":
        return layer_norm(x, _w(weights, name + "_w"), _w(weights, name + "_b"), cfg.eps)
    return layer_norm(x, None, None, cfg.eps)


def modulate(x, shift, scale):
    """AdaLN modulation: x * (1 + scale) + shift, per sample (shift/scale [B, d])."""
    return (x * (F32(1.0) + scale[:, None, :]) + shift[:, None, :]).astype(F32)


def conditioning(cfg, weights, t: float, class_ids) -> Optional[np.ndarray]:
    """DiT conditioning c = W_t2 silu(W_t1 sinusoid(t)) + class_emb[y]  ([B, d])."""
    if cfg.block != "adaln":
        return None
    temb = linear(silu(linear(sinusoid(t, cfg.t_freq)[None, :], weights["w_t1"])),
                  weights["w_t2"])
    return (temb + weights["class_emb"][np.asarray(class_ids)]).astype(F32)


def block_modulation(weights, b, c):
    """shift1, scale1, gate1, shift2, scale2, gate2 = chunk6(W_mod silu(c))."""
    mod = linear(silu(c), weights[f"blocks.{b}.w_mod"])
    return np.split(mod, 6, axis=-1)


def stem(cfg, weights, state, t: float, class_ids) -> np.ndarray:
    """Token states h_0 [B, N, d] (fp32)."""
    if cfg.stem == "time_add":
        return (np.asarray(state, dtype=F32) + sinusoid(t, cfg.d)[None, None, :]).astype(F32)
    if cfg.stem == "patch":
        return (linear(np.asarray(state, dtype=F32), weights["w_stem"])
                + weights["pos_emb"][None]).astype(F32)
    if cfg.stem == "patch_tokens":
        z = np.asarray(state, dtype=F32)
        B = z.shape[0]
        time_tok = np.broadcast_to(sinusoid(t, cfg.d)[None, None, :], (B, 1, cfg.d))
        cls_tok = weights["class_emb"][np.asarray(class_ids)][:, None, :]
        patches = linear(z, weights["w_stem"])
        h = np.concatenate([time_tok, cls_tok, patches], axis=1)
        return (h + weights["pos_emb"][None]).astype(F32)
    if cfg.stem == "identity":
        return np.array(state, dtype=F32, copy=True)
    if cfg.stem == "embed":
        return weights["embed"][np.asarray(state)].astype(F32)
    raise ValueError(cfg.stem)


def head(cfg, weights, h, c) -> np.ndarray:
    if cfg.head == "identity":
        return np.array(h, dtype=F32, copy=True)
    if cfg.head == "adaln_linear":
        shift, scale = np.split(linear(silu(c), weights["w_modf"]), 2, axis=-1)
        x = modulate(layer_norm(h, None, None, cfg.eps), shift, scale)
        return linear(x, weights["w_head"])[..., :cfg.out_channels]
    x = norm(cfg, h, weights, "normf")
    if cfg.n_prefix:
        x = x[:, cfg.n_prefix:]
    return linear(x, weights["w_head"])


def ctx_kv(cfg, weights, b, ctx):
    kv = linear(np.asarray(ctx, dtype=F32), weights[f"blocks.{b}.wx_kv"])
    return kv[..., :cfg.d], kv[..., cfg.d:]


def branch(cfg, weights, b: int, kind: str, h, c=None, ctx=None) -> np.ndarray:
    """Branch update F_u(h; c) of block b (Sec. 3.1), kind in {attn, xattn, mlp}."""
    p = f"blocks.{b}."
    d = cfg.d
    mod = block_modulation(weights, b, c) if cfg.block == "adaln" else None
    if kind == "attn":
        x = norm(cfg, h, weights, p + "norm1")
        if mod is not None:
            x = modulate(x, mod[0], mod[1])
        qkv = linear(x, weights[p + "w_qkv"])
        o = attention(qkv[..., :d], qkv[..., d:2 * d], qkv[..., 2 * d:], cfg.n_heads,
                      cfg.rope_theta if cfg.rope else None)
        y = linear(o, weights[p + "w_o"])
        if mod is not None:
            y = (mod[2][:, None, :] * y).astype(F32)
        return y
    if kind == "xattn":
        x = layer_norm(h, weights[p + "normx_w"], weights[p + "normx_b"], cfg.eps)
        q = linear(x, weights[p + "wx_q"])
        k, v = ctx_kv(cfg, weights, b, ctx)
        o = attention(q, k, v, cfg.n_heads)
        return linear(o, weights[p + "wx_o"])
    if kind == "mlp":
        x = norm(cfg, h, weights, p + "norm2")
        if mod is not None:
            x = modulate(x, mod[3], mod[4])
        u = linear(x, weights[p + "w_1"])
        f = cfg.d_ff
        if cfg.mlp == "swiglu":
            a = (silu(u[..., :f]) * u[..., f:]).astype(F32)
        elif cfg.mlp == "geglu":
            a = (u[..., :f] * gelu_erf(u[..., f:])).astype(F32)
        elif cfg.mlp == "gelu_tanh":
            a = gelu_tanh(u)
        else:
            a = gelu_erf(u)
        y = linear(a, weights[p + "w_2"])
        if mod is not None:
            y = (mod[5][:, None, :] * y).astype(F32)
        return y
    raise ValueError(kind)


def skip_combine(weights, j, h, skip):
    """U-ViT long skip: h <- W_skip_j [h ; skip]."""
    return linear(np.concatenate([h, skip], axis=-1), weights[f"skips.{j}.w"])


# ---------------------------------------------------------------------------
# scheduled forward (Algorithm 2)
# ---------------------------------------------------------------------------

class Trace:
    """Optional record of (unit, active, h_in, h_out) for invariant checks."""

    def __init__(self):
        self.units: List[tuple] = []


def denoise(cfg, weights, state, t: float, s: int, S_units: Sequence[int], cache: Dict,
            class_ids=None, ctx=None, trace: Optional[Trace] = None,
            active_units: Optional[Sequence[bool]] = None, with_head: bool = True):
    """One denoiser evaluation at step s (1-based) under lifetimes S_units.

    ``cache`` maps unit index -> stored Delta and is updated in place: an active unit
    (s <= S_u) computes Delta_{u,s} and refreshes its entry, a frozen unit (s > S_u)
    adds the entry written at its last active step.  Units are visited in graph order.
    ``active_units``, when given, replaces the lifetime rule (unit u is active iff
    active_units[u]):
    the input-aware policy of App. B.1 chooses the active set per step.
    With ``with_head`` False it returns (h_L, c) instead of the head's output, for callers
    that apply the head to a subset of tokens.
    """
    h = stem(cfg, weights, state, t, class_ids)
    c = conditioning(cfg, weights, t, class_ids)
    skips: List[np.ndarray] = []
    u = 0
    for b in range(cfg.n_blocks):
        if cfg.n_skips and b > cfg.n_skips:
            j = b - cfg.n_skips - 1
            h = skip_combine(weights, j, h, skips.pop())
        for kind in cfg.branches:
            h_in = h
            if (active_units[u] if active_units is not None else s <= S_units[u]):
                delta = branch(cfg, weights, b, kind, h, c, ctx)
                cache[u] = delta
                h = (h + delta).astype(F32)
                active = True
            else:
                if u not in cache:
                    raise RuntimeError(f"unit {u} frozen at step {s} before any refresh")
                h = (h + cache[u]).astype(F32)
                active = False
            if trace is not None:
                trace.units.append((u, active, h_in, h))
            u += 1
        if cfg.n_skips and b < cfg.n_skips:
            skips.append(h)
    if not with_head:
        return h, c
    return head(cfg, weights, h, c)


def denoise_full(cfg, weights, state, t: float, class_ids=None, ctx=None) -> np.ndarray:
    """Unscheduled forward: every branch evaluated and added (no cache)."""
    h = stem(cfg, weights, state, t, class_ids)
    c = conditioning(cfg, weights, t, class_ids)
    skips: List[np.ndarray] = []
    for b in range(cfg.n_blocks):
        if cfg.n_skips and b > cfg.n_skips:
            h = skip_combine(weights, b - cfg.n_skips - 1, h, skips.pop())
        for kind in cfg.branches:
            h = (h + branch(cfg, weights, b, kind, h, c, ctx)).astype(F32)
        if cfg.n_skips and b < cfg.n_skips:
            skips.append(h)
    return head(cfg, weights, h, c)


def to_numpy_weights(weights_torch) -> Dict[str, np.ndarray]:
    """bf16 torch tensors -> float32 NumPy arrays (exact: bf16 embeds in fp32)."""
    return {k: v.detach().float().cpu().numpy() for k, v in weights_torch.items()}
