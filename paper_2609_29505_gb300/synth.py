"""Seeded synthetic models and inputs shaped like the paper's workloads.

This module holds shapes and random-number generation only; it contains none
of the method's arithmetic (no spectra, no scores, no forward pass).  Both the
CUDA path and the CPU oracle receive the tensors it produces, so the two sides
always see identical bytes.

Workloads (Sec. 5 and Table ``tab:protocol`` of the paper name LLaDA-8B,
DiT-XL/2, U-ViT-L and SDXL; their datasets and checkpoints are not used):

* every linear weight is ``U diag(s) V^T`` with power-law singular values
  ``s_i ~ i^-alpha``, ``alpha ~ U[0.3, 1.5]`` per matrix, scaled so that the
  Frobenius norm is ``sqrt(min(m, n))`` (RMS singular value 1), then rounded
  to bf16;
* norm gains are ``1 + 0.1 N(0,1)``, LayerNorm shifts ``0.1 N(0,1)``;
* embeddings (token, class, position) are ``N(0,1)`` (position ``0.1 N(0,1)``);
* inputs are ``N(0,1)`` rounded to bf16-representable values; class ids are
  uniform; LLaDA token ids follow a seeded reveal sequence that does not depend
  on the model's outputs.

Random numbers come from ``torch.Generator`` seeded per config; generation may
run on the CPU (small configs) or on a CUDA device (large configs), and every
consumer receives the same tensors within a run.
"""
from __future__ import annotations

import copy
import math
from dataclasses import dataclass, field, asdict
from typing import Dict, List, Optional

import torch

WEIGHT_SEED_BASE = 1234
INPUT_SEED = 4321
LLADA_MASK_ID = 126336


@dataclass
class ModelConfig:
    """Shape of one synthetic denoiser (all sizes in elements)."""

    name: str
    stem: str            # time_add | patch | patch_tokens | identity | embed
    block: str           # prenorm | adaln | xattn
    norm: str            # rms | ln (affine) | ln_plain (no affine, AdaLN)
    mlp: str             # swiglu | gelu_tanh | gelu_erf | geglu
    head: str            # linear | adaln_linear | identity | logits
    n_blocks: int
    d: int
    n_heads: int
    d_head: int
    d_ff: int
    batch: int
    n_tokens: int        # tokens per sample seen by the blocks
    d_in: int            # channels of the input state (0 for token ids)
    d_out: int           # rows of the head weight (0 for identity)
    out_channels: int    # channels written per output token
    T: int               # denoising horizon
    rope: bool = False
    rope_theta: float = 10000.0
    eps: float = 1e-6
    n_prefix: int = 0    # U-ViT time + class tokens ahead of the patches
    n_skips: int = 0     # U-ViT long skips
    ctx_len: int = 0     # SDXL conditioning tokens
    d_ctx: int = 0
    vocab: int = 0
    n_classes: int = 0
    t_freq: int = 0      # DiT sinusoidal frequency width fed to the t-MLP
    seed: int = WEIGHT_SEED_BASE
    horizons: List[int] = field(default_factory=list)

    @property
    def branches(self) -> List[str]:
        """Residual branches of one block, in graph order."""
        if self.block == "xattn":
            return ["attn", "xattn", "mlp"]
        return ["attn", "mlp"]

    @property
    def n_units(self) -> int:
        return self.n_blocks * len(self.branches)

    @property
    def gated(self) -> bool:
        return self.mlp in ("swiglu", "geglu")

    @property
    def rows(self) -> int:
        return self.batch * self.n_tokens

    @property
    def n_in_tokens(self) -> int:
        """Tokens per sample in the input state (U-ViT: patches only)."""
        return self.n_tokens - self.n_prefix

    @property
    def n_out_tokens(self) -> int:
        return self.n_tokens - self.n_prefix

    def with_(self, **kw) -> "ModelConfig":
        c = copy.deepcopy(self)
        for k, v in kw.items():
            setattr(c, k, v)
        return c

    def as_dict(self) -> Dict:
        return asdict(self)


def _cfg(**kw) -> ModelConfig:
    return ModelConfig(**kw)


# The five workloads, in the order they are listed for this method.
CONFIGS: Dict[str, ModelConfig] = {
    "tiny": _cfg(name="tiny", stem="time_add", block="prenorm", norm="rms", mlp="swiglu",
                 head="linear", n_blocks=4, d=256, n_heads=4, d_head=64, d_ff=688, batch=1,
                 n_tokens=64, d_in=256, d_out=256, out_channels=256, T=10,
                 seed=WEIGHT_SEED_BASE + 0, horizons=[10]),
    "dit": _cfg(name="dit", stem="patch", block="adaln", norm="ln_plain", mlp="gelu_tanh",
                head="adaln_linear", n_blocks=28, d=1152, n_heads=16, d_head=72, d_ff=4608,
                batch=8, n_tokens=256, d_in=16, d_out=32, out_channels=16, T=50,
                n_classes=1001, t_freq=256, seed=WEIGHT_SEED_BASE + 1, horizons=[50]),
    "uvit": _cfg(name="uvit", stem="patch_tokens", block="prenorm", norm="ln", mlp="gelu_erf",
                 head="linear", n_blocks=21, d=1024, n_heads=16, d_head=64, d_ff=4096,
                 batch=16, n_tokens=258, d_in=16, d_out=16, out_channels=16, T=50,
                 n_prefix=2, n_skips=10, n_classes=1001, seed=WEIGHT_SEED_BASE + 2,
                 horizons=[50]),
    "sdxl": _cfg(name="sdxl", stem="identity", block="xattn", norm="ln", mlp="geglu",
                 head="identity", n_blocks=10, d=1280, n_heads=20, d_head=64, d_ff=5120,
                 batch=2, n_tokens=1024, d_in=1280, d_out=0, out_channels=1280, T=30,
                 ctx_len=77, d_ctx=2048, seed=WEIGHT_SEED_BASE + 3, horizons=[30]),
    "llada": _cfg(name="llada", stem="embed", block="prenorm", norm="rms", mlp="swiglu",
                  head="logits", n_blocks=32, d=4096, n_heads=32, d_head=128, d_ff=12288,
                  batch=4, n_tokens=1024, d_in=0, d_out=126464, out_channels=126464, T=64,
                  rope=True, vocab=126464, seed=WEIGHT_SEED_BASE + 4, horizons=[64, 10]),
}

# Reduced models with the same structure and the same awkward sizes (head dim 72,
# ragged token counts, K tails, a vocabulary that is not a tile multiple) that the
# CPU oracle evaluates in seconds.  They still span several 128-row tiles.
SMALL_CONFIGS: Dict[str, ModelConfig] = {
    "tiny": CONFIGS["tiny"],
    "dit_small": CONFIGS["dit"].with_(name="dit_small", n_blocks=3, d=288, n_heads=4, d_ff=1152,
                                      batch=2, n_tokens=136, T=8, n_classes=11, t_freq=64,
                                      horizons=[8]),
    "uvit_small": CONFIGS["uvit"].with_(name="uvit_small", n_blocks=5, d=256, n_heads=4,
                                        d_ff=1024, batch=3, n_tokens=66, n_skips=2, T=8,
                                        n_classes=11, horizons=[8]),
    "sdxl_small": CONFIGS["sdxl"].with_(name="sdxl_small", n_blocks=2, d=320, n_heads=5,
                                        d_ff=640, batch=2, n_tokens=200, d_in=320,
                                        out_channels=320, ctx_len=77, d_ctx=256, T=6,
                                        horizons=[6]),
    "llada_small": CONFIGS["llada"].with_(name="llada_small", n_blocks=3, d=512, n_heads=4,
                                          d_ff=1376, batch=2, n_tokens=192, vocab=1000,
                                          d_out=1000, out_channels=1000, T=8, horizons=[8]),
}

# Longer context: the LLaDA-8B-shaped model on one 4096-token sequence (the length of the
# paper's Needle-in-a-Haystack 4K setting), same weights seed as "llada".
EXTRA_CONFIGS: Dict[str, ModelConfig] = {
    "llada_4k": CONFIGS["llada"].with_(name="llada_4k", batch=1, n_tokens=4096, horizons=[64]),
}

ALL_CONFIGS: Dict[str, ModelConfig] = {**CONFIGS, **SMALL_CONFIGS, **EXTRA_CONFIGS}

BUDGETS = (1.0, 0.5, 0.33)


def get_config(name: str) -> ModelConfig:
    return copy.deepcopy(ALL_CONFIGS[name])


def mask_id(cfg: ModelConfig) -> int:
    """Id of the [MASK] token: LLaDA's id when it fits the vocabulary, else the last id."""
    return LLADA_MASK_ID if cfg.vocab > LLADA_MASK_ID else cfg.vocab - 1


# ---------------------------------------------------------------------------
# weight generation
# ---------------------------------------------------------------------------

def _bf16(x: torch.Tensor) -> torch.Tensor:
    return x.to(torch.bfloat16)


def _orthonormal(gen: torch.Generator, rows: int, cols: int, device) -> torch.Tensor:
    """Columns of a Haar-like orthonormal frame: QR of a Gaussian, with the sign fix."""
    g = torch.randn(rows, cols, generator=gen, device=device, dtype=torch.float32)
    q, r = torch.linalg.qr(g, mode="reduced")
    sign = torch.sign(torch.diagonal(r))
    sign[sign == 0] = 1.0
    return q * sign


def power_law_matrix(gen: torch.Generator, m: int, n: int, device) -> torch.Tensor:
    """bf16 [m, n] matrix U diag(s) V^T, s_i ~ i^-alpha, ||W||_F = sqrt(min(m, n))."""
    d = min(m, n)
    alpha = 0.3 + 1.2 * torch.rand((), generator=gen, device=device, dtype=torch.float64).item()
    i = torch.arange(1, d + 1, dtype=torch.float64)
    s = i.pow(-alpha)
    s = s * (math.sqrt(d) / torch.linalg.vector_norm(s))
    u = _orthonormal(gen, m, d, device)
    v = _orthonormal(gen, n, d, device)
    w = (u * s.to(device=device, dtype=torch.float32)) @ v.T
    return _bf16(w)


def _gauss(gen, shape, device, scale=1.0, offset=0.0) -> torch.Tensor:
    return _bf16(offset + scale * torch.randn(*shape, generator=gen, device=device,
                                                dtype=torch.float32))


def weight_names(cfg: ModelConfig) -> List[str]:
    return list(weight_shapes(cfg).keys())


def weight_shapes(cfg: ModelConfig) -> Dict[str, tuple]:
    """Name -> shape of every weight tensor (row-major [out, in] for linears)."""
    d, f = cfg.d, cfg.d_ff
    s: Dict[str, tuple] = {}
    has_bias = cfg.norm == "ln"
    has_gain = cfg.norm in ("rms", "ln")
    for b in range(cfg.n_blocks):
        p = f"blocks.{b}."
        if has_gain:
            s[p + "norm1_w"] = (d,)
        if has_bias:
            s[p + "norm1_b"] = (d,)
        s[p + "w_qkv"] = (3 * d, d)
        s[p + "w_o"] = (d, d)
        if cfg.block == "xattn":
            s[p + "normx_w"] = (d,)
            s[p + "normx_b"] = (d,)
            s[p + "wx_q"] = (d, d)
            s[p + "wx_kv"] = (2 * d, cfg.d_ctx)
            s[p + "wx_o"] = (d, d)
        if has_gain:
            s[p + "norm2_w"] = (d,)
        if has_bias:
            s[p + "norm2_b"] = (d,)
        s[p + "w_1"] = (2 * f if cfg.gated else f, d)
        s[p + "w_2"] = (d, f)
        if cfg.block == "adaln":
            s[p + "w_mod"] = (6 * d, d)
    if cfg.stem in ("patch", "patch_tokens"):
        s["w_stem"] = (d, cfg.d_in)
        s["pos_emb"] = (cfg.n_tokens, d)
    if cfg.block == "adaln":
        s["w_t1"] = (d, cfg.t_freq)
        s["w_t2"] = (d, d)
    if cfg.n_classes:
        s["class_emb"] = (cfg.n_classes, d)
    for k in range(cfg.n_skips):
        s[f"skips.{k}.w"] = (d, 2 * d)
    if cfg.head != "identity":
        if cfg.head == "adaln_linear":
            s["w_modf"] = (2 * d, d)
        else:
            s["normf_w"] = (d,)
            if cfg.norm == "ln":
                s["normf_b"] = (d,)
        s["w_head"] = (cfg.d_out, d)
    if cfg.stem == "embed":
        s["embed"] = (cfg.vocab, d)
    return s


def make_weights(cfg: ModelConfig, device="cpu") -> Dict[str, torch.Tensor]:
    """All weights of ``cfg`` as bf16 tensors on ``device`` (seeded by ``cfg.seed``)."""
    gen = torch.Generator(device=device)
    gen.manual_seed(cfg.seed)
    out: Dict[str, torch.Tensor] = {}
    for name, shape in weight_shapes(cfg).items():
        leaf = name.split(".")[-1]
        if len(shape) == 1:
            if leaf.endswith("_b"):
                out[name] = _gauss(gen, shape, device, scale=0.1)
            else:
                out[name] = _gauss(gen, shape, device, scale=0.1, offset=1.0)
        elif leaf in ("class_emb", "embed"):
            out[name] = _gauss(gen, shape, device)
        elif leaf == "pos_emb":
            out[name] = _gauss(gen, shape, device, scale=0.1)
        else:
            out[name] = power_law_matrix(gen, shape[0], shape[1], device)
    return out


# ---------------------------------------------------------------------------
# inputs
# ---------------------------------------------------------------------------

@dataclass
class Inputs:
    """Per-trajectory inputs: initial state, conditioning, timesteps."""

    z0: Optional[torch.Tensor]          # fp32 [B, N_in, d_in] (None for token models)
    class_ids: Optional[torch.Tensor]   # int32 [B]
    ctx: Optional[torch.Tensor]         # bf16 [B, ctx_len, d_ctx]
    ids_target: Optional[torch.Tensor]  # int32 [B, N] (token models)
    reveal_order: Optional[torch.Tensor]  # int64 [B, N] permutation (token models)


def timestep(cfg: ModelConfig, s: int, T: Optional[int] = None) -> float:
    """Timestep fed at evaluation s (1 = noisiest): t_s = 1000 (T - s + 1) / T."""
    T = T or cfg.T
    return 1000.0 * (T - s + 1) / T


def make_inputs(cfg: ModelConfig, device="cpu", seed: int = INPUT_SEED) -> Inputs:
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    B = cfg.batch
    z0 = class_ids = ctx = ids = order = None
    if cfg.stem == "embed":
        ids = torch.randint(0, mask_id(cfg), (B, cfg.n_tokens), generator=gen, device=device,
                            dtype=torch.int64).to(torch.int32)
        order = torch.stack([torch.randperm(cfg.n_tokens, generator=gen, device=device)
                             for _ in range(B)])
    else:
        z0 = _bf16(torch.randn(B, cfg.n_in_tokens, cfg.d_in, generator=gen, device=device,
                               dtype=torch.float32)).float()
    if cfg.n_classes:
        class_ids = torch.randint(0, cfg.n_classes - 1, (B,), generator=gen, device=device,
                                  dtype=torch.int64).to(torch.int32)
    if cfg.ctx_len:
        ctx = _gauss(gen, (B, cfg.ctx_len, cfg.d_ctx), device)
    return Inputs(z0, class_ids, ctx, ids, order)


def token_ids_at(cfg: ModelConfig, inp: Inputs, s: int, T: Optional[int] = None) -> torch.Tensor:
    """Token ids at evaluation s: the first floor((s-1) N / T) positions of each row's
    reveal order carry their target id, every other position is [MASK]."""
    T = T or cfg.T
    n_rev = ((s - 1) * cfg.n_tokens) // T
    ids = torch.full_like(inp.ids_target, mask_id(cfg))
    if n_rev > 0:
        pos = inp.reveal_order[:, :n_rev]
        ids.scatter_(1, pos, torch.gather(inp.ids_target, 1, pos))
    return ids


def weights_checksum(weights) -> str:
    """sha256 over every weight tensor's name, shape, dtype and two exact integer checksums of
    its raw 16- or 32-bit words (a plain sum and a position-weighted sum), computed where the
    tensor lives in chunks, so that device-resident weights need no host copy.  It identifies
    one generated model (a stored schedule or stored scores belong to these exact bytes)."""
    import hashlib

    import numpy as np

    h = hashlib.sha256()
    for name in sorted(weights):
        t = weights[name]
        if not isinstance(t, torch.Tensor):
            t = torch.from_numpy(np.ascontiguousarray(t))
        v = t.detach().contiguous().reshape(-1)
        if v.element_size() == 2:
            v = v.view(torch.int16)
        elif v.element_size() == 4:
            v = v.view(torch.int32)
        s1 = s2 = 0
        chunk = 1 << 24
        for i in range(0, v.numel(), chunk):
            x = v[i:i + chunk].to(torch.int64)
            pos = torch.arange(i, i + x.numel(), device=x.device, dtype=torch.int64) % 65521 + 1
            s1 += int(x.sum())
            s2 += int(((x + 65537) * pos).sum())
        h.update(f"{name}|{tuple(t.shape)}|{t.dtype}|{s1}|{s2};".encode())
    return h.hexdigest()


def unit_names(cfg: ModelConfig) -> List[str]:
    """Residual units (branches) in graph order: 'b{block}.{branch}'."""
    return [f"b{b}.{br}" for b in range(cfg.n_blocks) for br in cfg.branches]


def block_groups(cfg: ModelConfig) -> List[int]:
    """Default atomic grouping: all branches of one block form one group."""
    return [b for b in range(cfg.n_blocks) for _ in cfg.branches]


def branch_groups(cfg: ModelConfig) -> List[int]:
    """Branch granularity: every branch is its own group."""
    return list(range(cfg.n_units))
