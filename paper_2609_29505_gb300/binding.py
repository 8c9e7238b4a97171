"""ctypes binding of libsgd (include/sgd.h, include/sgd_kernels.h).

Argument marshalling only: every step of the denoiser path runs in libsgd's
kernels.  The functions keep the C names; ``Denoiser`` is a small convenience
wrapper that builds the descriptor and weight structs from a config and a dict
of device tensors and keeps those tensors alive.

There is no fallback: if ``libsgd.so`` is missing or fails to load, every call
raises ``RuntimeError``.
"""
from __future__ import annotations

import ctypes as C
import os
from typing import Dict, List, Optional, Sequence

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libsgd.so")

# status codes (sgd_status)
SGD_OK = 0
SGD_ERR_ARG = -1
SGD_ERR_SHAPE = -2
SGD_ERR_SCHEDULE = -3
SGD_ERR_CACHE_INVALID = -4
SGD_ERR_CUDA = -5
SGD_ERR_DEVICE_TIMEOUT = -6
SGD_ERR_OOM = -7
SGD_ERR_STATE = -8
SGD_ERR_RANGE = -9
SGD_SELFTEST_TIMEOUT_CODE = 99  # status code recorded by sgd_selftest_wait_timeout

STEM = {"time_add": 0, "patch": 1, "patch_tokens": 2, "identity": 3, "embed": 4}
BLOCK = {"prenorm": 0, "adaln": 1, "xattn": 2}
NORM = {"rms": 0, "ln": 1, "ln_plain": 2}
MLP = {"swiglu": 0, "gelu_tanh": 1, "gelu_erf": 2, "geglu": 3}
HEAD = {"linear": 0, "adaln_linear": 1, "identity": 2, "logits": 3}
FLAG_SIMT_GEMM = 1
FLAG_MMA_SYNC_ATTENTION = 2
FLAG_GEMM_BK64 = 8
FLAG_PDL = 16
FLAG_FOLD_NORM = 32

EPI_F16, EPI_F32, EPI_DELTA, EPI_GATED, EPI_GELU, EPI_ROPE = range(6)
KERNEL_NAMES = ["gemm_tc", "gemm_simt", "attention", "norm", "frozen_run", "small"]

# every symbol include/*.h declares
EXPORTED = [
    "sgd_create", "sgd_set_schedule", "sgd_step", "sgd_step_host", "sgd_get_active_mask",
    "sgd_get_info", "sgd_reset", "sgd_check_device", "sgd_destroy", "sgd_last_error",
    "sgd_compile_schedule", "sgd_step_profile", "sgd_sampler_update", "sgd_kernel_gemm",
    "sgd_kernel_attention", "sgd_kernel_norm", "sgd_kernel_frozen_run", "sgd_kernel_status",
    "sgd_set_exec_mode", "sgd_step_host_async", "sgd_host_wait", "sgd_kernel_gemm_static_ws",
    "sgd_set_policy", "sgd_get_drift", "sgd_selftest_wait_timeout", "sgd_kernel_f16_clamped",
    "sgd_kernel_gemm_stat_slots", "sgd_kernel_attention_hs",
]
EXEC_JAGGED_GRAPH, EXEC_EAGER, EXEC_PADDED_GRAPH = 0, 1, 2
POLICY_STATIC, POLICY_DRIFT = 0, 1


class sgd_model_desc(C.Structure):
    _fields_ = [(n, C.c_int) for n in (
        "stem", "block", "norm", "mlp", "head", "n_blocks", "d", "n_heads", "d_head", "d_ff",
        "batch", "n_tokens", "n_prefix", "d_in", "d_out", "out_channels", "n_skips", "ctx_len",
        "d_ctx", "vocab", "n_classes", "t_freq", "rope")] + [
        ("rope_theta", C.c_float), ("eps", C.c_float), ("flags", C.c_int)]


class sgd_block_weights(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in (
        "norm1_w", "norm1_b", "w_qkv", "w_o", "normx_w", "normx_b", "wx_q", "wx_kv", "wx_o",
        "norm2_w", "norm2_b", "w_1", "w_2", "w_mod")]


class sgd_weights(C.Structure):
    _fields_ = [("blocks", C.POINTER(sgd_block_weights)), ("w_stem", C.c_void_p),
                ("pos_emb", C.c_void_p), ("w_t1", C.c_void_p), ("w_t2", C.c_void_p),
                ("class_emb", C.c_void_p), ("skip_w", C.POINTER(C.c_void_p)),
                ("normf_w", C.c_void_p), ("normf_b", C.c_void_p), ("w_modf", C.c_void_p),
                ("w_head", C.c_void_p), ("embed", C.c_void_p)]


class sgd_cond(C.Structure):
    _fields_ = [("class_ids", C.c_void_p), ("ctx", C.c_void_p)]


class sgd_info(C.Structure):
    _fields_ = [("n_units", C.c_int), ("n_patterns", C.c_int), ("n_graphs", C.c_int),
                ("T", C.c_int), ("layer_steps", C.c_int64), ("cache_bytes", C.c_size_t),
                ("workspace_bytes", C.c_size_t), ("weight_bytes", C.c_size_t),
                ("policy", C.c_int), ("n_groups", C.c_int), ("graph_steps", C.c_int64),
                ("eager_steps", C.c_int64)]


class sgd_op_record(C.Structure):
    _fields_ = [("name", C.c_char * 48), ("kernel", C.c_int), ("ms", C.c_float),
                ("flops", C.c_double), ("bytes", C.c_double)]


class sgd_epilogue_args(C.Structure):
    _fields_ = [("kind", C.c_int), ("alpha", C.c_float), ("out", C.c_void_p), ("ldo", C.c_int),
                ("h", C.c_void_p),
                ("ldh", C.c_int), ("cache", C.c_void_p), ("ld_cache", C.c_int),
                ("gate", C.c_void_p), ("ld_gate", C.c_int), ("rows_per_batch", C.c_int),
                ("act", C.c_int), ("rope_cos", C.c_void_p), ("rope_sin", C.c_void_p),
                ("rope_tokens", C.c_int), ("d_head", C.c_int), ("rope_cols", C.c_int),
                ("norm", C.c_int), ("rstat", C.c_void_p), ("stat_slots", C.c_int),
                ("stat_ld", C.c_int), ("norm_eps", C.c_float), ("colsum", C.c_void_p),
                ("colbias", C.c_void_p), ("h16", C.c_void_p), ("stat_out", C.c_void_p),
                ("stat_out_ld", C.c_int), ("stat_cnt", C.c_void_p), ("stat_final", C.c_void_p)]


_lib = None


def lib() -> C.CDLL:
    """Load libsgd.so (raises if it is absent: there is no fallback path)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"libsgd.so not built ({LIB_PATH}); run __graft_entry__.build()")
        L = C.CDLL(LIB_PATH)
        vp, i, i64, f = C.c_void_p, C.c_int, C.c_int64, C.c_float
        sig = {
            "sgd_create": (i, [C.POINTER(sgd_model_desc), C.POINTER(sgd_weights), C.POINTER(vp)]),
            "sgd_set_schedule": (i, [vp, i, i, vp, vp]),
            "sgd_step": (i, [vp, vp, vp, f, C.POINTER(sgd_cond), i, vp]),
            "sgd_step_host": (i, [vp, vp, vp, f, vp, vp, i, vp]),
            "sgd_get_active_mask": (i, [vp, i, vp, i]),
            "sgd_get_info": (i, [vp, C.POINTER(sgd_info)]),
            "sgd_reset": (i, [vp]),
            "sgd_check_device": (i, [vp, vp]),
            "sgd_destroy": (None, [vp]),
            "sgd_last_error": (C.c_char_p, []),
            "sgd_compile_schedule": (i, [i, i, vp, vp, vp, vp, vp]),
            "sgd_step_profile": (i, [vp, vp, vp, f, C.POINTER(sgd_cond), i, vp,
                                     C.POINTER(sgd_op_record), i, C.POINTER(C.c_int)]),
            "sgd_sampler_update": (i, [vp, vp, f, f, i64, vp]),
            "sgd_kernel_gemm": (i, [vp, i, vp, i, i, i, i, C.POINTER(sgd_epilogue_args), i, vp]),
            "sgd_kernel_gemm_static_ws": (i, [vp, i, vp, i, i, i, i, C.POINTER(sgd_epilogue_args), i, vp]),
            "sgd_kernel_attention": (i, [vp, i, vp, vp, i, vp, i, i, i, i, i, i, i, vp]),
            "sgd_kernel_attention_hs": (i, [vp, i, vp, vp, i, i, vp, i, i, i, i, i, i, i, vp]),
            "sgd_kernel_norm": (i, [vp, vp, i, i, i, vp, vp, vp, vp, i, i, f, vp]),
            "sgd_kernel_frozen_run": (i, [vp, C.POINTER(vp), i, i64, vp]),
            "sgd_kernel_status": (i, [C.POINTER(C.c_int)]),
            "sgd_kernel_f16_clamped": (i, [C.POINTER(C.c_int)]),
            "sgd_kernel_gemm_stat_slots": (i, [i, i, i, C.POINTER(sgd_epilogue_args), i, C.POINTER(C.c_int)]),
            "sgd_set_exec_mode": (i, [vp, i]),
            "sgd_step_host_async": (i, [vp, vp, vp, f, vp, vp, i, vp]),
            "sgd_host_wait": (i, [vp]),
            "sgd_set_policy": (i, [vp, i]),
            "sgd_selftest_wait_timeout": (i, [vp]),
            "sgd_get_drift": (i, [vp, i, vp, i]),
        }
        for name, (res, args) in sig.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _lib = L
    return _lib


class SgdError(RuntimeError):
    def __init__(self, code: int, where: str):
        msg = lib().sgd_last_error().decode(errors="replace")
        super().__init__(f"{where} failed with status {code}: {msg}")
        self.code = code


def check(code: int, where: str) -> int:
    if code != SGD_OK:
        raise SgdError(code, where)
    return code


def _ptr(t) -> Optional[int]:
    return None if t is None else t.data_ptr()


def _stream(stream) -> Optional[int]:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    return stream if isinstance(stream, int) else stream.cuda_stream


# ---------------------------------------------------------------------------
# thin wrappers with the C names
# ---------------------------------------------------------------------------

def sgd_compile_schedule(T: int, lifetimes: Sequence[int], groups: Sequence[int]):
    """Host-only schedule compiler: (pattern_of_step[T], writes_at_step[T], n_patterns)."""
    S = np.ascontiguousarray(lifetimes, dtype=np.int32)
    G = np.ascontiguousarray(groups, dtype=np.int32)
    pos = np.zeros(T, np.int32)
    wr = np.zeros(T, np.int32)
    n = C.c_int32()
    check(lib().sgd_compile_schedule(T, len(S), S.ctypes.data, G.ctypes.data, pos.ctypes.data,
                                     wr.ctypes.data, C.byref(n)), "sgd_compile_schedule")
    return pos, wr, int(n.value)


def sgd_kernel_gemm(A, B, M, N, K, epi: sgd_epilogue_args, use_simt=False, lda=None, ldb=None,
                    stream=None):
    return check(lib().sgd_kernel_gemm(_ptr(A), lda or K, _ptr(B), ldb or K, M, N, K,
                                       C.byref(epi), int(use_simt), _stream(stream)),
                 "sgd_kernel_gemm")


def sgd_kernel_gemm_static_ws(A, B, M, N, K, epi: sgd_epilogue_args, variant=0, lda=None, ldb=None,
                              stream=None):
    """sgd_kernel_gemm that allocates no device memory (stream-K scratch in a fixed array)."""
    return check(lib().sgd_kernel_gemm_static_ws(_ptr(A), lda or K, _ptr(B), ldb or K, M, N, K,
                                                 C.byref(epi), int(variant), _stream(stream)),
                 "sgd_kernel_gemm_static_ws")


def sgd_kernel_attention(q, ldq, k, v, ldkv, o, ldo, batch, n_q, n_kv, n_heads, d_head,
                         impl=0, stream=None):
    return check(lib().sgd_kernel_attention(_ptr(q), ldq, _ptr(k), _ptr(v), ldkv, _ptr(o), ldo,
                                            batch, n_q, n_kv, n_heads, d_head, impl,
                                            _stream(stream)), "sgd_kernel_attention")


def sgd_kernel_attention_hs(q, ldq, k, v, ldkv, head_stride, o, ldo, batch, n_q, n_kv, n_heads,
                            d_head, impl=0, stream=None):
    return check(lib().sgd_kernel_attention_hs(_ptr(q), ldq, _ptr(k), _ptr(v), ldkv, head_stride,
                                               _ptr(o), ldo, batch, n_q, n_kv, n_heads, d_head,
                                               impl, _stream(stream)), "sgd_kernel_attention_hs")


def sgd_kernel_norm(h, out, rows, d, kind, g=None, b=None, shift=None, scale=None, ld_mod=0,
                    rows_per_batch=1, eps=1e-6, stream=None):
    return check(lib().sgd_kernel_norm(_ptr(h), _ptr(out), rows, d, kind, _ptr(g), _ptr(b),
                                       _ptr(shift), _ptr(scale), ld_mod, rows_per_batch, eps,
                                       _stream(stream)), "sgd_kernel_norm")


def sgd_kernel_frozen_run(h, caches, stream=None):
    arr = (C.c_void_p * len(caches))(*[c.data_ptr() for c in caches])
    return check(lib().sgd_kernel_frozen_run(_ptr(h), arr, len(caches), h.numel(),
                                             _stream(stream)), "sgd_kernel_frozen_run")


def sgd_kernel_status() -> int:
    st = C.c_int(0)
    check(lib().sgd_kernel_status(C.byref(st)), "sgd_kernel_status")
    return int(st.value)


def sgd_kernel_gemm_stat_slots(M, N, K, epi: "sgd_epilogue_args", variant=0) -> int:
    n = C.c_int(0)
    check(lib().sgd_kernel_gemm_stat_slots(M, N, K, C.byref(epi), int(variant), C.byref(n)),
          "sgd_kernel_gemm_stat_slots")
    return int(n.value)


def sgd_kernel_f16_clamped() -> int:
    st = C.c_int(0)
    check(lib().sgd_kernel_f16_clamped(C.byref(st)), "sgd_kernel_f16_clamped")
    return int(st.value)


def sgd_sampler_update(z, eps, alpha, beta, stream=None):
    return check(lib().sgd_sampler_update(_ptr(z), _ptr(eps), alpha, beta, z.numel(),
                                          _stream(stream)), "sgd_sampler_update")


def make_desc(cfg, flags: int = 0) -> sgd_model_desc:
    return sgd_model_desc(
        stem=STEM[cfg.stem], block=BLOCK[cfg.block], norm=NORM[cfg.norm], mlp=MLP[cfg.mlp],
        head=HEAD[cfg.head], n_blocks=cfg.n_blocks, d=cfg.d, n_heads=cfg.n_heads,
        d_head=cfg.d_head, d_ff=cfg.d_ff, batch=cfg.batch, n_tokens=cfg.n_tokens,
        n_prefix=cfg.n_prefix, d_in=cfg.d_in, d_out=cfg.d_out, out_channels=cfg.out_channels,
        n_skips=cfg.n_skips, ctx_len=cfg.ctx_len, d_ctx=cfg.d_ctx, vocab=cfg.vocab,
        n_classes=cfg.n_classes, t_freq=cfg.t_freq, rope=int(cfg.rope),
        rope_theta=cfg.rope_theta, eps=cfg.eps, flags=flags)


class Denoiser:
    """One libsgd context for a model config and its device weights."""

    def __init__(self, cfg, weights: Dict[str, "object"], flags: int = 0):
        self.cfg = cfg
        self._w = weights  # keep the tensors alive for the context's lifetime
        self.n_units = cfg.n_units
        blocks = (sgd_block_weights * cfg.n_blocks)()
        for b in range(cfg.n_blocks):
            for f, _ in sgd_block_weights._fields_:
                setattr(blocks[b], f, _ptr(weights.get(f"blocks.{b}.{f}")))
        self._blocks = blocks
        skips = (C.c_void_p * max(cfg.n_skips, 1))()
        for j in range(cfg.n_skips):
            skips[j] = _ptr(weights[f"skips.{j}.w"])
        self._skips = skips
        W = sgd_weights(blocks=blocks, skip_w=skips)
        for f in ("w_stem", "pos_emb", "w_t1", "w_t2", "class_emb", "normf_w", "normf_b",
                  "w_modf", "w_head", "embed"):
            setattr(W, f, _ptr(weights.get(f)))
        self._desc = make_desc(cfg, flags)
        h = C.c_void_p()
        check(lib().sgd_create(C.byref(self._desc), C.byref(W), C.byref(h)), "sgd_create")
        self.handle = h.value
        self.T = 0

    def close(self):
        if getattr(self, "handle", None):
            lib().sgd_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def set_schedule(self, T: int, lifetimes: Sequence[int], groups: Sequence[int]):
        S = np.ascontiguousarray(lifetimes, dtype=np.int32)
        G = np.ascontiguousarray(groups, dtype=np.int32)
        check(lib().sgd_set_schedule(self.handle, T, len(S), S.ctypes.data, G.ctypes.data),
              "sgd_set_schedule")
        self.T = T

    def _cond(self, class_ids=None, ctx=None) -> sgd_cond:
        return sgd_cond(class_ids=_ptr(class_ids), ctx=_ptr(ctx))

    def step(self, state, out, t: float, step: int, class_ids=None, ctx=None, stream=None):
        cond = self._cond(class_ids, ctx)
        return check(lib().sgd_step(self.handle, _ptr(state), _ptr(out), float(t),
                                    C.byref(cond), step, _stream(stream)), "sgd_step")

    def step_host(self, state_host, out_host, t: float, step: int, class_ids_host=None,
                  ctx_host=None, stream=None):
        """Host (preferably pinned) torch tensors in and out; synchronous."""
        return check(lib().sgd_step_host(self.handle, _ptr(state_host), _ptr(out_host),
                                         float(t), _ptr(class_ids_host), _ptr(ctx_host), step,
                                         _stream(stream)), "sgd_step_host")

    def step_host_async(self, state_host, out_host, t: float, step: int, class_ids_host=None,
                        ctx_host=None, stream=None):
        """Queued host-buffer step; out_host is valid after host_wait()."""
        return check(lib().sgd_step_host_async(self.handle, _ptr(state_host), _ptr(out_host),
                                               float(t), _ptr(class_ids_host), _ptr(ctx_host),
                                               step, _stream(stream)), "sgd_step_host_async")

    def host_wait(self):
        return check(lib().sgd_host_wait(self.handle), "sgd_host_wait")

    def profile_step(self, state, out, t: float, step: int, class_ids=None, ctx=None,
                     stream=None, max_records: int = 4096) -> List[dict]:
        cond = self._cond(class_ids, ctx)
        recs = (sgd_op_record * max_records)()
        n = C.c_int(0)
        check(lib().sgd_step_profile(self.handle, _ptr(state), _ptr(out), float(t),
                                     C.byref(cond), step, _stream(stream), recs, max_records,
                                     C.byref(n)), "sgd_step_profile")
        return [dict(name=recs[i].name.decode(), kernel=KERNEL_NAMES[recs[i].kernel],
                     ms=recs[i].ms, flops=recs[i].flops, bytes=recs[i].bytes)
                for i in range(n.value)]

    def active_mask(self, step: int) -> np.ndarray:
        m = np.zeros(self.n_units, np.uint8)
        check(lib().sgd_get_active_mask(self.handle, step, m.ctypes.data, self.n_units),
              "sgd_get_active_mask")
        return m

    def info(self) -> dict:
        i = sgd_info()
        check(lib().sgd_get_info(self.handle, C.byref(i)), "sgd_get_info")
        return {f: getattr(i, f) for f, _ in sgd_info._fields_}

    def reset(self):
        check(lib().sgd_reset(self.handle), "sgd_reset")

    def set_exec_mode(self, mode: int):
        check(lib().sgd_set_exec_mode(self.handle, mode), "sgd_set_exec_mode")

    def set_policy(self, policy: int):
        """POLICY_STATIC (lifetimes) or POLICY_DRIFT (the input-aware baseline of App. B.1)."""
        check(lib().sgd_set_policy(self.handle, policy), "sgd_set_policy")

    def drift(self, step: int) -> np.ndarray:
        """Lagged drifts the drift policy ranked to choose `step`'s active groups."""
        n = self.info()["n_groups"]
        d = np.zeros(n, np.float64)
        check(lib().sgd_get_drift(self.handle, step, d.ctypes.data, n), "sgd_get_drift")
        return d

    def check_device(self, stream=None):
        return check(lib().sgd_check_device(self.handle, _stream(stream)), "sgd_check_device")
