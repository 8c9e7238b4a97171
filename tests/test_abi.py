"""Host-side checks of the C ABI (no GPU needed): the library loads, exports every
function that include/*.h declares, and its host-only paths validate arguments."""
import ctypes as C
import os
import re

import numpy as np
import pytest

from paper_2609_29505_gb300 import binding, synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2609_29505_gb300 import build
    build.build()
    return binding.lib()


def _declared():
    names = set()
    for f in os.listdir(os.path.join(ROOT, "include")):
        if f.endswith(".h"):
            src = open(os.path.join(ROOT, "include", f)).read()
            src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
            names |= set(re.findall(r"\b(sgd_[a-z0-9_]+)\s*\(", src))
    return names


def test_every_declared_symbol_is_exported(lib):
    declared = _declared()
    assert declared == set(binding.EXPORTED)
    for name in declared:
        assert hasattr(lib, name), name


def test_compile_schedule_patterns():
    # 3 blocks x 2 branches, T = 5: lifetimes 5, 2, 3 per block
    S = [5, 5, 2, 2, 3, 3]
    G = [0, 0, 1, 1, 2, 2]
    pos, wr, n = binding.sgd_compile_schedule(5, S, G)
    # active sets: s=1,2 all; s=3 blocks {0,2}; s=4,5 block {0}
    assert list(pos) == [0, 0, 1, 2, 2]
    assert n == 3
    # stores happen where a lifetime ends before T: s = 2 (block 1), s = 3 (block 2)
    assert list(wr) == [0, 2, 2, 0, 0]


def test_compile_schedule_matches_oracle_active_sets():
    from oracle import spectral as osp
    rng = np.random.default_rng(0)
    for _ in range(20):
        T = int(rng.integers(1, 12))
        n_blocks = int(rng.integers(1, 9))
        Sb = rng.integers(1, T + 1, size=n_blocks)
        S = np.repeat(Sb, 2)
        G = np.repeat(np.arange(n_blocks), 2)
        pos, wr, n = binding.sgd_compile_schedule(T, S, G)
        A = osp.active_sets(S, T)
        # same pattern id <=> same active set
        for a in range(T):
            for b in range(T):
                assert (pos[a] == pos[b]) == bool(np.array_equal(A[a], A[b]))
        assert n == len({tuple(r) for r in A})
        for s in range(1, T + 1):
            assert wr[s - 1] == sum(1 for x in S if x == s and s < T)


@pytest.mark.parametrize("S,G,code", [
    ([0, 0], [0, 0], binding.SGD_ERR_SCHEDULE),      # lifetime below 1
    ([6, 6], [0, 0], binding.SGD_ERR_SCHEDULE),      # lifetime above T
    ([3, 2], [0, 0], binding.SGD_ERR_SCHEDULE),      # atomic group split
])
def test_compile_schedule_rejects(S, G, code):
    with pytest.raises(binding.SgdError) as e:
        binding.sgd_compile_schedule(5, S, G)
    assert e.value.code == code


def test_create_rejects_bad_shapes_before_touching_a_device(lib):
    cfg = synth.get_config("tiny")
    for kw in (dict(d_head=96, d=384), dict(d=250), dict(n_blocks=0), dict(d_ff=100)):
        desc = binding.make_desc(cfg.with_(**kw))
        blocks = (binding.sgd_block_weights * max(cfg.n_blocks, 1))()
        W = binding.sgd_weights(blocks=blocks)
        h = C.c_void_p()
        rc = lib.sgd_create(C.byref(desc), C.byref(W), C.byref(h))
        assert rc == binding.SGD_ERR_SHAPE, (kw, rc)
        assert lib.sgd_last_error()


def test_create_rejects_missing_weights(lib):
    cfg = synth.get_config("tiny")
    desc = binding.make_desc(cfg)
    blocks = (binding.sgd_block_weights * cfg.n_blocks)()
    W = binding.sgd_weights(blocks=blocks, w_head=16, normf_w=16)
    h = C.c_void_p()
    assert lib.sgd_create(C.byref(desc), C.byref(W), C.byref(h)) == binding.SGD_ERR_ARG
    assert lib.sgd_create(None, C.byref(W), C.byref(h)) == binding.SGD_ERR_ARG


def test_null_context_calls_fail_cleanly(lib):
    assert lib.sgd_reset(None) == binding.SGD_ERR_ARG
    assert lib.sgd_set_schedule(None, 4, 2, None, None) == binding.SGD_ERR_ARG
    m = np.zeros(2, np.uint8)
    assert lib.sgd_get_active_mask(None, 1, m.ctypes.data, 2) == binding.SGD_ERR_ARG
    lib.sgd_destroy(None)


def test_kernel_entry_points_validate_on_host(lib):
    epi = binding.sgd_epilogue_args(kind=99)
    assert lib.sgd_kernel_gemm(None, 8, None, 8, 8, 8, 8, C.byref(epi), 0, None) == binding.SGD_ERR_ARG
    epi = binding.sgd_epilogue_args(kind=binding.EPI_F16, out=64, ldo=8)
    # K not a multiple of 8
    assert lib.sgd_kernel_gemm(64, 12, 64, 12, 8, 8, 12, C.byref(epi), 0, None) == binding.SGD_ERR_SHAPE
    assert lib.sgd_kernel_attention(64, 8, 64, 64, 8, 64, 8, 1, 4, 4, 1, 96, 0, None) == binding.SGD_ERR_SHAPE
    assert lib.sgd_kernel_attention(64, 8, 64, 64, 8, 64, 8, 1, 4, 4, 1, 64, 7, None) == binding.SGD_ERR_ARG
    assert lib.sgd_kernel_norm(None, None, 1, 8, 0, None, None, None, None, 0, 1, 1e-6, None) == binding.SGD_ERR_ARG
    arr = (C.c_void_p * 1)(None)
    assert lib.sgd_kernel_frozen_run(None, arr, 1, 8, None) == binding.SGD_ERR_ARG
