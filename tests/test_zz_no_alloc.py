"""The allocation-free GEMM entry point (sgd_kernel_gemm_static_ws) against the allocating
one (sgd_kernel_gemm).

Both run the same kernels with the same stream-K split, so their outputs must agree bit for
bit.  Each case calls the allocation-free entry twice in a row: the second call checks that
the fixed scratch (partial tiles and tile tickets) is ready for the next call.  The file is
named to be collected last, so that in a full run it also follows every other GPU test,
which use the library's allocating workspaces in the same process."""
import ctypes as C
import math

import numpy as np
import pytest
import torch

from paper_2609_29505_gb300 import binding


@pytest.fixture(scope="module")
def B():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    from paper_2609_29505_gb300 import build
    build.build()
    binding.lib()
    return binding


def _rand(rng, shape, scale=1.0):
    return torch.from_numpy((rng.standard_normal(shape) * scale).astype(np.float32)).half()


KINDS = {"f16": binding.EPI_F16, "delta": binding.EPI_DELTA, "gelu": binding.EPI_GELU,
         "gated": binding.EPI_GATED}


def _problem(M, N, K, epi, seed):
    rng = np.random.default_rng(seed)
    A = _rand(rng, (M, K)).cuda()
    W = _rand(rng, (2 * N if epi == "gated" else N, K), 1 / math.sqrt(K)).cuda()
    h0 = torch.from_numpy(rng.standard_normal((M, N)).astype(np.float32)).cuda()
    return A, W, h0


def _run(entry, A, W, h0, M, N, K, epi, variant, stream=None):
    """One call of `entry`; returns the tensors it wrote (fresh buffers per call)."""
    if epi == "delta":
        h = h0.clone()
        cache = torch.zeros(M, N, dtype=torch.float16, device="cuda")
        e = binding.sgd_epilogue_args(kind=KINDS[epi], h=h.data_ptr(), ldh=N, cache=cache.data_ptr(),
                                      ld_cache=N)
        entry(A, W, M, N, K, e, variant, stream=stream)
        return h, cache
    out = torch.empty(M, N, dtype=torch.float16, device="cuda")
    e = binding.sgd_epilogue_args(kind=KINDS[epi], out=out.data_ptr(), ldo=N)
    entry(A, W, M, N, K, e, variant, stream=stream)
    return (out,)


@pytest.mark.gpu
@pytest.mark.parametrize("M,N,K,epi,variant", [
    (4096, 4096, 4096, "f16", 9),     # stream-K forced (attention-output shape)
    (4096, 4096, 12288, "delta", 9),  # stream-K forced (MLP down-projection shape)
    (2048, 1152, 1152, "delta", 9),   # stream-K forced, 128-column tiles
    (1000, 1376, 512, "gelu", 9),     # ragged M and N
    (2048, 2752, 1024, "gated", 9),   # 48 split tiles x 4 segments: 24 MiB of partials
    (520, 264, 688, "f16", 8),        # data-parallel: the scratch is not touched
])
def test_static_ws_matches_allocating_entry(B, M, N, K, epi, variant):
    A, W, h0 = _problem(M, N, K, epi, M + N + K)
    ref = _run(B.sgd_kernel_gemm, A, W, h0, M, N, K, epi, variant)
    first = _run(B.sgd_kernel_gemm_static_ws, A, W, h0, M, N, K, epi, variant)
    second = _run(B.sgd_kernel_gemm_static_ws, A, W, h0, M, N, K, epi, variant)
    torch.cuda.synchronize()
    assert B.sgd_kernel_status() == 0
    for r, x, y in zip(ref, first, second):
        assert torch.equal(x, r)
        assert torch.equal(y, r)


@pytest.mark.gpu
def test_static_ws_allocates_no_device_memory(B):
    """Free device memory is unchanged by stream-K calls of the allocation-free entry; the
    allocating entry, given a stream it has not seen, creates a workspace for it (which
    shows that the measurement can see such an allocation)."""
    M = N = K = 4096
    A, W, h0 = _problem(M, N, K, "f16", 11)
    out = torch.empty(M, N, dtype=torch.float16, device="cuda")
    e = B.sgd_epilogue_args(kind=B.EPI_F16, out=out.data_ptr(), ldo=N)
    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()
    # first launches on both streams before measuring (module load with its fixed scratch,
    # and whatever the driver sets up for a stream's first work)
    B.sgd_kernel_gemm_static_ws(A, W, M, N, K, e, 9, stream=s1.cuda_stream)
    B.sgd_kernel_gemm_static_ws(A, W, M, N, K, e, 9, stream=s2.cuda_stream)
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    for _ in range(3):
        B.sgd_kernel_gemm_static_ws(A, W, M, N, K, e, 9, stream=s1.cuda_stream)
    s1.synchronize()
    assert torch.cuda.mem_get_info()[0] == free0
    B.sgd_kernel_gemm(A, W, M, N, K, e, 9, stream=s2.cuda_stream)
    s2.synchronize()
    assert torch.cuda.mem_get_info()[0] < free0
    assert B.sgd_kernel_status() == 0


@pytest.mark.gpu
def test_static_ws_rejects_a_split_larger_than_its_scratch(B):
    """Forced stream-K on 4096 x 2304 x 4096 needs 136 tiles x 3 segments x 128 KB of
    partials (51 MiB), more than the 32 MiB array: rejected before any launch.  Without
    stream-K (variant 8) the same problem runs and matches the allocating entry."""
    M, N, K = 4096, 2304, 4096
    A, W, h0 = _problem(M, N, K, "f16", 12)
    out = torch.full((M, N), 7.0, dtype=torch.float16, device="cuda")
    e = B.sgd_epilogue_args(kind=B.EPI_F16, out=out.data_ptr(), ldo=N)
    with pytest.raises(B.SgdError) as err:
        B.sgd_kernel_gemm_static_ws(A, W, M, N, K, e, 9)
    assert err.value.code == B.SGD_ERR_SHAPE
    torch.cuda.synchronize()
    assert bool((out == 7.0).all())
    (got,) = _run(B.sgd_kernel_gemm_static_ws, A, W, h0, M, N, K, "f16", 8)
    (ref,) = _run(B.sgd_kernel_gemm, A, W, h0, M, N, K, "f16", 8)
    torch.cuda.synchronize()
    assert torch.equal(got, ref)
    assert B.sgd_kernel_status() == 0


def test_static_ws_validates_on_host():
    """Argument errors are reported before the device is touched (runs without a GPU)."""
    from paper_2609_29505_gb300 import build
    build.build()
    L = binding.lib()
    epi = binding.sgd_epilogue_args(kind=99)
    assert L.sgd_kernel_gemm_static_ws(None, 8, None, 8, 8, 8, 8, C.byref(epi), 0, None) == binding.SGD_ERR_ARG
    epi = binding.sgd_epilogue_args(kind=binding.EPI_F16, out=64, ldo=8)
    assert L.sgd_kernel_gemm_static_ws(64, 12, 64, 12, 8, 8, 12, C.byref(epi), 0, None) == binding.SGD_ERR_SHAPE
    for bad_variant in (2, 4, 13, -1):  # not a variant code
        assert L.sgd_kernel_gemm_static_ws(64, 8, 64, 8, 8, 8, 8, C.byref(epi), bad_variant, None) == binding.SGD_ERR_ARG
