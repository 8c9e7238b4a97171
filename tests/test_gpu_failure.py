"""Failure detection on the GPU without a fault: a kernel's bounded wait on an mbarrier that
nothing completes expires after its limit, records a code in the device status word and
returns; the host reads the code (sgd_kernel_status, or SGD_ERR_DEVICE_TIMEOUT from
sgd_check_device) and the context keeps working."""
import math
import time

import numpy as np
import pytest
import torch

from oracle import denoiser as odn
from oracle import trajectory as otj

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def B():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    from paper_2609_29505_gb300 import binding, build
    build.build()
    binding.lib()
    return binding


def _expire_one_wait(B):
    stream = torch.cuda.current_stream().cuda_stream
    t0 = time.time()
    B.check(B.lib().sgd_selftest_wait_timeout(stream), "sgd_selftest_wait_timeout")
    torch.cuda.synchronize()
    return time.time() - t0


def test_expired_wait_sets_the_status_word_and_kernels_still_run(B):
    assert B.sgd_kernel_status() in (0, B.SGD_SELFTEST_TIMEOUT_CODE)  # clears any leftover
    assert B.sgd_kernel_status() == 0
    elapsed = _expire_one_wait(B)
    assert 1.5 < elapsed < 60.0, elapsed            # the 2 s limit, then the kernel returned
    assert B.sgd_kernel_status() == B.SGD_SELFTEST_TIMEOUT_CODE
    assert B.sgd_kernel_status() == 0                 # read once, then cleared
    # the device is still usable: a tcgen05 GEMM against the oracle
    rng = np.random.default_rng(3)
    M, N, K = 300, 520, 688
    A = torch.from_numpy(rng.standard_normal((M, K)).astype(np.float32)).half().cuda()
    W = torch.from_numpy((rng.standard_normal((N, K)) / math.sqrt(K)).astype(np.float32)).half().cuda()
    out = torch.empty(M, N, dtype=torch.float16, device="cuda")
    B.sgd_kernel_gemm(A, W, M, N, K, B.sgd_epilogue_args(kind=B.EPI_F16, out=out.data_ptr(), ldo=N))
    torch.cuda.synchronize()
    want = odn.linear(A.float().cpu().numpy(), W.float().cpu().numpy())
    got = out.float().cpu().numpy()
    assert np.linalg.norm(got - want) / np.linalg.norm(want) < 2e-3
    assert B.sgd_kernel_status() == 0


def test_check_device_reports_the_timeout_and_the_trajectory_continues(B):
    from test_gpu_parity import Case
    c = Case("tiny", 0.5)
    m = c.model(B)
    out = c.out_buffer()
    x = torch.from_numpy(c.inp.z0.numpy()).cuda()
    m.step(x, out, otj.timestep(c.T, 1), 1)
    _expire_one_wait(B)
    with pytest.raises(B.SgdError) as err:
        m.check_device()
    assert err.value.code == B.SGD_ERR_DEVICE_TIMEOUT
    m.check_device()  # the word was cleared by the report
    # a fresh trajectory on the same context still matches the oracle's first step
    m.reset()
    m.step(x, out, otj.timestep(c.T, 1), 1)
    m.check_device()
    ref = otj.run(c.cfg, c.W, c.sched["lifetimes"], c.T, z0=c.inp.z0.numpy(), steps=1)
    got = out.float().cpu().numpy()
    assert np.linalg.norm(got - ref["outputs"][0]) / np.linalg.norm(ref["outputs"][0]) < 5e-3
    m.close()
