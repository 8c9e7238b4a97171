"""End-to-end parity of the scheduled denoiser step on the GPU (through the C ABI)
against the CPU oracle, for every architecture family at reduced size and for
three layer-step budgets.

* active sets: bit-exact against the oracle's A_s = {u : s <= S_u};
* per step (teacher forced: the GPU evaluates the oracle's state z_s, its caches
  are its own): relative L2 of eps_s <= 5e-3;
* closed loop (the GPU integrates its own states with the library's sampler
  update): relative L2 of the final state and of the last eps <= 1e-2.
"""
import os

import numpy as np
import pytest
import torch

from oracle import denoiser as odn
from oracle import spectral as osp
from oracle import trajectory as otj
from paper_2609_29505_gb300 import schedule, synth

pytestmark = pytest.mark.gpu

# SGD_TEST_SIMT=1 runs every GEMM of the model on the SIMT reference kernel (debugging aid)
FLAGS = 1 if os.environ.get("SGD_TEST_SIMT") == "1" else 0
STEP_TOL = 5e-3
FINAL_TOL = 1e-2
SMALL = ["tiny", "dit_small", "uvit_small", "sdxl_small", "llada_small"]


@pytest.fixture(scope="module")
def B():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    from paper_2609_29505_gb300 import binding, build
    build.build()
    binding.lib()
    return binding


def rel(a, b):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return float(np.linalg.norm(a - b) / np.linalg.norm(b))


def oracle_schedule(cfg, w_cpu, T, budget, granularity="block"):
    """Algorithm 1 by the oracle (float64 spectra of the same bf16 weights)."""
    W64 = {k: v.double().numpy() for k, v in w_cpu.items()}
    groups = synth.block_groups(cfg) if granularity == "block" else synth.branch_groups(cfg)
    return osp.schedule(cfg, W64, T, budget, groups)


class Case:
    """One small model at one budget: the product's schedule must equal the oracle's
    (integer lifetimes); the oracle trajectory runs on the oracle's own lifetimes."""

    def __init__(self, name, budget, flags=0, granularity="block"):
        self.cfg = cfg = synth.get_config(name)
        self.T = cfg.T
        self.w_cpu = synth.make_weights(cfg, "cpu")
        self.inp = synth.make_inputs(cfg, "cpu")
        self.W = odn.to_numpy_weights(self.w_cpu)
        self.sched = schedule.build_schedule(cfg, self.w_cpu, self.T, budget=budget,
                                             granularity=granularity)
        self.osched = oracle_schedule(cfg, self.w_cpu, self.T, budget, granularity)
        np.testing.assert_array_equal(self.sched["lifetimes"], self.osched["lifetimes"])
        self.w_dev = {k: v.cuda() for k, v in self.w_cpu.items()}
        self.cls = None if self.inp.class_ids is None else self.inp.class_ids.cuda()
        self.ctx = None if self.inp.ctx is None else self.inp.ctx.cuda()
        self.flags = flags

    def ids_at(self, s):
        return synth.token_ids_at(self.cfg, self.inp, s, self.T)

    def oracle(self):
        cfg = self.cfg
        return otj.run(cfg, self.W, self.osched["lifetimes"], self.T,
                       z0=None if self.inp.z0 is None else self.inp.z0.numpy(),
                       class_ids=None if self.inp.class_ids is None else self.inp.class_ids.numpy(),
                       ctx=None if self.inp.ctx is None else self.inp.ctx.float().numpy(),
                       ids_at=(lambda s: self.ids_at(s).numpy()) if cfg.stem == "embed" else None)

    def model(self, B):
        m = B.Denoiser(self.cfg, self.w_dev, flags=self.flags)
        m.set_schedule(self.T, self.sched["lifetimes"], self.sched["groups"])
        return m

    def out_buffer(self):
        cfg = self.cfg
        if cfg.head == "logits":
            return torch.empty(cfg.batch, cfg.n_tokens, cfg.d_out, dtype=torch.float16, device="cuda")
        if cfg.head == "identity":
            return torch.empty(cfg.batch, cfg.n_tokens, cfg.d, device="cuda")
        return torch.empty(cfg.batch, cfg.n_out_tokens, cfg.out_channels, device="cuda")


_cases = {}


def case(name, budget, granularity="block"):
    key = (name, budget, granularity)
    if key not in _cases:
        c = Case(name, budget, FLAGS, granularity)
        c.ref = c.oracle()
        _cases[key] = c
    return _cases[key]


@pytest.mark.parametrize("budget", [1.0, 0.5, 0.33])
@pytest.mark.parametrize("name", SMALL)
def test_active_sets_and_teacher_forced_steps(B, name, budget):
    c = case(name, budget)
    m = c.model(B)
    want_masks = osp.active_sets(c.osched["lifetimes"], c.T)
    out = c.out_buffer()
    errs = []
    for s in range(1, c.T + 1):
        np.testing.assert_array_equal(m.active_mask(s), want_masks[s - 1])
        x = c.ids_at(s).cuda() if c.cfg.stem == "embed" else torch.from_numpy(c.ref["states"][s - 1]).cuda()
        m.step(x, out, otj.timestep(c.T, s), s, class_ids=c.cls, ctx=c.ctx)
        errs.append(rel(out.float().cpu().numpy(), c.ref["outputs"][s - 1]))
    m.check_device()
    info = m.info()
    m.close()
    assert info["layer_steps"] == int(np.sum(c.sched["lifetimes"]))
    assert max(errs) <= STEP_TOL, f"per-step rel L2 {['%.2e' % e for e in errs]}"


@pytest.mark.parametrize("budget", [1.0, 0.5])
@pytest.mark.parametrize("name", ["tiny", "dit_small", "uvit_small", "sdxl_small"])
def test_closed_loop_final_state(B, name, budget):
    c = case(name, budget)
    m = c.model(B)
    out = c.out_buffer()
    z = c.inp.z0.clone().cuda()
    for s in range(1, c.T + 1):
        m.step(z, out, otj.timestep(c.T, s), s, class_ids=c.cls, ctx=c.ctx)
        B.sgd_sampler_update(z, out, 1.0, 1.0 / c.T)
    torch.cuda.synchronize()
    m.close()
    assert rel(z.cpu().numpy(), c.ref["states"][-1]) <= FINAL_TOL
    assert rel(out.cpu().numpy(), c.ref["outputs"][-1]) <= FINAL_TOL


def test_graph_replay_equals_profiled_eager_launches(B):
    c = case("dit_small", 0.5)
    outs = []
    for mode in ("graph", "profile"):
        m = c.model(B)
        out = c.out_buffer()
        z = torch.from_numpy(c.ref["states"][0]).cuda()
        res = []
        for s in range(1, c.T + 1):
            if mode == "graph":
                m.step(z, out, otj.timestep(c.T, s), s, class_ids=c.cls)
            else:
                recs = m.profile_step(z, out, otj.timestep(c.T, s), s, class_ids=c.cls)
                assert recs and all(r["ms"] >= 0 for r in recs)
            res.append(out.cpu().clone())
        m.close()
        outs.append(res)
    for a, b in zip(*outs):
        assert torch.equal(a, b)


def test_host_buffer_step_equals_device_step(B):
    c = case("uvit_small", 0.5)
    m = c.model(B)
    out_d = c.out_buffer()
    out_h = torch.empty(out_d.shape, dtype=out_d.dtype).pin_memory()
    cls_h = c.inp.class_ids.clone().pin_memory()
    for s in range(1, 4):
        z = torch.from_numpy(c.ref["states"][s - 1])
        m.step(z.cuda(), out_d, otj.timestep(c.T, s), s, class_ids=c.cls)
        torch.cuda.synchronize()
        a = out_d.cpu()
    m.reset()
    for s in range(1, 4):
        z = torch.from_numpy(c.ref["states"][s - 1]).pin_memory()
        m.step_host(z, out_h, otj.timestep(c.T, s), s, class_ids_host=cls_h)
    assert torch.equal(out_h, a)
    m.close()


def test_step_order_and_state_errors(B):
    c = case("tiny", 0.5)
    m = B.Denoiser(c.cfg, c.w_dev)
    out = c.out_buffer()
    z = c.inp.z0.clone().cuda()
    with pytest.raises(B.SgdError) as e:
        m.step(z, out, 1.0, 1)
    assert e.value.code == B.SGD_ERR_STATE
    m.set_schedule(c.T, c.sched["lifetimes"], c.sched["groups"])
    with pytest.raises(B.SgdError) as e:
        m.step(z, out, 1.0, 2)
    assert e.value.code == B.SGD_ERR_CACHE_INVALID
    m.step(z, out, 1.0, 1)
    with pytest.raises(B.SgdError) as e:
        m.step(z, out, 1.0, 3)
    assert e.value.code == B.SGD_ERR_CACHE_INVALID
    m.step(z, out, 1.0, 2)
    m.reset()
    with pytest.raises(B.SgdError) as e:
        m.step(z, out, 1.0, 3)
    assert e.value.code == B.SGD_ERR_CACHE_INVALID
    bad = np.array(c.sched["lifetimes"]).copy()
    bad[0] = bad[1] + 1 if bad[1] < c.T else bad[1] - 1
    with pytest.raises(B.SgdError) as e:
        m.set_schedule(c.T, bad, c.sched["groups"])
    assert e.value.code == B.SGD_ERR_SCHEDULE
    m.check_device()
    m.close()


@pytest.mark.parametrize("name", ["llada_small", "uvit_small", "sdxl_small", "dit_small"])
def test_execution_modes_against_oracle(B, name):
    """Every execution mode of Table tab:kernel -- jagged graphs, eager op-by-op launches
    (host-side skipping) and padded graphs (frozen branches evaluated and discarded) --
    matches the oracle teacher forced (per-step relative L2 <= 5e-3), and the three give
    the same outputs bit for bit."""
    c = case(name, 0.5)
    results = {}
    for mode in (B.EXEC_JAGGED_GRAPH, B.EXEC_EAGER, B.EXEC_PADDED_GRAPH):
        m = c.model(B)
        m.set_exec_mode(mode)
        out = c.out_buffer()
        res, errs = [], []
        for s in range(1, c.T + 1):
            x = c.ids_at(s).cuda() if c.cfg.stem == "embed" else torch.from_numpy(c.ref["states"][s - 1]).cuda()
            m.step(x, out, otj.timestep(c.T, s), s, class_ids=c.cls, ctx=c.ctx)
            res.append(out.cpu().clone())
            errs.append(rel(res[-1].float().numpy(), c.ref["outputs"][s - 1]))
        m.check_device()
        m.close()
        results[mode] = res
        assert max(errs) <= STEP_TOL, f"mode {mode}: per-step rel L2 {['%.2e' % e for e in errs]}"
    for mode in (B.EXEC_EAGER, B.EXEC_PADDED_GRAPH):
        for a, b in zip(results[B.EXEC_JAGGED_GRAPH], results[mode]):
            assert torch.equal(a, b)


@pytest.mark.parametrize("budget", [0.5, 0.33])
@pytest.mark.parametrize("name", ["llada_small", "dit_small", "sdxl_small"])
def test_branch_granularity_against_oracle(B, name, budget):
    """Branch granularity (every branch its own atomic group, so an attention branch can be
    frozen while its block's MLP still runs, App. G): lifetimes equal to the oracle's,
    bit-exact active sets, per-step relative L2 <= 5e-3 teacher forced."""
    c = case(name, budget, "branch")
    S = np.asarray(c.osched["lifetimes"])
    nb = len(c.cfg.branches)
    assert any(len(set(S[b * nb:(b + 1) * nb])) > 1 for b in range(c.cfg.n_blocks)), \
        "schedule has no block with branches of different lifetimes"
    m = c.model(B)
    want_masks = osp.active_sets(S, c.T)
    out = c.out_buffer()
    errs = []
    for s in range(1, c.T + 1):
        np.testing.assert_array_equal(m.active_mask(s), want_masks[s - 1])
        x = c.ids_at(s).cuda() if c.cfg.stem == "embed" else torch.from_numpy(c.ref["states"][s - 1]).cuda()
        m.step(x, out, otj.timestep(c.T, s), s, class_ids=c.cls, ctx=c.ctx)
        errs.append(rel(out.float().cpu().numpy(), c.ref["outputs"][s - 1]))
    m.check_device()
    m.close()
    assert max(errs) <= STEP_TOL, f"per-step rel L2 {['%.2e' % e for e in errs]}"


@pytest.mark.parametrize("name", ["llada_small", "sdxl_small"])
def test_mma_sync_attention_path_within_parity(B, name):
    """The same model with every attention on the mma.sync kernel stays within parity."""
    c = case(name, 0.5)
    m = B.Denoiser(c.cfg, c.w_dev, flags=B.FLAG_MMA_SYNC_ATTENTION)
    m.set_schedule(c.T, c.sched["lifetimes"], c.sched["groups"])
    out = c.out_buffer()
    for s in range(1, c.T + 1):
        x = c.ids_at(s).cuda() if c.cfg.stem == "embed" else torch.from_numpy(c.ref["states"][s - 1]).cuda()
        m.step(x, out, otj.timestep(c.T, s), s, class_ids=c.cls, ctx=c.ctx)
        assert rel(out.float().cpu().numpy(), c.ref["outputs"][s - 1]) <= STEP_TOL
    m.close()


@pytest.mark.parametrize("pinned", [True, False], ids=["pinned-direct", "pageable-copy"])
def test_async_host_steps_equal_device_steps(B, pinned):
    """Queued host-buffer steps return the same bytes as device steps once sgd_host_wait
    has returned: pinned outputs written by the step's kernels over the host link, pageable
    ones through the double-buffered device output and the copy stream."""
    c = case("llada_small", 0.5)
    m = c.model(B)
    out_d = c.out_buffer()
    want = []
    for s in range(1, c.T + 1):
        m.step(c.ids_at(s).cuda(), out_d, otj.timestep(c.T, s), s)
        want.append(out_d.cpu().clone())
    m.reset()
    outs = [torch.empty(out_d.shape, dtype=out_d.dtype) for _ in range(c.T)]
    if pinned:
        outs = [o.pin_memory() for o in outs]
    ins = [c.ids_at(s).pin_memory() for s in range(1, c.T + 1)]
    for s in range(1, c.T + 1):
        m.step_host_async(ins[s - 1], outs[s - 1], otj.timestep(c.T, s), s)
    m.host_wait()
    for a, b in zip(outs, want):
        assert torch.equal(a, b)
    m.close()


def test_long_context_4096_tokens(B):
    """LLaDA-structured model on one 4096-token sequence (32 key tiles per query tile,
    RoPE over 4096 positions): bit-exact active sets, per-step relative L2 <= 5e-3."""
    cfg = synth.get_config("llada_small").with_(name="llada_small_4k", batch=1, n_tokens=4096,
                                                T=4, horizons=[4])
    w_cpu = synth.make_weights(cfg, "cpu")
    inp = synth.make_inputs(cfg, "cpu")
    W = odn.to_numpy_weights(w_cpu)
    sched = schedule.build_schedule(cfg, w_cpu, cfg.T, budget=0.5)
    osched = oracle_schedule(cfg, w_cpu, cfg.T, 0.5)
    np.testing.assert_array_equal(sched["lifetimes"], osched["lifetimes"])
    ref = otj.run(cfg, W, osched["lifetimes"], cfg.T,
                  ids_at=lambda s: synth.token_ids_at(cfg, inp, s).numpy())
    m = B.Denoiser(cfg, {k: v.cuda() for k, v in w_cpu.items()})
    m.set_schedule(cfg.T, sched["lifetimes"], sched["groups"])
    masks = osp.active_sets(osched["lifetimes"], cfg.T)
    out = torch.empty(1, cfg.n_tokens, cfg.d_out, dtype=torch.float16, device="cuda")
    for s in range(1, cfg.T + 1):
        np.testing.assert_array_equal(m.active_mask(s), masks[s - 1])
        m.step(synth.token_ids_at(cfg, inp, s).cuda(), out, otj.timestep(cfg.T, s), s)
        assert rel(out.float().cpu().numpy(), ref["outputs"][s - 1]) <= STEP_TOL
    m.check_device()
    m.close()


@pytest.mark.parametrize("name", ["dit_small", "llada_small", "uvit_small", "sdxl_small"])
def test_programmatic_dependent_launch_is_bit_identical(B, name):
    """Step programs launched with programmatic dependent launch (SGD_FLAG_PDL: each kernel's
    launch and prologue overlapping its predecessor's tail, in graphs and eagerly) give the
    same bits as fully serialised launches."""
    c = case(name, 0.5)
    results = []
    for flags, mode in ((0, B.EXEC_JAGGED_GRAPH), (B.FLAG_PDL, B.EXEC_JAGGED_GRAPH),
                        (B.FLAG_PDL, B.EXEC_EAGER)):
        m = B.Denoiser(c.cfg, c.w_dev, flags=flags)
        m.set_schedule(c.T, c.sched["lifetimes"], c.sched["groups"])
        m.set_exec_mode(mode)
        out = c.out_buffer()
        res = []
        for s in range(1, c.T + 1):
            x = c.ids_at(s).cuda() if c.cfg.stem == "embed" else torch.from_numpy(c.ref["states"][s - 1]).cuda()
            m.step(x, out, otj.timestep(c.T, s), s, class_ids=c.cls, ctx=c.ctx)
            res.append(out.cpu().clone())
        m.check_device()
        m.close()
        results.append(res)
    for other in results[1:]:
        for a, b in zip(results[0], other):
            assert torch.equal(a, b)


@pytest.mark.parametrize("budget", [1.0, 0.5])
@pytest.mark.parametrize("name", ["tiny", "uvit_small", "sdxl_small", "llada_small"])
def test_folded_norm_path_against_oracle(B, name, budget):
    """The pre-norm folded into the GEMMs (SGD_FLAG_FOLD_NORM; RMSNorm and LayerNorm models):
    bit-exact active sets and per-step relative L2 <= 5e-3 teacher forced, under jagged graphs,
    eager launches and padded graphs (which give the same bits), and the closed-loop final
    state within 1e-2."""
    c = case(name, budget)
    want_masks = osp.active_sets(c.osched["lifetimes"], c.T)
    results = {}
    for mode in (B.EXEC_JAGGED_GRAPH, B.EXEC_EAGER, B.EXEC_PADDED_GRAPH):
        m = B.Denoiser(c.cfg, c.w_dev, flags=B.FLAG_FOLD_NORM)
        m.set_schedule(c.T, c.sched["lifetimes"], c.sched["groups"])
        m.set_exec_mode(mode)
        out = c.out_buffer()
        res, errs = [], []
        for s in range(1, c.T + 1):
            np.testing.assert_array_equal(m.active_mask(s), want_masks[s - 1])
            x = c.ids_at(s).cuda() if c.cfg.stem == "embed" else torch.from_numpy(c.ref["states"][s - 1]).cuda()
            m.step(x, out, otj.timestep(c.T, s), s, class_ids=c.cls, ctx=c.ctx)
            res.append(out.cpu().clone())
            errs.append(rel(res[-1].float().numpy(), c.ref["outputs"][s - 1]))
        m.check_device()
        m.close()
        results[mode] = res
        assert max(errs) <= STEP_TOL, f"mode {mode}: per-step rel L2 {['%.2e' % e for e in errs]}"
    for mode in (B.EXEC_EAGER, B.EXEC_PADDED_GRAPH):
        for a, b in zip(results[B.EXEC_JAGGED_GRAPH], results[mode]):
            assert torch.equal(a, b)
    if c.cfg.stem != "embed":
        m = B.Denoiser(c.cfg, c.w_dev, flags=B.FLAG_FOLD_NORM)
        m.set_schedule(c.T, c.sched["lifetimes"], c.sched["groups"])
        out = c.out_buffer()
        z = c.inp.z0.clone().cuda()
        for s in range(1, c.T + 1):
            m.step(z, out, otj.timestep(c.T, s), s, class_ids=c.cls, ctx=c.ctx)
            B.sgd_sampler_update(z, out, 1.0, 1.0 / c.T)
        torch.cuda.synchronize()
        m.close()
        assert rel(z.cpu().numpy(), c.ref["states"][-1]) <= FINAL_TOL
