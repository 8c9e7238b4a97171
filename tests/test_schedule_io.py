"""Schedule persistence: a schedule saved with the digest of its weights loads back
identically, refuses other weights or another model, and compiles to the same per-step
patterns (host-only, no GPU)."""
import numpy as np
import pytest
import torch

from paper_2609_29505_gb300 import binding, schedule, synth


@pytest.fixture(scope="module")
def tiny():
    cfg = synth.get_config("tiny")
    w = synth.make_weights(cfg, "cpu")
    return cfg, w, schedule.build_schedule(cfg, w, cfg.T, budget=0.5)


def test_round_trip(tmp_path, tiny):
    cfg, w, sc = tiny
    p = tmp_path / "sched.json"
    schedule.save_schedule(str(p), sc, cfg, w)
    got = schedule.load_schedule(str(p), cfg, w)
    np.testing.assert_array_equal(got["lifetimes"], sc["lifetimes"])
    np.testing.assert_array_equal(got["groups"], sc["groups"])
    assert got["tau"] == sc["tau"] and got["T"] == sc["T"] and got["s_min"] == sc["s_min"]
    assert got["ratio"] == sc["ratio"] and got["ranking"] == "scr" and got["granularity"] == "block"


def test_digest_is_deterministic_and_sees_a_one_bit_change(tiny):
    cfg, w, _ = tiny
    d0 = schedule.weights_digest(w)
    assert schedule.weights_digest(synth.make_weights(cfg, "cpu")) == d0
    for name in sorted(w)[:3] + sorted(w)[-3:]:
        w2 = dict(w)
        t = w[name].clone().contiguous()
        bits = t.view(torch.int16).reshape(-1)
        bits[bits.numel() // 2] ^= 1  # flip one mantissa bit in the middle of the tensor
        w2[name] = t
        assert schedule.weights_digest(w2) != d0, name


def test_load_refuses_other_weights_or_model(tmp_path, tiny):
    cfg, w, sc = tiny
    p = tmp_path / "sched.json"
    schedule.save_schedule(str(p), sc, cfg, w)
    other = dict(w)
    name = sorted(w)[0]
    other[name] = w[name] * 2
    with pytest.raises(ValueError, match="weights differ"):
        schedule.load_schedule(str(p), cfg, other)
    with pytest.raises(ValueError, match="schedule for tiny"):
        schedule.load_schedule(str(p), synth.get_config("dit_small"))
    schedule.save_schedule(str(p), sc, cfg)  # without a digest
    with pytest.raises(ValueError, match="without a weights digest"):
        schedule.load_schedule(str(p), cfg, w)


def test_loaded_schedule_compiles_to_the_same_patterns(tmp_path, tiny):
    cfg, w, sc = tiny
    from paper_2609_29505_gb300 import build
    build.build()
    p = tmp_path / "sched.json"
    schedule.save_schedule(str(p), sc, cfg, w)
    got = schedule.load_schedule(str(p), cfg, w)
    a = binding.sgd_compile_schedule(cfg.T, sc["lifetimes"], sc["groups"])
    b = binding.sgd_compile_schedule(got["T"], got["lifetimes"], got["groups"])
    np.testing.assert_array_equal(a[0], b[0])
    np.testing.assert_array_equal(a[1], b[1])
    assert a[2] == b[2]
