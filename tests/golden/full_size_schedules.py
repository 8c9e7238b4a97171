"""Writes and reads ``full_size_schedules.json``: the oracle's schedule for every full-size synthetic
model, so that tests and the benchmark's CPU arms can compare against it without
re-running float64 spectra of 16 GB of weights on host cores (tens of minutes for the
LLaDA-8B-shaped model).

For each model (synth.CONFIGS minus tiny, whose oracle schedule takes a second), the
weights are generated exactly as the tests and the benchmark generate them (synth, on a
CUDA device), identified by synth.weights_checksum, and scored by ``oracle.spectral``
alone (float64 Gram eigenvalues, Sec. 3.2 Eq. scr-reg; App. G scores).  Stored per model:
the checksum, the branch scores (App. G, graph order) and the lifetimes of Algorithm 1
(Eq. schedule, block and branch granularity) for each horizon of the model and each
budget in synth.BUDGETS.  Nothing here calls the CUDA library.

``oracle_lifetimes`` returns the stored lifetimes when the weights' checksum matches the
stored one (the same bytes were scored), and otherwise scores the given weights with
``oracle.spectral`` on the spot.

Usage (needs a CUDA device for the weight generator):
    python tests/golden/full_size_schedules.py [model ...]
"""
from __future__ import annotations

import json
import os
import sys
import time

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(os.path.dirname(HERE))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

OUT = os.path.join(HERE, "full_size_schedules.json")
MODELS = ["dit", "uvit", "sdxl", "llada"]
SCORED = ("w_qkv", "w_o", "wx_q", "wx_kv", "wx_o", "w_1", "w_2")


class Float64View:
    """Read-only mapping name -> float64 host copy of one weight, made on first use and
    not kept, so that only the matrices of the block being scored are on the host."""

    def __init__(self, weights):
        self.w = weights

    def __getitem__(self, name):
        import numpy as np
        t = self.w[name]
        if isinstance(t, np.ndarray):
            return t.astype(np.float64)
        return t.double().cpu().numpy()


def schedule_key(T: int, budget: float, granularity: str) -> str:
    return f"T={T} budget={budget:g} {granularity}"


def oracle_entry(cfg, weights, log=print):
    from oracle import spectral as osp
    from paper_2609_29505_gb300 import synth

    t0 = time.time()
    bq = osp.branch_scores(cfg, Float64View(weights))
    log(f"{cfg.name}: branch scores in {time.time() - t0:.0f} s")
    entry = {"checksum": synth.weights_checksum(weights), "eta": osp.ETA,
             "branch_scores": [float(x) for x in bq], "lifetimes": {}, "ratio": {}}
    for T in cfg.horizons:
        for budget in synth.BUDGETS:
            for gran, groups in (("block", synth.block_groups(cfg)), ("branch", synth.branch_groups(cfg))):
                sc = osp.schedule(cfg, None, T, budget, groups, branch_q=bq)
                key = schedule_key(T, budget, gran)
                entry["lifetimes"][key] = [int(x) for x in sc["lifetimes"]]
                entry["ratio"][key] = float(sc["ratio"])
    return entry


# models that share another model's weights (same seed and shapes)
ALIASES = {"llada_4k": "llada"}


def load():
    if not os.path.exists(OUT):
        return {}
    with open(OUT) as f:
        return json.load(f)


def oracle_lifetimes(cfg, weights, T: int, budget: float, granularity: str = "block",
                     stored=None):
    """(per-unit lifetimes from oracle.spectral, "stored" | "computed") for ``weights``."""
    import numpy as np

    from oracle import spectral as osp
    from paper_2609_29505_gb300 import synth

    doc = load() if stored is None else stored
    entry = doc.get(ALIASES.get(cfg.name, cfg.name))
    key = schedule_key(T, budget, granularity)
    if entry and key in entry["lifetimes"] and entry["checksum"] == synth.weights_checksum(weights):
        return np.asarray(entry["lifetimes"][key], dtype=np.int64), "stored"
    groups = synth.block_groups(cfg) if granularity == "block" else synth.branch_groups(cfg)
    sc = osp.schedule(cfg, Float64View(weights), T, budget, groups)
    return np.asarray(sc["lifetimes"], dtype=np.int64), "computed"


def main(names):
    import torch

    from paper_2609_29505_gb300 import synth

    if not torch.cuda.is_available():
        raise SystemExit("the full-size weights are generated on a CUDA device")
    doc = {}
    if os.path.exists(OUT):
        with open(OUT) as f:
            doc = json.load(f)
    doc["_about"] = ("oracle.spectral (float64) scores and Algorithm 1 lifetimes of the "
                     "full-size synthetic models; written by full_size_schedules.py; "
                     f"torch {torch.__version__}")
    for name in names:
        cfg = synth.get_config(name)
        w = synth.make_weights(cfg, "cuda")
        torch.cuda.synchronize()
        doc[name] = oracle_entry(cfg, w)
        del w
        torch.cuda.empty_cache()
        with open(OUT, "w") as f:
            json.dump(doc, f, indent=1, sort_keys=True)
    print(OUT)


if __name__ == "__main__":
    main(sys.argv[1:] or MODELS)
