"""CPU oracle for spectral-guided static layer scheduling — TEST INFRASTRUCTURE ONLY.

A plain, slow, obviously-correct NumPy implementation of what the scheduled
denoiser path computes, written from the paper ("Spectral-Guided Diffusion:
Accelerating Inference via Static Spectral Layer Scheduling"):

* ``oracle.spectral``  — SCR_eta (Sec. 3.2, Eq. scr-reg), the matrix score g(W)
  (App. G, Eq. app-matrix-score), branch scores (Eqs. app-attn-score,
  app-xattn-score, app-mlp-score), unit aggregation and normalisation
  (Eqs. app-block-score, app-score-normalization), lifetimes (Sec. 4.1,
  Eq. schedule, Algorithm 1) and the per-step active sets.
* ``oracle.denoiser``  — the residual-unit semantics of Sec. 3.1 executed as in
  Algorithm 2 (jagged-stream execution): active units compute their branch
  update, store it and add it; frozen units add the stored update to the
  current residual stream.  FP32 activations, float64 spectra.
* ``oracle.trajectory`` — the deterministic sampler of Sec. 3.1 around it.

Only ``tests/``, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` /
``--impl reference`` legs of ``bench.py`` may import this package.  It shares
no code with the CUDA path and never imports it.

Parity status: every function is pinned by ``tests/test_oracle_*.py`` against
closed forms, invariants, special cases and brute force.  The block
architectures (norms, attention, MLP variants) are not specified by the paper;
they follow textbook definitions and are pinned by textbook special cases.
"""
