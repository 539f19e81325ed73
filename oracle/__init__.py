"""Float64 CPU oracle for the JAGG backward path.

TEST INFRASTRUCTURE ONLY.  Only `tests/`, `__graft_entry__.smoke()` and the
`cpu_baseline` / `--impl reference` legs of `bench.py` may import anything here.  The
product path (`paper_2607_17572_gb300`) never imports this package, and this package
imports nothing from the product.  The two share only the seeded inputs of `synth`.

Contents (each function cites the passage of the paper it follows):
  dit.py              DiT / MMDiT forward and hand-derived reverse mode (the pinned
                      backbone; the paper uses Flux and Qwen-Image off the shelf and does
                      not describe them, so the architecture is a stated reading)
  grpo.py             Eq. advantage, Eq. logprob, Eq. grpo_loss, Phase 2 signals,
                      Eq. alpha / Eq. s_base_corr aggregation, jagg_frac routing,
                      cosine / norm-ratio reductions
  linear_velocity.py  a velocity model linear in (z, t) for the exactness theorem
  rollout.py          one sampler step (flow Euler-Maruyama or stochastic DDIM) with the
                      log-prob of its sample; the flow-SDE rollout built from it
  path.py             JAGG and full per-step window gradients (Algorithm 1)

Every function computes in float64 with numpy; library matmuls are the only primitives.
Parity status: every function is pinned by a `-m "not gpu"` test in tests/test_oracle_*.py
(finite differences, library routines, closed forms, the exactness theorem); the one
quantity left unpinned is the cosine table of real Flux/Qwen-Image rollouts, which needs
trained weights ("parity unpinned").
"""
