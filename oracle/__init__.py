"""CPU oracle for Urgency-Aware Denoising (UAD) -- TEST INFRASTRUCTURE ONLY.

A plain, slow, fp64 numpy restatement of what the CUDA path computes, written from the
paper and sharing no code with the CUDA path. Only ``tests/``, ``__graft_entry__.smoke()``
and ``bench.py``'s cpu_baseline / ``--impl reference`` legs may import it; the product
library never calls it and has no CPU fallback.

Modules
  plan.py   per-token step budgets -> per-step flow times and Euler steps (Sec. 4.2, Eqs. 4-5;
            Sec. 4.3, Eq. 7)
  uad.py    the denoising loop: Euler integration (Eqs. 1-2), UAER early release (Sec. 4.2),
            Trajectory Reconciliation (Eqs. 6-7), ghost actions, Ghost Action Correction
            (Eqs. 8-9); takes the velocity field as a callable
  model.py  the synthetic action expert F_theta (Eq. 1) with per-action time conditioning
            (App. C.1); its composition is this project's stated architecture, not the
            paper's (the paper fixes none) -- parity unpinned beyond its components,
            structural invariants and closed-form special cases
  so3.py    rotation vectors and Ghost Action Correction by composition on SO(3) (App. C.1)
  clock.py  action availability latency under the control-time alignment clock
            (Sec. 5.1 Metrics, App. C.3) and the latency model (App. B, Eqs. 11-12)
"""
