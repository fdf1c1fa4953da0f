"""Learning-rate correction factor of RelaySGD (appendix "Learning-rate
correction for RelaySGD").

Under the robust rebuild, an update spreads uniformly but not in full: if
every worker starts from a scalar model 0 and applies one update of +1, and
RelaySGD then runs with no further updates, the models converge to a value
alpha_n < 1 that depends only on the topology (under Algorithm 1's division
by nbar nothing is lost and the value is 1).  A learning rate tuned for
all-reduce SGD is then scaled by 1 / alpha_n.  This helper runs that
procedure through the library on the GPU (one coordinate quad), nothing else.
"""
from __future__ import annotations

import numpy as np

from . import _native as nat


def lr_correction(n: int, edges, mode: int = 1, tol: float = 1e-7, max_steps: int = 100_000,
                  device="cuda"):
    """Returns (alpha_n, the per-worker limits [n]) for the given tree.
    Raises RuntimeError if the models still move by more than `tol` after
    `max_steps` steps (the limit was not reached)."""
    import torch
    run = nat.RelayRun(n, 4, edges, device=device, mode=mode)
    run.init(0.0, 0, np.zeros((n, 1), np.float32), 0.0, 0, 0.0)   # x^0 = 0
    run.mu.fill_(1.0)                                             # one update of +1:
    run.step(1.0, 0)                                              # x - 1 (x - mu) = 1
    prev = run.x[:, 0].clone()
    converged = False
    for k in range(max_steps):
        run.step(0.0, 0)                                          # no further updates
        if k % 64 == 63:
            cur = run.x[:, 0].clone()
            if float((cur - prev).abs().max()) <= tol:
                converged = True
                break
            prev = cur
    if not converged:
        raise RuntimeError(f"lr_correction: models still moving by more than {tol} after {max_steps} steps")
    torch.cuda.synchronize(run.device)
    limits = run.x[:, 0].double().cpu().numpy()
    return float(limits.mean()), limits
