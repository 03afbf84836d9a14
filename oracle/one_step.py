"""CPU oracle for FastVR's one-step restoration update -- TEST INFRASTRUCTURE.

Only the tests, the smoke check and the benchmark may import this module.

Eq. `eq:one_step` (Sec. 3.2, Stage II; the same update is used at inference,
Sec. 4.1): starting from the low-quality latent z_LQ at t = tau, the
restored latent is z_hat = z_LQ - sigma_tau * v, where v is the DiT's
predicted velocity.  Plain float64 NumPy.

parity pins: tests/test_one_step.py -- with the target velocity of Eq.
`eq:target_velocity`, u = (z_LQ - z_HQ) / sigma_tau, the update returns z_HQ;
sigma = 0 and v = 0 are the identity.
"""
import numpy as np


def one_step_update(z_lq: np.ndarray, v: np.ndarray, sigma: float) -> np.ndarray:
    return np.asarray(z_lq, np.float64) - float(sigma) * np.asarray(v, np.float64)
