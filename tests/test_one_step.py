"""The one-step restoration update z_hat = z_LQ - sigma_tau * v (Eq.
`eq:one_step`): pins for the oracle (CPU) and GPU parity through the C ABI."""
import numpy as np
import pytest
import torch

from oracle import one_step as OS


def _rng(seed):
    return np.random.default_rng(seed)


# ------------------------------------------------------------ oracle pins
def test_target_velocity_recovers_the_hq_latent():
    # Eq. `eq:target_velocity`: u = (z_LQ - z_HQ) / sigma_tau; stepping from
    # z_LQ with the target velocity must land on z_HQ (Eq. `eq:trajectory`
    # at t = 0).
    g = _rng(0)
    z_lq, z_hq = g.standard_normal((2, 48, 7, 9))
    for sigma in (0.05, 0.4, 0.9977):
        u = (z_lq - z_hq) / sigma
        assert np.abs(OS.one_step_update(z_lq, u, sigma) - z_hq).max() <= 1e-12


def test_zero_sigma_or_velocity_is_the_identity():
    g = _rng(1)
    z, v = g.standard_normal((2, 1000))
    assert np.array_equal(OS.one_step_update(z, v, 0.0), z)
    assert np.array_equal(OS.one_step_update(z, np.zeros_like(v), 0.7), z)


def test_update_is_linear_in_the_velocity():
    g = _rng(2)
    z, v1, v2 = g.standard_normal((3, 500))
    a = OS.one_step_update(z, v1 + v2, 0.3)
    b = OS.one_step_update(z, v1, 0.3) + OS.one_step_update(z, v2, 0.3) - z
    assert np.abs(a - b).max() <= 1e-12


def test_planted_sign_mistake_fails_the_target_velocity_pin(monkeypatch):
    monkeypatch.setattr(OS, "one_step_update",
                        lambda z, v, s: np.asarray(z) + s * np.asarray(v))
    with pytest.raises(AssertionError):
        test_target_velocity_recovers_the_hq_latent()


# ------------------------------------------------------------- GPU parity
def _bf16_ulps(a: torch.Tensor, b: torch.Tensor) -> torch.Tensor:
    """Distance in bf16 units in the last place (same-sign values)."""
    ia = a.view(torch.int16).to(torch.int32)
    ib = b.view(torch.int16).to(torch.int32)
    return (ia - ib).abs()


@pytest.mark.gpu
@pytest.mark.parametrize("n", [48 * 30 * 68 * 120, 1003, 7])
def test_gpu_bf16_matches_oracle(n):
    from paper_2609_36757_gb300 import fastvr as FV
    g = torch.Generator().manual_seed(n)
    z = torch.randn(n, generator=g).to(torch.bfloat16)
    v = torch.randn(n, generator=g).to(torch.bfloat16)
    sigma = 0.8125
    out = FV.one_step_update(z.cuda(), v.cuda(), sigma).cpu()
    ref = OS.one_step_update(z.double().numpy(), v.double().numpy(),
                             float(np.float32(sigma)))
    ref_bf16 = torch.from_numpy(ref).to(torch.bfloat16)
    ulps = _bf16_ulps(out, ref_bf16)
    # fp32 FMA then one rounding vs the exact value rounded once: equal
    # except where the fp32 result sits on a bf16 rounding boundary
    assert int(ulps.max()) <= 1
    assert (ulps == 0).float().mean().item() >= 0.999


@pytest.mark.gpu
def test_gpu_fp32_latents_and_in_place():
    from paper_2609_36757_gb300 import fastvr as FV
    n = 48 * 3 * 68 * 120 + 5
    g = torch.Generator().manual_seed(3)
    z = torch.randn(n, generator=g)
    v = torch.randn(n, generator=g).to(torch.bfloat16)
    sigma = 0.35
    zd = z.cuda()
    FV.one_step_update(zd, v.cuda(), sigma, out=zd)  # in place
    ref = OS.one_step_update(z.double().numpy(), v.double().numpy(),
                             float(np.float32(sigma)))
    ref32 = torch.from_numpy(ref.astype(np.float32))
    got = zd.cpu()
    exact = (got == ref32).float().mean().item()
    assert exact >= 0.99999
    assert torch.allclose(got, ref32, rtol=2 ** -23, atol=0)


@pytest.mark.gpu
def test_gpu_step_with_target_velocity_lands_on_hq():
    from paper_2609_36757_gb300 import fastvr as FV
    g = torch.Generator().manual_seed(4)
    z_lq = torch.randn(100000, generator=g)
    z_hq = torch.randn(100000, generator=g)
    sigma = 0.5  # exact in binary: u = 2 (z_lq - z_hq) is exact in fp32
    u = ((z_lq - z_hq) / sigma).to(torch.bfloat16)
    out = FV.one_step_update(z_lq.cuda(), u.cuda(), sigma).cpu()
    # only the rounding of u to bf16 separates the result from z_HQ
    bound = (sigma * (u.float() - (z_lq - z_hq) / sigma)).abs() + 1e-6
    assert ((out - z_hq).abs() <= bound * 1.0001 + 1e-6).all()


@pytest.mark.gpu
def test_gpu_chained_updates_on_the_same_stream():
    """Back-to-back launches with no synchronisation: each update reads what
    the kernel queued just before it wrote (the launches overlap their
    set-up with the previous kernel's drain and must still wait for its
    data)."""
    from paper_2609_36757_gb300 import fastvr as FV
    n = 48 * 3 * 68 * 120 + 3
    g = torch.Generator().manual_seed(6)
    z = torch.randn(n, generator=g)
    vs = [torch.randn(n, generator=g).to(torch.bfloat16) for _ in range(4)]
    zd = z.cuda()
    vd = [v.cuda() for v in vs]
    torch.cuda.synchronize()
    sig = [0.5, 0.25, 0.75, 0.125]
    for v, s in zip(vd, sig):
        FV.one_step_update(zd, v, s, out=zd)   # in place, one after another
        zd = zd * 1.0                           # a torch kernel in between
    ref = z.double().numpy()
    for v, s in zip(vs, sig):
        ref = OS.one_step_update(ref.astype(np.float32).astype(np.float64),
                                 v.double().numpy(), float(np.float32(s)))
    got = zd.cpu().double().numpy()
    assert np.abs(got - ref).max() <= 4 * 2.0 ** -23 * np.abs(ref).max() + 1e-6
