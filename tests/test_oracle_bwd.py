"""Pins for the oracle's backward (gradients of the one-shot chunk-causal
attention): torch autograd through library attention (SDPA in float64 with
the Eq. 1 mask, whose construction is itself pinned by the hand-evaluated
masks), central finite differences of the oracle's own forward on tiny
inputs, and planted mistakes that must fail."""
import numpy as np
import pytest
import torch

from oracle import attention as A


def _rand(shape, seed, scale=1.0):
    g = np.random.default_rng(seed)
    return torch.from_numpy(g.standard_normal(shape) * scale).to(
        torch.bfloat16).double().numpy()


def _torch_grads(q, k, v, do, N, kf, W, scale):
    B, L, H, d = q.shape
    mask = torch.from_numpy(A.token_mask(L // N, N, kf, W))
    tq, tk, tv = (torch.from_numpy(x).permute(0, 2, 1, 3).clone().requires_grad_()
                  for x in (q, k, v))
    o = torch.nn.functional.scaled_dot_product_attention(
        tq, tk, tv, attn_mask=mask, scale=scale)
    o.backward(torch.from_numpy(do).permute(0, 2, 1, 3))
    return [t.grad.permute(0, 2, 1, 3).numpy() for t in (tq, tk, tv)]


CASES = [(1, 2, 8, 3, 2, 5, 1), (2, 1, 4, 2, 3, 7, -1), (1, 1, 6, 4, 1, 6, 0),
         (1, 2, 8, 1, 1, 12, -1), (1, 1, 4, 5, 2, 6, 2)]


@pytest.mark.parametrize("case", CASES)
def test_backward_matches_torch_autograd_through_sdpa(case):
    B, H, d, N, kf, T, W = case
    L = N * T
    q, k, v, do = (_rand((B, L, H, d), s) for s in (1, 2, 3, 4))
    got = A.blockcausal_attention_bwd(q, k, v, do, N, kf, W, d ** -0.5)
    want = _torch_grads(q, k, v, do, N, kf, W, d ** -0.5)
    for g, w in zip(got, want):
        assert np.abs(g - w).max() <= 1e-12


def test_backward_matches_finite_differences():
    B, H, d, N, kf, T, W = 1, 1, 3, 2, 2, 4, 1
    L = N * T
    q, k, v, do = (_rand((B, L, H, d), s) for s in (5, 6, 7, 8))
    scale = 0.7
    grads = A.blockcausal_attention_bwd(q, k, v, do, N, kf, W, scale)

    def loss(q_, k_, v_):
        o, _ = A.blockcausal_attention(q_, k_, v_, N, kf, W, scale)
        return float((o * do).sum())

    eps = 1e-6
    for which, g in enumerate(grads):
        for idx in [(0, 0, 0, 0), (0, 3, 0, 1), (0, L - 1, 0, 2), (0, 5, 0, 0)]:
            args = [q.copy(), k.copy(), v.copy()]
            args[which][idx] += eps
            up = loss(*args)
            args[which][idx] -= 2 * eps
            dn = loss(*args)
            assert abs((up - dn) / (2 * eps) - g[idx]) <= 1e-7


def _mutant_no_delta(q, k, v, do, N, kf, W, scale):
    B, L, H, d = q.shape
    mask = A.token_mask(L // N, N, kf, W)
    dq, dk, dv = (np.zeros_like(x) for x in (q, k, v))
    for b in range(B):
        for h in range(H):
            p = A.softmax_rows(q[b, :, h], k[b, :, h], scale, mask)
            dv[b, :, h] = p.T @ do[b, :, h]
            ds = p * (do[b, :, h] @ v[b, :, h].T)  # the row term is dropped
            dq[b, :, h] = scale * ds @ k[b, :, h]
            dk[b, :, h] = scale * ds.T @ q[b, :, h]
    return dq, dk, dv


def _mutant_transposed_dv(q, k, v, do, N, kf, W, scale):
    dq, dk, dv = _ORIG(q, k, v, do, N, kf, W, scale)
    B, L, H, d = q.shape
    mask = A.token_mask(L // N, N, kf, W)
    for b in range(B):
        for h in range(H):
            p = A.softmax_rows(q[b, :, h], k[b, :, h], scale, mask)
            dv[b, :, h] = p @ do[b, :, h]  # p instead of p^T
    return dq, dk, dv


_ORIG = A.blockcausal_attention_bwd


@pytest.mark.parametrize("mutant", [_mutant_no_delta, _mutant_transposed_dv])
def test_planted_backward_mistake_fails_a_pin(monkeypatch, mutant):
    monkeypatch.setattr(A, "blockcausal_attention_bwd", mutant)
    with pytest.raises(AssertionError):
        test_backward_matches_torch_autograd_through_sdpa(CASES[0])
