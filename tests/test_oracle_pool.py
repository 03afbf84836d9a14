"""CPU check of the parity tests' oracle pool: the workers' results are the
oracle's own on the same bf16 values (the 16-bit patterns are widened to
float64 exactly), so the pool changes where the oracle runs, not what it
computes."""
import numpy as np
import torch

import oracle_pool
from oracle import attention as OA
from parity_helpers import bf16_bits, to64


def test_bf16_widening_is_exact():
    x = torch.randn(1000, dtype=torch.float32).to(torch.bfloat16)
    x[:4] = torch.tensor([0.0, -0.0, float("inf"), 1e-40]).to(torch.bfloat16)
    got = oracle_pool.bf16_bits_to_f64(bf16_bits(x))
    np.testing.assert_array_equal(got, to64(x))


def test_pool_rows_equal_the_serial_oracle():
    g = torch.Generator().manual_seed(5)
    results = {}
    pend = oracle_pool.Pending(lambda key, r: results.__setitem__(key, r))
    cases = []
    for i in range(6):
        q = torch.randn(7, 64, generator=g).to(torch.bfloat16)
        k = torch.randn(50 + 30 * i, 64, generator=g).to(torch.bfloat16)
        v = torch.randn(50 + 30 * i, 64, generator=g).to(torch.bfloat16)
        cases.append((q, k, v))
        pend.submit(i, (bf16_bits(q), bf16_bits(k), bf16_bits(v), 0.125))
    pend.finish()
    for i, (q, k, v) in enumerate(cases):
        o, lse = OA.softmax_attention(to64(q), to64(k), to64(v), 0.125)
        np.testing.assert_allclose(results[i][0], o, rtol=0, atol=1e-12)
        np.testing.assert_allclose(results[i][1], lse, rtol=0, atol=1e-12)
