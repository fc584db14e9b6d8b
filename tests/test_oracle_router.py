"""Pins of the router oracle (the linear map that produces the logits of
Eq. 1, Sec. 4.1) against library routines: torch's bf16 widening, numpy's
float64 matrix product and torch float64 autograd."""
import numpy as np
import pytest
import torch

import oracle


def bf16_bits(a):
    """bf16 bit patterns (uint16) of a float tensor, by torch's rounding."""
    return a.to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)


def test_bf16_widening_matches_torch():
    rng = np.random.default_rng(0)
    pats = rng.integers(0, 1 << 16, 20000).astype(np.uint16)
    exp = (pats >> 7) & 0xFF
    pats = pats[exp != 0xFF]                                 # finite values only
    specials = np.array([0x0000, 0x8000, 0x0001, 0x807F, 0x3F80, 0xBF80, 0x7F7F], np.uint16)
    pats = np.concatenate([pats, specials])
    want = torch.from_numpy(pats.view(np.int16)).view(torch.bfloat16).double().numpy()
    got = oracle.bf16_to_double(pats)
    assert np.array_equal(got, want)
    assert np.array_equal(np.signbit(got), np.signbit(want))


@pytest.mark.parametrize("T,H,E", [(1, 64, 8), (37, 128, 16), (200, 192, 128)])
def test_router_logits_match_numpy(T, H, E):
    g = torch.Generator().manual_seed(T + H + E)
    X = bf16_bits(torch.randn(T, H, generator=g))
    Wr = bf16_bits(torch.randn(E, H, generator=g) * 0.02)
    z = oracle.router_logits(X, Wr)
    want = oracle.bf16_to_double(X) @ oracle.bf16_to_double(Wr).T
    np.testing.assert_allclose(z, want, rtol=1e-13, atol=1e-15)


def test_router_gradients_match_autograd():
    T, H, E = 45, 128, 16
    g = torch.Generator().manual_seed(5)
    X = bf16_bits(torch.randn(T, H, generator=g))
    Wr = bf16_bits(torch.randn(E, H, generator=g) * 0.02)
    dz = torch.randn(T, E, generator=g, dtype=torch.float64)
    Xt = torch.from_numpy(oracle.bf16_to_double(X)).requires_grad_(True)
    Wt = torch.from_numpy(oracle.bf16_to_double(Wr)).requires_grad_(True)
    (Xt @ Wt.T).backward(dz)
    dW, dX = oracle.router_grad(X, Wr, dz.numpy(), with_dx=True)
    np.testing.assert_allclose(dW, Wt.grad.numpy(), rtol=1e-12, atol=1e-14)
    np.testing.assert_allclose(dX, Xt.grad.numpy(), rtol=1e-12, atol=1e-14)
