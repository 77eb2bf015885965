"""Pins of the RoPE oracle (oracle/rope.py) to facts other than itself (CPU only).

RoPE as used before the attention module (Sec. 3): consecutive components of
q and k are rotated by m * f_b^(-2j/d) at position m. Pinned against a
complex-number formulation in torch, closed-form angles, the relative-position
property that makes RoPE attention depend on m - n only, finite differences
and torch autograd through RoPE + attention, and torch's bf16 rounding.
"""
import math

import numpy as np
import pytest

from oracle import oracle as orc
from oracle import rope


def _rand(shape, seed):
    return np.random.default_rng(seed).standard_normal(shape)


def test_complex_formulation_matches():
    """Consecutive pairs as complex numbers x[2j] + i x[2j+1], multiplied by
    exp(i m theta_j) (torch complex128)."""
    torch = pytest.importorskip("torch")
    B, L, H, d, base = 2, 37, 3, 16, 10000.0
    x = _rand((B, L, H, d), 0)
    xc = torch.view_as_complex(torch.from_numpy(x).reshape(B, L, H, d // 2, 2).contiguous())
    theta = base ** (-torch.arange(0, d, 2, dtype=torch.float64) / d)
    ang = torch.arange(L, dtype=torch.float64)[:, None] * theta[None, :]
    rot = xc * torch.polar(torch.ones_like(ang), ang)[None, :, None, :]
    ref = torch.view_as_real(rot).reshape(B, L, H, d).numpy()
    np.testing.assert_allclose(rope.rope_rotate(x, base), ref, rtol=0, atol=1e-12)


def test_closed_form_angles():
    """d = 4, f_b = 10^4: theta_0 = 1 and theta_1 = 10^-2. A unit vector e_0
    at position m turns by m radians, e_2 by m / 100."""
    x = np.zeros((1, 201, 1, 4))
    x[0, :, 0, 0] = 1.0
    x2 = np.zeros_like(x)
    x2[0, :, 0, 2] = 1.0
    r, r2 = rope.rope_rotate(x, 1e4), rope.rope_rotate(x2, 1e4)
    for m in (0, 1, 3, 100, 200):
        np.testing.assert_allclose(r[0, m, 0], [math.cos(m), math.sin(m), 0, 0], atol=1e-14)
        np.testing.assert_allclose(r2[0, m, 0], [0, 0, math.cos(m / 100), math.sin(m / 100)], atol=1e-14)


def test_orthogonal_and_inverse():
    x = _rand((2, 50, 2, 8), 1)
    r = rope.rope_rotate(x, 1e5)
    n = lambda a: np.sqrt(a[..., 0::2] ** 2 + a[..., 1::2] ** 2)
    np.testing.assert_allclose(n(r), n(x), rtol=1e-13)
    np.testing.assert_allclose(rope.rope_unrotate(r, 1e5), x, atol=1e-13)


def test_relative_position_property():
    """<R_m q, R_n k> depends on m - n only: shifting both positions by t
    leaves every score unchanged."""
    d, base, L = 16, 1e4, 64
    q, k = _rand(d, 2), _rand(d, 3)
    Q = rope.rope_rotate(np.broadcast_to(q, (1, L, 1, d)).copy(), base)[0, :, 0]
    K = rope.rope_rotate(np.broadcast_to(k, (1, L, 1, d)).copy(), base)[0, :, 0]
    S = Q @ K.T
    for t in (1, 5, 20):
        np.testing.assert_allclose(S[t:, t:], S[:-t, :-t], rtol=0, atol=1e-12)
    # and the diagonal (m = n) is the unrotated product
    np.testing.assert_allclose(np.diag(S), np.full(L, q @ k), atol=1e-12)


def _rope_attn_loss(q, k, v, dO, doc, scale, base):
    L, d = q.shape
    qr = rope.rope_rotate(q[None, :, None, :], base)[0, :, 0]
    kr = rope.rope_rotate(k[None, :, None, :], base)[0, :, 0]
    o, _ = orc.attn_fwd(qr[None], kr[None], v[None], doc[None], scale)
    return float((o[0] * dO).sum())


def _rope_attn_grads(q, k, v, dO, doc, scale, base):
    qr = rope.rope_rotate(q[None, :, None, :], base)[0, :, 0]
    kr = rope.rope_rotate(k[None, :, None, :], base)[0, :, 0]
    dqr, dkr, dv = orc.attn_bwd(qr[None], kr[None], v[None], dO[None], doc[None], scale)
    dq = rope.rope_unrotate(dqr[0][None, :, None, :], base)[0, :, 0]
    dk = rope.rope_unrotate(dkr[0][None, :, None, :], base)[0, :, 0]
    return dq, dk, dv[0]


@pytest.mark.parametrize("base", [1e4, 1e5, 3.0])
def test_rope_attention_finite_differences(base):
    """dq, dk of attention on rotated q, k (R^T of the rotated-space gradients)
    equal central differences of sum(o * dO) with respect to the un-rotated q, k."""
    L, d, scale = 9, 6, 0.8
    doc = np.array([0, 0, 0, 0, 1, 1, 1, 1, 1], dtype=np.int32)
    q, k, v, dO = (_rand((L, d), s) for s in (10, 11, 12, 13))
    dq, dk, _ = _rope_attn_grads(q, k, v, dO, doc, scale, base)
    h = 1e-6
    for name, x, g in (("q", q, dq), ("k", k, dk)):
        num = np.zeros_like(x)
        for idx in np.ndindex(x.shape):
            xp, xm = x.copy(), x.copy()
            xp[idx] += h
            xm[idx] -= h
            a = dict(q=q, k=k); a[name] = xp
            b = dict(q=q, k=k); b[name] = xm
            num[idx] = (_rope_attn_loss(a["q"], a["k"], v, dO, doc, scale, base) -
                        _rope_attn_loss(b["q"], b["k"], v, dO, doc, scale, base)) / (2 * h)
        assert np.linalg.norm(num - g) / np.linalg.norm(num) < 1e-6, name


def test_rope_attention_torch_autograd():
    """torch fp64 autograd through the complex-number RoPE and a dense masked
    softmax attention agrees with the oracle composition."""
    torch = pytest.importorskip("torch")
    L, d, scale, base = 12, 8, 0.5, 1e4
    doc = np.array([0] * 5 + [1] * 7, dtype=np.int32)
    q, k, v, dO = (_rand((L, d), s) for s in (20, 21, 22, 23))
    tq, tk, tv = (torch.tensor(x, requires_grad=True) for x in (q, k, v))
    theta = base ** (-torch.arange(0, d, 2, dtype=torch.float64) / d)
    ang = torch.arange(L, dtype=torch.float64)[:, None] * theta[None, :]
    rotc = torch.polar(torch.ones_like(ang), ang)

    def rot(x):
        return torch.view_as_real(torch.view_as_complex(x.reshape(L, d // 2, 2)) * rotc).reshape(L, d)

    s = scale * rot(tq) @ rot(tk).T
    i = torch.arange(L)
    tdoc = torch.from_numpy(doc)
    live = (i[None, :] <= i[:, None]) & (tdoc[None, :] == tdoc[:, None])
    o = torch.softmax(s.masked_fill(~live, float("-inf")), dim=-1) @ tv
    (o * torch.from_numpy(dO)).sum().backward()
    dq, dk, dv = _rope_attn_grads(q, k, v, dO, doc, scale, base)
    np.testing.assert_allclose(dq, tq.grad.numpy(), atol=1e-10)
    np.testing.assert_allclose(dk, tk.grad.numpy(), atol=1e-10)
    np.testing.assert_allclose(dv, tv.grad.numpy(), atol=1e-10)


def test_half_split_layout_is_a_channel_permutation():
    """Rotating pairs (j, j + d/2) instead of (2j, 2j+1) is the same rotation
    after a fixed permutation of the head channels, applied to q and k alike;
    attention scores are unchanged."""
    L, d, base = 20, 8, 1e4
    q, k = _rand((1, L, 1, d), 30), _rand((1, L, 1, d), 31)
    perm = np.empty(d, dtype=int)
    perm[0::2] = np.arange(d // 2)
    perm[1::2] = np.arange(d // 2) + d // 2        # interleaved channel c <- half-split channel perm[c]
    a = rope.angles(L, d, base)[None, :, None, :]
    c, s = np.cos(a), np.sin(a)

    def half_split(x):
        x1, x2 = x[..., : d // 2], x[..., d // 2:]
        return np.concatenate([x1 * c - x2 * s, x1 * s + x2 * c], axis=-1)

    S_half = half_split(q)[0, :, 0] @ half_split(k)[0, :, 0].T
    S_ours = rope.rope_rotate(q[..., perm], base)[0, :, 0] @ rope.rope_rotate(k[..., perm], base)[0, :, 0].T
    np.testing.assert_allclose(S_ours, S_half, atol=1e-12)


def test_bf16_rounding_matches_torch():
    """round_to_bf16 equals torch's float32 -> bfloat16 conversion (nearest,
    ties to even) on float32 values, including exact ties and subnormals."""
    torch = pytest.importorskip("torch")
    x = (np.random.default_rng(5).standard_normal(200000) * 10).astype(np.float32)
    x[:6] = [1.00390625, 1.01171875, -1.00390625, 3.0e-39, -2.5e-40, 65504.0]
    ref = torch.from_numpy(x).to(torch.bfloat16).to(torch.float64).numpy()
    np.testing.assert_array_equal(rope.round_to_bf16(x.astype(np.float64)), ref)
