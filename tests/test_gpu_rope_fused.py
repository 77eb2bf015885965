"""GPU parity of the forward with RoPE fused into its tile loads (dd_attn_fwd_rope)
against the fp64 oracle (oracle/rope.py + oracle/attn_oracle.c): the rotated q, k
it returns, and fused forward -> backward (the backward takes those rotated q, k
and returns dq, dk with respect to the un-rotated ones).

Sequences of at most 4 key tiles (L <= 512) rotate Q and K tiles in the kernel;
longer ones rotate k in a pass first and Q tiles in the kernel. Both forms are
covered, with plain and document-masked inputs, ragged lengths and every head dim."""
import numpy as np
import pytest

from attn_cases import bits_f64, check_full, check_sampled, default_scale, to_device
from oracle import rope
from paper_2405_13226_gb300 import workloads as wl

pytestmark = pytest.mark.gpu


def _check_rotated(got, src_bits, base):
    """got = bf16 R x from the fused forward, whose (cos, sin) of a row are stepped from the
    position table by an angle-sum step of 8 positions (error a few 1e-7 after up to 15
    steps): |got - oracle| <= one bf16 spacing at the correctly rounded oracle value +
    4e-6 (|x_2j| + |x_2j+1|), values differ from the correctly rounded ones rarely, and from
    dd_rope_qk's output (same formula, table values) in fewer than 1e-3 of the elements."""
    import torch
    from paper_2405_13226_gb300 import ddattn
    x = bits_f64(src_bits)
    ref = rope.round_to_bf16(rope.rope_rotate(x, base))
    mag = np.repeat(np.abs(x[..., 0::2]) + np.abs(x[..., 1::2]), 2, axis=-1)
    g = got.float().cpu().numpy().astype(np.float64)
    spacing = np.ldexp(1.0, np.frexp(np.abs(ref))[1] - 8)
    err = np.abs(g - ref)
    assert np.all(err <= spacing + 4e-6 * mag), float((err / (spacing + 4e-6 * mag)).max())
    assert (err > 0).mean() < 2e-3, (err > 0).mean()
    src = to_device(src_bits)
    sep, _ = ddattn.rope_qk(src, src, base)
    torch.cuda.synchronize()
    a = got.view(torch.int16).cpu().numpy().astype(np.int32)
    b = sep.view(torch.int16).cpu().numpy().astype(np.int32)
    assert (a != b).mean() < 1e-3, (a != b).mean()


@pytest.mark.parametrize("B,L,H,d", [(2, 256, 2, 64), (2, 200, 2, 128), (1, 513, 3, 128), (3, 130, 2, 64),
                                     (2, 384, 2, 80), (1, 2300, 2, 128), (1, 2176, 2, 80)])
@pytest.mark.parametrize("base", [1e4, 1e5])
def test_fused_rope_attention_small(B, L, H, d, base):
    """fused rope + fwd -> bwd against round(R q), round(R k) -> attention -> R^T, every
    element; L = 200, 256 and 384 rotate K tiles in the kernel, the others take the k pass."""
    rot = []
    qb, kb, vb, gb = wl.attn_inputs(B, L, H, d, seed=17)
    errs, _ = check_full(qb, kb, vb, gb, default_scale(d), rope_base=base, fused_rope=True, rotated=rot)
    _check_rotated(rot[0], qb, base)
    _check_rotated(rot[1], kb, base)
    print(errs)


@pytest.mark.parametrize("L", [512, 4096])
def test_fused_rope_document_mask(L):
    """Document-masked chunks (work items start their K tiles at their documents' starts)."""
    off = wl.concat_and_chunk_offsets(3, n_chunks=2, chunk=L)
    rot = []
    qb, kb, vb, gb = wl.attn_inputs(2, L, 2, 128, seed=18)
    errs, _ = check_full(qb, kb, vb, gb, default_scale(128), off, rope_base=1e4, fused_rope=True, rotated=rot)
    _check_rotated(rot[0], qb, 1e4)
    _check_rotated(rot[1], kb, 1e4)
    print(errs)


def test_fused_rope_matches_separate_pass_and_in_place():
    """Same inputs through dd_rope_qk + dd_attn_fwd and through dd_attn_fwd_rope (out of
    place, and with q_rot = q), at lengths of both forms: o and lse agree with the separate
    path to the rounding of the rare last-bit differences of the rotated inputs, the
    in-place call equals the out-of-place one bit for bit, and k is left untouched."""
    import torch
    from paper_2405_13226_gb300 import ddattn
    bits = lambda t: t.view(torch.int16) if t.dtype == torch.bfloat16 else t
    for B, L, H, d, base in ((2, 500, 4, 128, 1e5), (2, 1000, 4, 128, 1e5), (1, 2200, 2, 128, 1e4),
                             (2, 700, 2, 80, 1e5)):
        qb, kb, vb, _ = wl.attn_inputs(B, L, H, d, seed=19)
        q, k, v = (to_device(x) for x in (qb, kb, vb))
        k_before = k.clone()
        qr, kr = ddattn.rope_qk(q, k, base)
        o_sep, lse_sep = ddattn.fwd(qr, kr, v)
        o, lse, q_rot, k_rot = ddattn.fwd_rope(q, k, v, base)
        q2 = q.clone()
        o2, lse2, q_rot2, k_rot2 = ddattn.fwd_rope(q2, k, v, base, q_rot=q2)
        torch.cuda.synchronize()
        assert torch.equal(k, k_before)
        assert q_rot2.data_ptr() == q2.data_ptr()
        for a, b2 in ((o, o2), (lse, lse2), (q_rot, q_rot2), (k_rot, k_rot2)):
            assert torch.equal(bits(a), bits(b2)), (B, L, H, d)
        assert (o.float() - o_sep.float()).abs().max().item() <= 2e-2, (B, L, H, d)
        assert (lse - lse_sep).abs().max().item() <= 1e-3, (B, L, H, d)


def test_fused_rope_one_token_and_position_zero():
    """L = 1 (one position, the identity rotation) and position 0 of a longer sequence:
    rotated rows equal the inputs bit for bit; attention of a single key is v."""
    import torch
    from paper_2405_13226_gb300 import ddattn
    for L in (1, 640):
        qb, kb, vb, _ = wl.attn_inputs(3, L, 2, 128, seed=20)
        q, k, v = (to_device(x) for x in (qb, kb, vb))
        o, lse, q_rot, k_rot = ddattn.fwd_rope(q, k, v, 1e4)
        torch.cuda.synchronize()
        for got, src in ((q_rot, qb), (k_rot, kb)):
            np.testing.assert_array_equal(got[:, 0].view(torch.int16).cpu().numpy().view(np.uint16), src[:, 0])
        np.testing.assert_array_equal(o[:, 0].view(torch.int16).cpu().numpy().view(np.uint16), vb[:, 0])


@pytest.mark.parametrize("L", [512, 2048, 8192])
def test_fused_rope_bucket_full_size(L):
    """Full buckets of 65536 tokens (H = 16, d = 128), f_b = 100k, sampled rows (L = 512:
    K tiles rotated in the kernel; 2048, 8192: the k pass)."""
    qb, kb, vb, gb = wl.attn_inputs(65536 // L, L, 16, 128, seed=21)
    errs = check_sampled(qb, kb, vb, gb, default_scale(128), [(0, 0), (65536 // L - 1, 15)], n_rand=6,
                         rope_base=1e5, fused_rope=True)
    print(errs)


def test_fused_rope_long_context_full_size():
    """B = 4 x L = 16384, H = 32, q/k x3, f_b = 100k: the largest positions (the inputs of
    the separate path's long-context test)."""
    qb, kb, vb, gb = wl.attn_inputs(4, 16384, 32, 128, seed=10, qk_mult=3.0)
    errs = check_sampled(qb, kb, vb, gb, default_scale(128), [(3, 31)], n_rand=4, rope_base=1e5, fused_rope=True)
    print(errs)


def test_fused_rope_3b_heads_full_size():
    """OpenLM-3B heads (H = 32, d = 80) at L = 2048."""
    qb, kb, vb, gb = wl.attn_inputs(32, 2048, 32, 80, seed=23)
    errs = check_sampled(qb, kb, vb, gb, default_scale(80), [(0, 0), (31, 31)], n_rand=6, rope_base=1e5,
                         fused_rope=True)
    print(errs)
