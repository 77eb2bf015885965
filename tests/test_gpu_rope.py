"""GPU parity of the RoPE path against the fp64 oracle (oracle/rope.py +
oracle/attn_oracle.c): dd_rope_qk, and rope -> forward -> backward with the
transposed rotation fused into the backward's dq / dk outputs."""
import numpy as np
import pytest

from attn_cases import bits_f64, check_full, check_sampled, default_scale, to_device
from oracle import rope
from paper_2405_13226_gb300 import workloads as wl

pytestmark = pytest.mark.gpu


def _oracle_rot(x_bits, base):
    """round_to_bf16(R x) in float64, and |x_2j| + |x_2j+1| per element."""
    x = bits_f64(x_bits)
    mag = np.repeat(np.abs(x[..., 0::2]) + np.abs(x[..., 1::2]), 2, axis=-1)
    return rope.round_to_bf16(rope.rope_rotate(x, base)), mag


@pytest.mark.parametrize("B,L,H,d,base", [(2, 700, 3, 64, 1e4), (1, 1, 2, 128, 1e4), (3, 384, 16, 128, 1e5),
                                          (1, 16384, 2, 128, 1e5)])
def test_rope_qk_matches_oracle(B, L, H, d, base):
    """R q rounded to bf16. The kernel evaluates x_2j cos - x_2j+1 sin in fp32
    (error ~1e-7 (|x_2j| + |x_2j+1|), which is several bf16 ulps where the sum
    cancels) before rounding, so: |gpu - oracle| <= one bf16 spacing at the
    oracle value + 1e-6 (|x_2j| + |x_2j+1|); identical almost everywhere."""
    import torch
    from paper_2405_13226_gb300 import ddattn
    qb, kb, _, _ = wl.attn_inputs(B, L, H, d, seed=4)
    q, k = to_device(qb), to_device(kb)
    qr, kr = ddattn.rope_qk(q, k, base)
    torch.cuda.synchronize()
    for got, src in ((qr, qb), (kr, kb)):
        g = got.float().cpu().numpy().astype(np.float64)
        ref, mag = _oracle_rot(src, base)
        spacing = np.ldexp(1.0, np.frexp(np.abs(ref))[1] - 8)
        err = np.abs(g - ref)
        assert np.all(err <= spacing + 1e-6 * mag), float((err / (spacing + 1e-6 * mag)).max())
        assert (err > 0).mean() < 1e-3, (err > 0).mean()
    # position 0 is the identity
    np.testing.assert_array_equal(qr[:, 0].view(torch.int16).cpu().numpy().view(np.uint16), qb[:, 0])


def test_rope_qk_in_place_equals_out_of_place():
    import torch
    from paper_2405_13226_gb300 import ddattn
    qb, kb, _, _ = wl.attn_inputs(2, 1000, 4, 128, seed=5)
    q, k = to_device(qb), to_device(kb)
    qr, kr = ddattn.rope_qk(q, k, 1e4)
    ddattn.rope_qk(q, k, 1e4, q_rot=q, k_rot=k)
    torch.cuda.synchronize()
    assert torch.equal(q.view(torch.int16), qr.view(torch.int16))
    assert torch.equal(k.view(torch.int16), kr.view(torch.int16))


def _inputs(B, L, H, d, seed=0, qk_mult=1.0):
    return wl.attn_inputs(B, L, H, d, seed=seed, qk_mult=qk_mult)


@pytest.mark.parametrize("B,L,H,d", [(2, 256, 2, 64), (2, 200, 2, 128), (1, 513, 3, 128), (3, 130, 2, 64)])
@pytest.mark.parametrize("base", [1e4, 1e5])
def test_rope_attention_small(B, L, H, d, base):
    """rope -> fwd -> bwd against round(R q), round(R k) -> attention -> R^T."""
    errs, _ = check_full(*_inputs(B, L, H, d, seed=7), default_scale(d), rope_base=base)
    print(errs)


def test_rope_attention_document_mask():
    off = wl.concat_and_chunk_offsets(3, n_chunks=2, chunk=1024)
    errs, _ = check_full(*_inputs(2, 1024, 2, 128, seed=8), default_scale(128), off, rope_base=1e4)
    print(errs)


def test_rope_bucket_full_size():
    """L = 8192 bucket (B = 8, H = 16, d = 128), f_b = 100k, sampled rows."""
    qb, kb, vb, gb = _inputs(8, 8192, 16, 128, seed=9)
    errs = check_sampled(qb, kb, vb, gb, default_scale(128), [(0, 0), (7, 15)], n_rand=6, rope_base=1e5)
    print(errs)


def test_rope_long_context_full_size():
    """B = 4 x L = 16384, H = 32, q/k x3, f_b = 100k: the largest positions."""
    qb, kb, vb, gb = _inputs(4, 16384, 32, 128, seed=10, qk_mult=3.0)
    errs = check_sampled(qb, kb, vb, gb, default_scale(128), [(3, 31)], n_rand=4, rope_base=1e5)
    print(errs)
