"""Other model shapes of the paper's OpenLM family (model table of the
Appendix): the 3B model's heads (H = 32, d = 2560 / 32 = 80) and the 7B
model's (H = 32, d = 4096 / 32 = 128), against the fp64 oracle."""
import pytest

from attn_cases import check_full, check_sampled, default_scale
from paper_2405_13226_gb300 import workloads as wl

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("B,L,H,d", [(2, 256, 2, 80), (3, 200, 2, 80), (1, 513, 3, 80), (1, 1, 2, 80),
                                     (2, 7, 1, 80), (1, 1024, 1, 80)])
def test_d80_causal_every_element(B, L, H, d):
    errs, _ = check_full(*wl.attn_inputs(B, L, H, d, seed=L + 1), default_scale(d))
    print(errs)


@pytest.mark.parametrize("seed", [1, 4])
def test_d80_document_mask(seed):
    off = wl.concat_and_chunk_offsets(seed, n_chunks=2, chunk=1024)
    errs, _ = check_full(*wl.attn_inputs(2, 1024, 2, 80, seed=seed), default_scale(80), off)
    print(errs)


@pytest.mark.parametrize("base", [1e4, 1e5])
def test_d80_rope(base):
    errs, _ = check_full(*wl.attn_inputs(2, 300, 2, 80, seed=11), default_scale(80), rope_base=base)
    print(errs)


@pytest.mark.parametrize("L", [256, 2048, 8192])
def test_3b_shape_full_size(L):
    """3B heads: H = 32, d = 80, 65536 tokens per call, sampled rows."""
    B = wl.TOKENS_PER_STEP // L
    qb, kb, vb, gb = wl.attn_inputs(B, L, 32, 80, seed=L)
    errs = check_sampled(qb, kb, vb, gb, default_scale(80), [(0, 0), (B - 1, 31), (B // 2, 17)], n_rand=5)
    print(L, errs)


def test_7b_shape_full_size():
    """7B heads: H = 32, d = 128, L = 4096 bucket, sampled rows."""
    qb, kb, vb, gb = wl.attn_inputs(16, 4096, 32, 128, seed=3)
    errs = check_sampled(qb, kb, vb, gb, default_scale(128), [(0, 0), (15, 31)], n_rand=5)
    print(errs)
