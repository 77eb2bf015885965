"""CUDA path (through the C ABI) vs the fp64 oracle on the same seeded inputs.

Tolerances (bf16 inputs, fp32 accumulation): O max|diff| <= 1e-2 and relative
L2 <= 5e-3; dQ, dK, dV relative L2 <= 1e-2; LSE max|diff| <= 2e-3.
Small cases compare every element; the full-size cases run the exact launch
configuration of bench.py and compare sampled rows of selected (b, h) slices.
"""
import numpy as np
import pytest

from oracle import oracle as orc
from paper_2405_13226_gb300 import workloads as wl

from attn_cases import (bits_f64, check_full, check_sampled, default_scale, doc_start_rows, oracle_full, run_cuda,
                        to_f64, rel_l2, TOL_GRAD_REL, TOL_LSE_MAX, TOL_O_MAX, TOL_O_REL)

pytestmark = pytest.mark.gpu


def _inputs(B, L, H, d, seed=0, qk_mult=1.0):
    return wl.attn_inputs(B, L, H, d, seed=seed, qk_mult=qk_mult)


def test_smoke_config_causal_d64():
    """B=4, L=256, H=2, d=64, N(0,1), scale 1/sqrt(d), no document mask: every element."""
    errs, _ = check_full(*_inputs(4, 256, 2, 64), default_scale(64))
    print(errs)


@pytest.mark.parametrize("B,L,H,d", [(2, 384, 2, 128), (1, 1024, 1, 128), (3, 200, 2, 128), (2, 129, 1, 64),
                                     (1, 1, 2, 128), (1, 1, 1, 64), (2, 7, 3, 128), (1, 300, 2, 64)])
def test_causal_ragged_and_edges(B, L, H, d):
    errs, _ = check_full(*_inputs(B, L, H, d, seed=L), default_scale(d))
    print(errs)


@pytest.mark.parametrize("B,L,H,d", [(1, 2176, 2, 128), (1, 2300, 2, 64), (1, 2432, 1, 80)])
def test_two_tile_forward_odd_and_ragged(B, L, H, d):
    """More than 16 query tiles: the forward pairs consecutive query tiles in one
    CTA. 17 tiles (the last pair has one tile), a ragged 18th tile, d = 80."""
    errs, _ = check_full(*_inputs(B, L, H, d, seed=L), default_scale(d))
    print(errs)


def test_two_tile_forward_documents_on_pair_boundaries():
    """Documents starting at the first tile of a pair (256), at the second tile of a
    pair (384, 1152) and inside a tile, L = 2304 (18 query tiles)."""
    off = np.array([0, 256, 384, 1000, 1152, 2304, 2304 + 129, 2 * 2304], dtype=np.int32)
    errs, _ = check_full(*_inputs(2, 2304, 1, 128, seed=11), default_scale(128), off)
    print(errs)


@pytest.mark.parametrize("d", [128, 80])
def test_walking_backward_many_items_documents(d):
    """Short sequences: the backward's CTAs each walk several key tiles (items) of
    different sequences and step counts. 20 x 896 (7 key tiles: 280 items over one CTA
    per SM, stride coprime with 7), documents of ragged lengths in every sequence."""
    B, L = 20, 896
    cuts = [0]
    rng = np.random.RandomState(12)
    for b in range(B):
        inner = sorted(set(rng.randint(1, L, size=3).tolist()))
        cuts += [b * L + x for x in inner] + [(b + 1) * L]
    off = np.array(cuts, dtype=np.int32)
    errs, _ = check_full(*_inputs(B, L, 2, d, seed=13), default_scale(d), off)
    print(errs)


@pytest.mark.parametrize("d", [64, 128])
@pytest.mark.parametrize("seed", [0, 5])
def test_document_mask_small(d, seed):
    """Concat-and-chunk with document masking: 2 chunks x 1024 tokens."""
    off = wl.concat_and_chunk_offsets(seed, n_chunks=2, chunk=1024)
    errs, _ = check_full(*_inputs(2, 1024, 2, d, seed=seed), default_scale(d), off)
    print(errs)


def test_document_mask_ragged_offsets():
    """Documents of 1, 2, 127, 129 ... tokens inside a ragged-length chunk."""
    L = 700
    off = np.array([0, 1, 3, 130, 259, 260, 600, L, L + 5, L + 200, 2 * L], dtype=np.int32)
    errs, _ = check_full(*_inputs(2, L, 2, 128, seed=3), default_scale(128), off)
    print(errs)


def test_single_key_rows_bitwise():
    """The first token of each document attends only to itself: P = 1, l = 1, so
    o equals v bit for bit and LSE equals scale * <q_i, k_i>."""
    off = wl.concat_and_chunk_offsets(1, n_chunks=2, chunk=1024)
    qb, kb, vb, gb = _inputs(2, 1024, 2, 128, seed=1)
    scale = default_scale(128)
    o, lse, *_ = run_cuda(qb, kb, vb, gb, scale, off)
    o_bits = o.view(__import__("torch").int16).cpu().numpy().view(np.uint16)
    lse = lse.cpu().numpy()
    q, k = bits_f64(qb), bits_f64(kb)
    for (b, i) in doc_start_rows(2, 1024, off):
        np.testing.assert_array_equal(o_bits[b, i], vb[b, i])
        for h in range(2):
            assert abs(lse[b, h, i] - scale * q[b, i, h] @ k[b, i, h]) < 1e-4


def test_document_mask_equals_separate_calls():
    """A document-masked call equals separate plain causal calls on each document."""
    import torch
    L = 1024
    off = wl.concat_and_chunk_offsets(2, n_chunks=1, chunk=L)
    qb, kb, vb, gb = _inputs(1, L, 2, 128, seed=2)
    scale = default_scale(128)
    full = [to_f64(t) for t in run_cuda(qb, kb, vb, gb, scale, off)]
    for s, e in zip(off[:-1], off[1:]):
        part = [to_f64(t) for t in run_cuda(qb[:, s:e].copy(), kb[:, s:e].copy(), vb[:, s:e].copy(),
                                            gb[:, s:e].copy(), scale)]
        np.testing.assert_allclose(full[0][:, s:e], part[0], atol=2e-2)
        np.testing.assert_allclose(full[1][:, :, s:e], part[1], atol=1e-3)
        for a, bb in zip(full[2:], part[2:]):
            np.testing.assert_allclose(a[:, s:e], bb, atol=5e-2)


@pytest.mark.parametrize("L", wl.BUCKETS)
def test_bucket_sweep_full_size(L):
    """1B-model bucket: H=16, d=128, 65536 tokens per call (B = 65536 / L)."""
    B, H, d = wl.TOKENS_PER_STEP // L, 16, 128
    qb, kb, vb, gb = _inputs(B, L, H, d)
    slices = [(0, 0), (0, H - 1), (B - 1, 3), (B // 2, 9)]
    errs = check_sampled(qb, kb, vb, gb, default_scale(d), slices, n_rand=6)
    print(L, errs)


@pytest.mark.parametrize("seed", [0, 7])
def test_dm_baseline_full_size(seed):
    """Concat-and-chunk baseline: 8 chunks x 8192, H=16, d=128, document-masked."""
    off = wl.concat_and_chunk_offsets(seed)
    qb, kb, vb, gb = _inputs(8, 8192, 16, 128, seed=seed)
    gpu = run_cuda(qb, kb, vb, gb, default_scale(128), off)
    errs = check_sampled(qb, kb, vb, gb, default_scale(128), [(0, 0), (3, 5), (7, 15)], off, n_rand=6, gpu=gpu)
    print(errs)
    o_bits = gpu[0].view(__import__("torch").int16).cpu().numpy().view(np.uint16)
    for (b, i) in doc_start_rows(8, 8192, off):
        np.testing.assert_array_equal(o_bits[b, i], vb[b, i])


def test_dm_short_chunks_full_size():
    """Concat-and-chunk at 32 chunks x 2048 (H=16, d=128): the short-sequence
    forward path with document offsets over thousands of query tiles."""
    off = wl.concat_and_chunk_offsets(9, n_chunks=32, chunk=2048)
    qb, kb, vb, gb = _inputs(32, 2048, 16, 128, seed=9)
    gpu = run_cuda(qb, kb, vb, gb, default_scale(128), off)
    errs = check_sampled(qb, kb, vb, gb, default_scale(128), [(0, 0), (31, 15), (17, 6)], off, n_rand=6, gpu=gpu)
    print(errs)
    o_bits = gpu[0].view(__import__("torch").int16).cpu().numpy().view(np.uint16)
    for (b, i) in doc_start_rows(32, 2048, off):
        np.testing.assert_array_equal(o_bits[b, i], vb[b, i])


@pytest.mark.parametrize("seed", [0, 3])
def test_pack8k_dm_full_size(seed):
    """Pack-8k+DM: best-fit-decreasing bins of 8192 tokens with masked pad tails."""
    off = wl.packed_dm_offsets(seed)
    qb, kb, vb, gb = _inputs(8, 8192, 16, 128, seed=seed + 20)
    gpu = run_cuda(qb, kb, vb, gb, default_scale(128), off)
    errs = check_sampled(qb, kb, vb, gb, default_scale(128), [(0, 0), (5, 9)], off, n_rand=6, gpu=gpu)
    print(errs)
    o_bits = gpu[0].view(__import__("torch").int16).cpu().numpy().view(np.uint16)
    for (b, i) in doc_start_rows(8, 8192, off):
        np.testing.assert_array_equal(o_bits[b, i], vb[b, i])


def test_long_context_full_size():
    """B=4 x L=16384, H=32, d=128, q/k scaled x3 before bf16 rounding."""
    qb, kb, vb, gb = _inputs(4, 16384, 32, 128, qk_mult=3.0)
    errs = check_sampled(qb, kb, vb, gb, default_scale(128), [(0, 0), (3, 31)], n_rand=4)
    print(errs)


def test_every_token_its_own_document():
    """Degenerate document mask: each token is a one-token document, so every row
    attends only to itself: o = v and dv = dO exactly (P = 1), and dq, dk vanish up
    to the rounding of dS = P (dP - D), whose two fp32 dot products of the same
    vectors are summed in different orders."""
    import torch
    B, L, H, d = 2, 300, 2, 128
    off = np.arange(0, B * L + 1, dtype=np.int32)
    qb, kb, vb, gb = _inputs(B, L, H, d, seed=12)
    o, lse, dq, dk, dv = run_cuda(qb, kb, vb, gb, default_scale(d), off)
    np.testing.assert_array_equal(o.view(torch.int16).cpu().numpy().view(np.uint16), vb)
    assert float(dq.float().abs().max()) < 1e-4 and float(dk.float().abs().max()) < 1e-4
    np.testing.assert_array_equal(dv.view(torch.int16).cpu().numpy().view(np.uint16), gb)


def test_longest_document_full_size():
    """One 65536-token sequence (the longest document of the length model), H=1:
    the largest positions and tile counts; sampled rows against the oracle."""
    qb, kb, vb, gb = _inputs(1, 65536, 1, 128, seed=13)
    errs = check_sampled(qb, kb, vb, gb, default_scale(128), [(0, 0)], n_rand=6)
    print(errs)


def test_many_short_sequences():
    """B = 32768 sequences of L = 8 (H = 2, d = 64): a grid of 32768 x 2 CTAs of
    one ragged tile each."""
    qb, kb, vb, gb = _inputs(32768, 8, 2, 64, seed=14)
    errs = check_sampled(qb, kb, vb, gb, default_scale(64), [(0, 0), (32767, 1), (12345, 0)], n_rand=2)
    print(errs)


def _offsets_unlisted_cuts_and_empty_docs(B, L, seed, per_seq=3):
    """Document offsets that list NO sequence boundary b*L (0 < b < B): every inner
    boundary falls inside a document, which the kernels must cut there anyway. The
    list also repeats values (empty documents): 0 twice at the start, B*L twice at
    the end, and two inner offsets twice."""
    rng = np.random.default_rng(seed)
    cand = np.array([t for t in range(1, B * L) if t % L != 0])
    inner = np.sort(rng.choice(cand, size=per_seq * B, replace=False))
    dup = rng.choice(inner, size=2, replace=False)
    off = np.sort(np.concatenate([[0, 0], inner, dup, [B * L, B * L]])).astype(np.int32)
    assert not any(b * L in set(off.tolist()) for b in range(1, B))
    assert (np.diff(off) >= 0).all() and (np.diff(off) == 0).sum() >= 4
    return off


@pytest.mark.parametrize("d", [128, 80, 64])
@pytest.mark.parametrize("B,L", [(3, 1000), (2, 2500)])
def test_offsets_omit_sequence_cuts_and_repeat(B, L, d):
    """cu_doc_offsets that omit the sequence boundaries (documents straddle them) and
    repeat values (empty documents), every element against the oracle. L = 1000 runs
    the walking backward (at most 16 key tiles), L = 2500 the one-CTA-per-key-tile
    backward (d = 80, 128)."""
    off = _offsets_unlisted_cuts_and_empty_docs(B, L, seed=L + d)
    errs, _ = check_full(*_inputs(B, L, 2, d, seed=L + d), default_scale(d), off)
    print(errs)


@pytest.mark.parametrize("d", [128, 80])
def test_offsets_without_inner_entries_equal_causal(d):
    """Offsets [0, B*L] (one document over the whole flattened batch, no boundary
    listed) give the plain causal result: sequence boundaries always cut. o, lse, dk and
    dv are bitwise equal; dq sums its fp32 partials in an order that depends on the
    backward's walk (the document-masked call may take another one), so it agrees up to
    that rounding."""
    import torch
    B, L = 3, 1000
    qb, kb, vb, gb = _inputs(B, L, 2, d, seed=21)
    scale = default_scale(d)
    plain = run_cuda(qb, kb, vb, gb, scale)
    one_doc = run_cuda(qb, kb, vb, gb, scale, np.array([0, B * L], dtype=np.int32))
    for name, a, b in zip(("o", "lse", "dq", "dk", "dv"), plain, one_doc):
        if name == "dq":
            assert rel_l2(to_f64(b), to_f64(a)) <= 1e-3, name
        elif a.dtype == torch.bfloat16:
            assert torch.equal(a.view(torch.int16), b.view(torch.int16)), name
        else:
            assert torch.equal(a, b), name


@pytest.mark.parametrize("d,B,L,H,docs", [(128, 156, 130, 1, False), (80, 200, 130, 1, True),
                                          (128, 304, 60, 1, True)])
def test_short_sequences_pairs_per_cta_reuse_slot(d, B, L, H, docs):
    """Short sequences (at most 2 key tiles) where the backward's CTAs own whole (sequence,
    head) pairs and keep dQ in one slot each: more pairs than SMs, so CTAs own several
    pairs one after another and reuse their slot (up to 2 pairs per CTA); ragged lengths
    and documents. Every element against the oracle: dq, dk, dv and LSE at the parity
    tolerances, O by relative L2 and element by element within max(1e-2, one bf16 ulp of
    the reference). Nearly every row here has few keys, so |o| often exceeds 2, where one
    bf16 ulp is 0.0156 (0.031 above 4): an output one ulp from the correctly rounded value
    (an fp32 result on the other side of a rounding midpoint) is as close as bf16 allows."""
    off = None
    if docs:
        rng = np.random.default_rng(L + d)
        cuts = {0, B * L}
        for b in range(B):
            cuts |= {b * L + int(x) for x in rng.integers(1, L, size=int(rng.integers(0, 4)))}
        off = np.array(sorted(cuts), dtype=np.int32)
    qb, kb, vb, gb = _inputs(B, L, H, d, seed=B + L)
    o, lse, dq, dk, dv = run_cuda(qb, kb, vb, gb, default_scale(d), off)
    ro, rlse, rdq, rdk, rdv = oracle_full(qb, kb, vb, gb, default_scale(d), off)
    ulp = np.ldexp(1.0, np.frexp(np.abs(ro))[1] - 8)          # bf16 spacing at |o_ref|
    excess = np.abs(to_f64(o) - ro) - np.maximum(TOL_O_MAX, ulp)
    errs = {"o_excess_max": float(excess.max()), "o_max": float(np.abs(to_f64(o) - ro).max()),
            "o_rel": rel_l2(to_f64(o), ro),
            "lse_max": float(np.abs(to_f64(lse) - rlse).max()), "dq_rel": rel_l2(to_f64(dq), rdq),
            "dk_rel": rel_l2(to_f64(dk), rdk), "dv_rel": rel_l2(to_f64(dv), rdv)}
    print(errs)
    assert errs["o_excess_max"] <= 0 and errs["o_rel"] <= TOL_O_REL, errs
    assert errs["lse_max"] <= TOL_LSE_MAX, errs
    assert max(errs["dq_rel"], errs["dk_rel"], errs["dv_rel"]) <= TOL_GRAD_REL, errs
