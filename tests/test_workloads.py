"""Workload generators and statistics (CPU only)."""
import json
import os

import numpy as np
import pytest

from paper_2405_13226_gb300 import workloads as wl

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def test_binary_decomposition_invariants():
    """Sec. 2.1: pieces are distinct powers of two, largest first, adjacent, summing to l."""
    for n in [1, 2, 3, 255, 256, 257, 1000, 8191, 8192, 12345, 65536]:
        p = wl.binary_decompose(n)
        assert sum(p) == n
        assert all(x & (x - 1) == 0 for x in p)
        assert p == sorted(set(p), reverse=True)
    assert wl.binary_decompose(13) == [8, 4, 1]


def test_table1_average_lengths():
    """Average sequence length and Eq. (avg_context) reproduce Table 1 from its
    bucket token counts (printed values are rounded to integers)."""
    g = json.load(open(os.path.join(GOLDEN, "table1_mixtures.json")))
    lens = [2 ** i for i in g["buckets_log2"]]
    for name, m in g["mixtures"].items():
        seqs = []
        for L, t in zip(lens, m["tokens"]):
            seqs += [L] * int(t * 2 ** 20 // L)     # tokens scaled by 2^-10: same ratios
        assert abs(wl.avg_sequence_length(seqs) - m["avg_seq_len"]) <= 0.51, name
        assert abs(wl.avg_context_length(seqs) - m["avg_ctx_len"]) <= 0.51, name


def test_avg_context_brute_force():
    rng = np.random.default_rng(0)
    lens = rng.integers(1, 50, size=30)
    brute = sum(sum(range(n)) for n in lens) / lens.sum()
    assert wl.avg_context_length(lens) == pytest.approx(brute, rel=1e-12)


def test_dm_offsets_valid():
    for seed in range(16):
        off = wl.concat_and_chunk_offsets(seed)
        assert off.dtype == np.int32
        assert off[0] == 0 and off[-1] == 8 * 8192
        assert np.all(np.diff(off) > 0)
        assert set(range(0, 8 * 8192 + 1, 8192)) <= set(off.tolist())
        frac = wl.live_pairs(8, 8192, off) / wl.live_pairs(8, 8192)
        assert 0.0 < frac < 1.0


def test_dd_buckets_conserve_tokens_and_shares():
    counts = wl.dd_bucket_tokens(seed=0, n_docs=20000)
    assert set(counts) == set(wl.BUCKETS)
    assert all(c % L == 0 for L, c in counts.items())
    share = np.array([counts[L] for L in wl.BUCKETS], dtype=float)
    share /= share.sum()
    # Natural mixture of Table 1 restricted to D8..D13 (10,17,21,17,13,9): the
    # lognormal stand-in is close but not equal to RefinedWeb.
    paper = np.array([10, 17, 21, 17, 13, 9], dtype=float)
    paper /= paper.sum()
    assert np.abs(share - paper).max() < 0.06


def test_curriculum_stream():
    s = wl.curriculum_stream(seed=0, steps=200, bucket_tokens={256: 1, 1024: 3})
    assert len(s) == 200 and set(s) <= {256, 1024}
    assert 0.6 < s.count(1024) / 200 < 0.9
    assert s == wl.curriculum_stream(seed=0, steps=200, bucket_tokens={256: 1, 1024: 3})


def test_bf16_rounding_matches_torch():
    torch = pytest.importorskip("torch")
    x = np.random.default_rng(1).standard_normal(100000).astype(np.float32) * 7
    x[:4] = [1.00390625, 1.01171875, -1.00390625, 3.0e-39]   # ties and a subnormal
    ours = wl.f32_to_bf16_bits(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(ours, ref)


def test_flop_convention():
    assert wl.attn_flops(4, 256, 2, 64) == 14 * 64 * 2 * 4 * 256 * 257 // 2
    # DD step flops are linear in L at fixed tokens per step
    f = [wl.attn_flops(wl.TOKENS_PER_STEP // L, L, 16, 128) for L in wl.BUCKETS]
    assert f[-1] / f[0] == pytest.approx(8193 / 257)


def _run_curriculum(name, cycles, seed=0):
    counts = {L: 64 * L * 4 for L in wl.BUCKETS}          # 256 sequences' worth of tokens per bucket
    odds = dict(zip(wl.BUCKETS, wl.CURRICULA[name]))
    return counts, wl.length_curriculum(counts, odds, cycles, tokens_per_step=8192, seed=seed)


@pytest.mark.parametrize("name", list(wl.CURRICULA))
@pytest.mark.parametrize("cycles", [1, 8])
def test_algorithm1_consumes_every_bucket_exactly(name, cycles):
    """Algorithm 1: every token of every bucket is used once; each step is one
    bucket with b tokens (b / 2^i sequences)."""
    counts, steps = _run_curriculum(name, cycles)
    used = {L: 0 for L in wl.BUCKETS}
    for L in steps:
        used[L] += 8192
    assert used == counts
    assert len(steps) == sum(c // 8192 for c in counts.values())


def test_algorithm1_cycles_partition_the_stream():
    """With c cycles each bucket's subset of a cycle is exhausted before the
    next cycle starts: the stream splits into c blocks with n_i / c tokens each."""
    counts, steps = _run_curriculum("Grow-P2", 8)
    per_cycle_steps = sum(c // 8192 for c in counts.values()) // 8
    for j in range(8):
        block = steps[j * per_cycle_steps:(j + 1) * per_cycle_steps]
        for L in wl.BUCKETS:
            assert block.count(L) * 8192 == counts[L] // 8


def test_algorithm1_curriculum_order():
    """Grow-P100 draws short sequences first, Shrink-P100 long ones first; the
    first draw follows the normalised odds."""
    _, grow = _run_curriculum("Grow-P100", 1)
    _, shrink = _run_curriculum("Shrink-P100", 1)
    n = len(grow)
    assert np.mean(grow[: n // 4]) < np.mean(grow[-n // 4:])
    assert np.mean(shrink[: n // 4]) > np.mean(shrink[-n // 4:])
    firsts = [_run_curriculum("Grow-Linear", 1, seed=s)[1][0] for s in range(300)]
    frac256 = firsts.count(256) / 300            # odds 6 / 21
    assert abs(frac256 - 6 / 21) < 0.08


def test_best_fit_decreasing_against_brute_force():
    """Best-fit decreasing on small instances: every chunk placed once, no bin
    over capacity, and each chunk went to the fullest bin that could hold it at
    that moment (checked by replaying the placement)."""
    rng = np.random.default_rng(0)
    for _ in range(50):
        chunks = rng.integers(1, 20, size=rng.integers(1, 30)).tolist()
        bins = wl.best_fit_decreasing(chunks, 20)
        assert sorted(c for b in bins for c in b) == sorted(chunks)
        assert all(sum(b) <= 20 for b in bins)
        # replay: bins as lists of remaining capacity in creation order
        rem = []
        for c in sorted(chunks, reverse=True):
            feas = [k for k, r in enumerate(rem) if r >= c]
            if feas:
                k = min(feas, key=lambda k: (rem[k] - c, k))
                rem[k] -= c
            else:
                rem.append(20 - c)
        assert sorted(20 - r for r in rem) == sorted(sum(b) for b in bins)


def test_packed_dm_offsets_valid():
    for seed in range(4):
        off = wl.packed_dm_offsets(seed)
        assert off[0] == 0 and off[-1] == 8 * 8192 and np.all(np.diff(off) > 0)
        assert set(range(0, 8 * 8192 + 1, 8192)) <= set(off.tolist())
        # packing keeps documents whole far more often than concat-and-chunk
        assert len(wl.segment_lengths(8, 8192, off)) > 8
