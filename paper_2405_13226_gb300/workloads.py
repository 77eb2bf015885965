"""Seeded synthetic workloads shaped like the paper's training steps.

This module only makes inputs (tensors, document offsets, bucket streams) and
the workload statistics used to report them. It holds none of the attention
arithmetic; both the CUDA path's tests/bench and the fp64 oracle draw their
inputs from here.

Stand-ins: the paper trains on RefinedWeb (Sec. 3, ~525B tokens) whose length
distribution only appears as plots (Fig. 3). Document lengths here are drawn
from a lognormal(mu=6.0, sigma=1.3) model (natural-log parameters), rounded
half-to-even and clamped to [16, 65536] tokens.
"""
from __future__ import annotations

import numpy as np

# Tensor ids of the per-tensor random streams.
Q, K, V, DO = 0, 1, 2, 3

TOKENS_PER_STEP = 65536          # b = 8 x 8192 tokens per optimisation step (Sec. 3.1)
BUCKETS = (256, 512, 1024, 2048, 4096, 8192)


def _rng(seed: int, stream: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([int(seed), int(stream)])))


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 to bfloat16, nearest-even; returns the uint16 bit patterns."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    lsb = (u >> np.uint32(16)) & np.uint32(1)
    r = (u + np.uint32(0x7FFF) + lsb) >> np.uint32(16)
    return r.astype(np.uint16)


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    return (np.ascontiguousarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def normal_bf16(shape, seed: int, tensor_id: int, mult: float = 1.0) -> np.ndarray:
    """i.i.d. N(0,1) in fp32 (times `mult`, in fp32), rounded to bf16 bits."""
    x = _rng(seed, tensor_id).standard_normal(size=shape, dtype=np.float32)
    if mult != 1.0:
        x = x * np.float32(mult)
    return f32_to_bf16_bits(x)


def attn_inputs(B: int, L: int, H: int, d: int, seed: int = 0, qk_mult: float = 1.0):
    """q, k, v, dO as bf16 bit arrays of shape [B, L, H, d] (token-major)."""
    shape = (B, L, H, d)
    return (normal_bf16(shape, seed, Q, qk_mult), normal_bf16(shape, seed, K, qk_mult),
            normal_bf16(shape, seed, V), normal_bf16(shape, seed, DO))


# ----------------------------------------------------------------- documents
def lognormal_doc_lengths(rng: np.random.Generator, n: int, mu: float = 6.0, sigma: float = 1.3,
                          lo: int = 16, hi: int = 65536) -> np.ndarray:
    x = rng.lognormal(mean=mu, sigma=sigma, size=n)
    return np.clip(np.rint(x), lo, hi).astype(np.int64)


def concat_and_chunk_offsets(seed: int, n_chunks: int = 8, chunk: int = 8192) -> np.ndarray:
    """Concat-and-chunk baseline (Sec. 1): shuffle documents, concatenate, cut
    into `chunk`-token sequences. Returns int32 cu_doc_offsets over the
    flattened n_chunks*chunk tokens: every document start plus every chunk
    boundary (a document cut by a boundary continues as a new segment), from 0
    to n_chunks*chunk. The <EOT> separator is counted inside each length."""
    total = n_chunks * chunk
    rng = _rng(seed, 100)
    lengths = []
    acc = 0
    while acc < total:
        ln = int(lognormal_doc_lengths(rng, 1)[0])
        lengths.append(ln)
        acc += ln
    lengths = np.array(lengths, dtype=np.int64)
    rng.shuffle(lengths)
    starts = np.concatenate([[0], np.cumsum(lengths)[:-1]])
    starts = starts[starts < total]
    bounds = np.arange(0, total + 1, chunk, dtype=np.int64)
    off = np.union1d(starts, bounds)
    return off.astype(np.int32)


def binary_decompose(length: int) -> list[int]:
    """Sec. 2.1: a document of length l = 2^i1 + ... + 2^ik is cut into adjacent
    pieces of those lengths (largest first)."""
    out = []
    bit = 1 << max(int(length).bit_length() - 1, 0)
    while bit:
        if length & bit:
            out.append(bit)
        bit >>= 1
    return out


def dd_bucket_tokens(seed: int = 0, n_docs: int = 100_000, min_piece: int = 256,
                     max_piece: int = 8192) -> dict[int, int]:
    """Tokens per bucket D_i after binary decomposition of `n_docs` lognormal
    documents; pieces shorter than `min_piece` are dropped and pieces longer
    than `max_piece` are split into max_piece-token sequences."""
    lengths = lognormal_doc_lengths(_rng(seed, 200), n_docs)
    counts = {b: 0 for b in BUCKETS if min_piece <= b <= max_piece}
    for ln in lengths:
        for p in binary_decompose(int(ln)):
            if p < min_piece:
                continue
            if p > max_piece:
                counts[max_piece] += p
            else:
                counts[p] += p
    return counts


def curriculum_stream(seed: int = 0, steps: int = 200, bucket_tokens: dict[int, int] | None = None) -> list[int]:
    """Sequence length of each step: i.i.d. draws with probability proportional
    to each bucket's token count (a simplified form of Algorithm 1 with one
    cycle and odds equal to the natural mixture)."""
    if bucket_tokens is None:
        bucket_tokens = dd_bucket_tokens(seed)
    Ls = np.array(sorted(bucket_tokens))
    p = np.array([bucket_tokens[L] for L in Ls], dtype=np.float64)
    p /= p.sum()
    idx = _rng(seed, 300).choice(len(Ls), size=steps, p=p)
    return [int(Ls[i]) for i in idx]


# ----------------------------------------------------------------- Algorithm 1
# Sampling odds over D8..D13 of the paper's curricula (Table 2).
CURRICULA = {
    "Uniform": (1, 1, 1, 1, 1, 1),
    "Grow-Linear": (6, 5, 4, 3, 2, 1),
    "Grow-P2": (32, 16, 8, 4, 2, 1),
    "Grow-P100": (100 ** 5, 100 ** 4, 100 ** 3, 100 ** 2, 100, 1),
    "Shrink-P100": (1, 100, 100 ** 2, 100 ** 3, 100 ** 4, 100 ** 5),
}


def length_curriculum(bucket_tokens: dict[int, int], odds: dict[int, float], cycles: int,
                      tokens_per_step: int, seed: int = 0) -> list[int]:
    """Algorithm 1 (length-based sampling and curriculum): sequence length of
    every optimisation step.

    The n_i tokens of bucket D_i (sequences of length L = 2^i) are split into
    `cycles` disjoint subsets of n_i / c tokens. In each cycle, while some subset
    is non-empty: the odds of the non-empty subsets are normalised into
    probabilities, a bucket i is drawn with them, and b / 2^i sequences are
    taken from its subset without replacement (fewer if fewer remain)."""
    rng = _rng(seed, 400)
    Ls = sorted(bucket_tokens)
    per_cycle = {}
    for L in Ls:
        n_seq = bucket_tokens[L] // L
        base, extra = divmod(n_seq, cycles)
        per_cycle[L] = [base + (1 if j < extra else 0) for j in range(cycles)]
    steps = []
    for j in range(cycles):
        left = {L: per_cycle[L][j] for L in Ls}
        while any(left[L] > 0 for L in Ls):
            w = np.array([odds[L] if left[L] > 0 else 0.0 for L in Ls], dtype=np.float64)
            i = int(rng.choice(len(Ls), p=w / w.sum()))
            L = Ls[i]
            take = min(left[L], max(tokens_per_step // L, 1))
            left[L] -= take
            steps.append(L)
    return steps


# ----------------------------------------------------------------- best-fit packing
def best_fit_decreasing(chunk_lengths, capacity: int) -> list[list[int]]:
    """Appendix "Comparison to best-fit sequence packing": chunks (each at most
    `capacity` tokens) sorted from largest to smallest; each goes to the
    feasible bin that is left with the least remaining capacity, or to a new
    bin when none can hold it. Returns the chunk lengths of every bin."""
    import bisect
    order = sorted((int(c) for c in chunk_lengths), reverse=True)
    rem_keys: list[tuple[int, int]] = []      # (remaining capacity, bin id), sorted
    bins: list[list[int]] = []
    for c in order:
        if c > capacity:
            raise ValueError("chunk longer than the bin capacity")
        k = bisect.bisect_left(rem_keys, (c, -1))  # smallest remaining >= c
        if k == len(rem_keys):
            bins.append([c])
            bisect.insort(rem_keys, (capacity - c, len(bins) - 1))
        else:
            rem, bid = rem_keys.pop(k)
            bins[bid].append(c)
            bisect.insort(rem_keys, (rem - c, bid))
    return bins


def packed_dm_offsets(seed: int, n_chunks: int = 8, chunk: int = 8192, n_docs: int = 4000) -> np.ndarray:
    """Pack-8k+DM workload: lognormal documents cut into pieces of at most
    `chunk` tokens, packed by best-fit decreasing into `chunk`-token sequences
    whose unused tail is <PAD>. The first `n_chunks` bins form the step; each
    document piece and each pad tail is its own masked segment. Returns int32
    cu_doc_offsets over the n_chunks*chunk tokens."""
    lengths = lognormal_doc_lengths(_rng(seed, 500), n_docs)
    pieces = []
    for ln in lengths:
        while ln > chunk:
            pieces.append(chunk)
            ln -= chunk
        pieces.append(int(ln))
    bins = best_fit_decreasing(pieces, chunk)
    rng = _rng(seed, 501)
    pick = rng.permutation(len(bins))[:n_chunks]
    offs = [0]
    for k, bi in enumerate(pick):
        pos = k * chunk
        for c in bins[bi]:
            pos += c
            offs.append(pos)
        if pos < (k + 1) * chunk:          # pad tail
            offs.append((k + 1) * chunk)
    return np.unique(np.array(offs, dtype=np.int64)).astype(np.int32)


# ----------------------------------------------------------------- statistics
def segment_lengths(B: int, L: int, cu_doc_offsets=None) -> np.ndarray:
    """Lengths of the attention segments of a step: documents cut at sequence
    boundaries (one segment per sequence when there are no offsets)."""
    if cu_doc_offsets is None:
        return np.full(B, L, dtype=np.int64)
    cuts = np.union1d(np.asarray(cu_doc_offsets, dtype=np.int64), np.arange(0, B * L + 1, L))
    seg = np.diff(cuts)
    return seg[seg > 0]


def avg_sequence_length(lengths) -> float:
    """Appendix, average sequence length: mean of the l_i."""
    lengths = np.asarray(lengths, dtype=np.float64)
    return float(lengths.mean())


def avg_context_length(lengths) -> float:
    """Appendix, Eq. (avg_context): sum_i l_i(l_i-1) / (2 sum_i l_i)."""
    lengths = np.asarray(lengths, dtype=np.float64)
    return float((lengths * (lengths - 1)).sum() / (2.0 * lengths.sum()))


def live_pairs(B: int, L: int, cu_doc_offsets=None) -> int:
    """Causal (query, key) pairs of one call: sum over segments of l(l+1)/2."""
    seg = segment_lengths(B, L, cu_doc_offsets)
    return int((seg * (seg + 1) // 2).sum())


def attn_flops(B: int, L: int, H: int, d: int, cu_doc_offsets=None, fwd: bool = True, bwd: bool = True) -> int:
    """Algorithmic flops: per live pair and head, 2 contractions of length d
    forward (4d) and 5 backward including the score recompute (10d)."""
    per_pair = (4 * d if fwd else 0) + (10 * d if bwd else 0)
    return per_pair * H * live_pairs(B, L, cu_doc_offsets)


def attn_min_bytes(B: int, L: int, H: int, d: int, fwd: bool = True, bwd: bool = True) -> int:
    """Minimal HBM bytes: each bf16 tensor of B*L*H*d read or written once
    (forward: q,k,v read, o written; backward: q,k,v,o,dO read, dq,dk,dv
    written) plus the fp32 LSE (written forward, read backward)."""
    t = B * L * H * d * 2
    lse = B * L * H * 4
    return (4 * t + lse if fwd else 0) + (8 * t + lse if bwd else 0)
