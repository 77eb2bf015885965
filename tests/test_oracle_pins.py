"""Pins of the fp64 oracle to facts other than itself (CPU only).

Each test fixes the oracle against something the paper or the mathematics
determines: finite differences, closed forms of special cases, invariants of
softmax attention, the document-mask definition (Sec. 1 / Sec. 3.5: DM means
no cross-document attention), brute-force enumeration, and an independent
library computation (torch fp64 autograd) on tiny shapes.
"""
import numpy as np
import pytest

from oracle import oracle as orc
from paper_2405_13226_gb300 import workloads as wl


def _rand(shape, seed):
    return np.random.default_rng(seed).standard_normal(shape)


def _docs_from_lengths(lengths):
    return np.concatenate([np.full(n, i, dtype=np.int32) for i, n in enumerate(lengths)])


CASES = [
    # (L, d, document lengths inside the sequence)
    (1, 3, [1]),
    (5, 4, [5]),
    (8, 2, [8]),
    (8, 4, [3, 1, 4]),
    (7, 3, [2, 2, 3]),
]


def _loss_and_grads(q, k, v, dO, doc, scale):
    o, _ = orc.attn_fwd(q[None], k[None], v[None], doc[None], scale)
    return float((o[0] * dO).sum())


@pytest.mark.parametrize("L,d,lens", CASES)
def test_finite_differences(L, d, lens):
    """Pin (i): the analytic dq, dk, dv equal central differences of sum(o * dO)."""
    doc = _docs_from_lengths(lens)
    q, k, v, dO = (_rand((L, d), s) for s in (1, 2, 3, 4))
    scale = 0.7
    dq, dk, dv = orc.attn_bwd(q[None], k[None], v[None], dO[None], doc[None], scale)
    h = 1e-6
    for name, x, g in (("q", q, dq[0]), ("k", k, dk[0]), ("v", v, dv[0])):
        num = np.zeros_like(x)
        for idx in np.ndindex(x.shape):
            xp = x.copy(); xp[idx] += h
            xm = x.copy(); xm[idx] -= h
            args_p = dict(q=q, k=k, v=v); args_p[name] = xp
            args_m = dict(q=q, k=k, v=v); args_m[name] = xm
            fp = _loss_and_grads(args_p["q"], args_p["k"], args_p["v"], dO, doc, scale)
            fm = _loss_and_grads(args_m["q"], args_m["k"], args_m["v"], dO, doc, scale)
            num[idx] = (fp - fm) / (2 * h)
        rel = np.linalg.norm(num - g) / max(np.linalg.norm(num), 1e-30)
        assert rel < 1e-6, (name, rel)


def test_rows_sum_to_one():
    """Pin (ii): with v = 1 every output component is sum_j P_ij, which must be 1."""
    L, d = 40, 8
    doc = _docs_from_lengths([7, 1, 20, 12])
    q, k = _rand((L, d), 5) * 3, _rand((L, d), 6) * 3
    v = np.ones((L, d))
    o, _ = orc.attn_fwd(q[None], k[None], v[None], doc[None], 0.5)
    assert np.abs(o - 1.0).max() < 1e-12


def test_document_mask_equals_separate_causal_runs():
    """Pin (iii): DM attention over a concatenated chunk equals independent causal
    attention over each document (the meaning of document masking)."""
    lens = [5, 1, 13, 9, 4]
    L, d = sum(lens), 6
    doc = _docs_from_lengths(lens)
    q, k, v, dO = (_rand((L, d), s) for s in (7, 8, 9, 10))
    scale = 1 / np.sqrt(d)
    o, lse = orc.attn_fwd(q[None], k[None], v[None], doc[None], scale)
    dq, dk, dv = orc.attn_bwd(q[None], k[None], v[None], dO[None], doc[None], scale)
    s = 0
    for n in lens:
        sl = slice(s, s + n)
        one = np.zeros((1, n), dtype=np.int32)
        o1, lse1 = orc.attn_fwd(q[None, sl], k[None, sl], v[None, sl], one, scale)
        g1 = orc.attn_bwd(q[None, sl], k[None, sl], v[None, sl], dO[None, sl], one, scale)
        np.testing.assert_allclose(o[0, sl], o1[0], rtol=0, atol=1e-13)
        np.testing.assert_allclose(lse[0, sl], lse1[0], rtol=0, atol=1e-13)
        for a, b in zip((dq, dk, dv), g1):
            np.testing.assert_allclose(a[0, sl], b[0], rtol=0, atol=1e-13)
        s += n


def test_single_key_rows():
    """Pin (iv): the first token of every document sees only itself: o = v, LSE = s_ii."""
    lens = [4, 1, 6]
    L, d = sum(lens), 5
    doc = _docs_from_lengths(lens)
    q, k, v = (_rand((L, d), s) for s in (11, 12, 13))
    scale = 0.3
    o, lse = orc.attn_fwd(q[None], k[None], v[None], doc[None], scale)
    for start in np.cumsum([0] + lens[:-1]):
        np.testing.assert_array_equal(o[0, start], v[start])
        assert lse[0, start] == pytest.approx(scale * q[start] @ k[start], abs=1e-14)


def test_uniform_attention_closed_form():
    """Pin (v): q = 0 gives uniform weights: o_i = mean of v over A(i), LSE_i = ln|A(i)|."""
    lens = [3, 9, 1, 7]
    L, d = sum(lens), 4
    doc = _docs_from_lengths(lens)
    q = np.zeros((L, d))
    k, v = _rand((L, d), 14), _rand((L, d), 15)
    o, lse = orc.attn_fwd(q[None], k[None], v[None], doc[None], 1.0)
    start = 0
    for n in lens:
        for r in range(n):
            i = start + r
            np.testing.assert_allclose(o[0, i], v[start:i + 1].mean(axis=0), atol=1e-14)
            assert lse[0, i] == pytest.approx(np.log(r + 1), abs=1e-14)
        start += n


def test_key_shift_invariance():
    """Pin (vi): adding one vector to every key of a document shifts each score row
    by a constant, so o is unchanged; hence the dk of each document sums to 0."""
    lens = [6, 10]
    L, d = sum(lens), 4
    doc = _docs_from_lengths(lens)
    q, k, v, dO = (_rand((L, d), s) for s in (16, 17, 18, 19))
    c = _rand((d,), 20) * 2
    o, _ = orc.attn_fwd(q[None], k[None], v[None], doc[None], 0.8)
    o2, _ = orc.attn_fwd(q[None], (k + c)[None], v[None], doc[None], 0.8)
    np.testing.assert_allclose(o, o2, atol=1e-12)
    _, dk, _ = orc.attn_bwd(q[None], k[None], v[None], dO[None], doc[None], 0.8)
    s = 0
    for n in lens:
        assert np.abs(dk[0, s:s + n].sum(axis=0)).max() < 1e-12
        s += n


def test_torch_fp64_autograd_cross_check():
    """Pin (viii): an independent library computation -- torch fp64 masked softmax
    attention with autograd -- on tiny causal and document-masked inputs."""
    torch = pytest.importorskip("torch")
    for lens, d in (([9], 4), ([3, 5, 1], 3), ([2, 2, 2, 2], 5)):
        L = sum(lens)
        doc = _docs_from_lengths(lens)
        q, k, v, dO = (_rand((L, d), s) for s in (21, 22, 23, 24))
        scale = 0.9
        tq, tk, tv = (torch.tensor(x, requires_grad=True) for x in (q, k, v))
        idx = torch.arange(L)
        tdoc = torch.tensor(doc)
        allowed = (idx[None, :] <= idx[:, None]) & (tdoc[None, :] == tdoc[:, None])
        s = (tq @ tk.T) * scale
        s = s.masked_fill(~allowed, float("-inf"))
        tlse = torch.logsumexp(s, dim=-1)
        to = torch.softmax(s, dim=-1) @ tv
        (to * torch.tensor(dO)).sum().backward()
        o, lse = orc.attn_fwd(q[None], k[None], v[None], doc[None], scale)
        dq, dk, dv = orc.attn_bwd(q[None], k[None], v[None], dO[None], doc[None], scale)
        np.testing.assert_allclose(o[0], to.detach().numpy(), atol=1e-12)
        np.testing.assert_allclose(lse[0], tlse.detach().numpy(), atol=1e-12)
        np.testing.assert_allclose(dq[0], tq.grad.numpy(), atol=1e-12)
        np.testing.assert_allclose(dk[0], tk.grad.numpy(), atol=1e-12)
        np.testing.assert_allclose(dv[0], tv.grad.numpy(), atol=1e-12)


def test_pair_count_brute_force():
    """Pin (vii): enumerating the mask gives sum over segments of l(l+1)/2, the
    count the flop convention uses; for a DD step it is T(L+1)/2, linear in L."""
    off = wl.concat_and_chunk_offsets(seed=3, n_chunks=2, chunk=512)
    B, L = 2, 512
    brute = sum(orc.live_pairs(orc.doc_ids(L, b, off)) for b in range(B))
    assert brute == wl.live_pairs(B, L, off)
    for Lb in (1, 2, 7, 64):
        assert orc.live_pairs(orc.doc_ids(Lb, 0, None)) == Lb * (Lb + 1) // 2
    T = wl.TOKENS_PER_STEP
    for Lb in wl.BUCKETS:
        assert wl.live_pairs(T // Lb, Lb) == T * (Lb + 1) // 2


def test_doc_ids_follow_offsets_and_sequence_cuts():
    """Documents follow cu_doc_offsets; a document straddling a sequence boundary
    continues as a separate segment in the next sequence."""
    off = np.array([0, 3, 10, 16], dtype=np.int32)      # B=2, L=8: doc 1 spans tokens 3..9
    d0 = orc.doc_ids(8, 0, off)
    d1 = orc.doc_ids(8, 1, off)
    assert list(d0) == [0, 0, 0, 1, 1, 1, 1, 1]
    assert list(d1) == [1, 1, 2, 2, 2, 2, 2, 2]


def test_rows_and_full_agree():
    """The sampled-row entry points compute the same values as the full slice."""
    lens = [30, 2, 40]
    L, d = sum(lens), 8
    doc = _docs_from_lengths(lens)
    q, k, v, dO = (_rand((L, d), s) for s in (31, 32, 33, 34))
    o, lse = orc.attn_fwd(q[None], k[None], v[None], doc[None], 0.4)
    dq, dk, dv = orc.attn_bwd(q[None], k[None], v[None], dO[None], doc[None], 0.4)
    rows = np.array([0, 5, 31, 33, 71], dtype=np.int32)
    o_r, lse_r = orc.attn_fwd_rows(q, k, v, doc, 0.4, rows)
    dq_r, dk_r, dv_r = orc.attn_bwd_rows(q, k, v, dO, doc, 0.4, rows, rows[::-1])
    np.testing.assert_allclose(o_r, o[0, rows], atol=1e-14)
    np.testing.assert_allclose(lse_r, lse[0, rows], atol=1e-14)
    np.testing.assert_allclose(dq_r, dq[0, rows], atol=1e-14)
    np.testing.assert_allclose(dk_r, dk[0, rows[::-1]], atol=1e-14)
    np.testing.assert_allclose(dv_r, dv[0, rows[::-1]], atol=1e-14)
