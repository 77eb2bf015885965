"""Shared helpers for the GPU parity tests: seeded inputs, CUDA calls through
the C ABI, oracle references and error metrics."""
from __future__ import annotations

import math

import numpy as np

from oracle import oracle as orc
from oracle import rope
from paper_2405_13226_gb300 import workloads as wl

# Tolerances: bf16 inputs, fp32 accumulation (O: max abs and relative L2; grads: relative L2).
TOL_O_MAX = 1e-2
TOL_O_REL = 5e-3
TOL_GRAD_REL = 1e-2
TOL_LSE_MAX = 2e-3


def rel_l2(x, ref, floor: float = 1e-3) -> float:
    """||x - ref|| / ||ref||, with the denominator floored at `floor` RMS per
    element: a reference that is exactly zero (e.g. dq, dk of a one-token
    document, where dS = dP - D = 0) is compared on an absolute scale."""
    ref = np.asarray(ref, np.float64)
    den = max(float(np.linalg.norm(ref)), floor * np.sqrt(ref.size))
    return float(np.linalg.norm(np.asarray(x, np.float64) - ref) / den)


def to_device(bits, device="cuda"):
    import torch
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).to(device)


def to_f64(t) -> np.ndarray:
    return t.float().cpu().numpy().astype(np.float64)


def bits_f64(bits) -> np.ndarray:
    return wl.bf16_bits_to_f32(bits).astype(np.float64)


def run_cuda(qb, kb, vb, gb, scale, offsets=None, device="cuda", rope_base=0.0, fused_rope=False, rotated=None):
    """fwd + bwd through the C ABI on bf16 bit arrays [B, L, H, d] (with
    rope_base > 0: rope_qk first, or with fused_rope the forward that rotates q, k
    itself; dq, dk with respect to the un-rotated q, k). `rotated`, a list, receives
    the fused forward's q_rot, k_rot."""
    import torch
    from paper_2405_13226_gb300 import ddattn
    q, k, v, g = (to_device(x, device) for x in (qb, kb, vb, gb))
    off = None if offsets is None else torch.from_numpy(np.asarray(offsets, np.int32)).to(device)
    B, L, H, d = q.shape
    desc = ddattn.make_desc(B, L, H, d, scale, off, rope_base)
    ws = ddattn.new_workspace(desc, q.device, for_bwd=True)
    if rope_base and fused_rope:
        o, lse, q, k = ddattn.fwd_rope(q, k, v, rope_base, scale, off, workspace=ws)
        if rotated is not None:
            rotated += [q, k]
    elif rope_base:
        q, k = ddattn.rope_qk(q, k, rope_base)
    if not (rope_base and fused_rope):
        o, lse = ddattn.fwd(q, k, v, scale, off, workspace=ws)
    dq, dk, dv = ddattn.bwd(q, k, v, o, g, lse, scale, off, workspace=ws, rope_base=rope_base)
    torch.cuda.synchronize()
    st = ddattn.poll_status(ws)
    assert st == 0, "device status %d" % st
    return o, lse, dq, dk, dv


def rope_inputs(q, k, rope_base):
    """[B, L, H, d] float64 q, k -> the bf16-rounded rotated q, k the attention sees."""
    return rope.round_to_bf16(rope.rope_rotate(q, rope_base)), rope.round_to_bf16(rope.rope_rotate(k, rope_base))


def oracle_full(qb, kb, vb, gb, scale, offsets=None, rope_base=0.0):
    """Oracle over every (b, h) slice. Returns arrays in [B, L, H, d] / [B, H, L]."""
    B, L, H, d = qb.shape
    q, k, v, g = (bits_f64(x) for x in (qb, kb, vb, gb))
    if rope_base:
        q, k = rope_inputs(q, k, rope_base)
    q, k, v, g = (x.transpose(0, 2, 1, 3).reshape(B * H, L, d) for x in (q, k, v, g))
    doc = np.stack([orc.doc_ids(L, b, offsets) for b in range(B) for _ in range(H)])
    o, lse = orc.attn_fwd(q, k, v, doc, scale)
    dq, dk, dv = orc.attn_bwd(q, k, v, g, doc, scale)
    back = lambda x: x.reshape(B, H, L, d).transpose(0, 2, 1, 3)
    dq, dk = back(dq), back(dk)
    if rope_base:
        dq, dk = rope.rope_unrotate(dq, rope_base), rope.rope_unrotate(dk, rope_base)
    return back(o), lse.reshape(B, H, L), dq, dk, back(dv)


def check_full(qb, kb, vb, gb, scale, offsets=None, rope_base=0.0, fused_rope=False, rotated=None):
    o, lse, dq, dk, dv = run_cuda(qb, kb, vb, gb, scale, offsets, rope_base=rope_base, fused_rope=fused_rope,
                                  rotated=rotated)
    ro, rlse, rdq, rdk, rdv = oracle_full(qb, kb, vb, gb, scale, offsets, rope_base)
    go = to_f64(o)
    errs = {
        "o_max": float(np.abs(go - ro).max()),
        "o_rel": rel_l2(go, ro),
        "lse_max": float(np.abs(to_f64(lse) - rlse).max()),
        "dq_rel": rel_l2(to_f64(dq), rdq),
        "dk_rel": rel_l2(to_f64(dk), rdk),
        "dv_rel": rel_l2(to_f64(dv), rdv),
    }
    assert errs["o_max"] <= TOL_O_MAX, errs
    assert errs["o_rel"] <= TOL_O_REL, errs
    assert errs["lse_max"] <= TOL_LSE_MAX, errs
    for key in ("dq_rel", "dk_rel", "dv_rel"):
        assert errs[key] <= TOL_GRAD_REL, errs
    return errs, (o, lse, dq, dk, dv)


def sample_rows(L: int, n_rand: int, seed: int) -> np.ndarray:
    fixed = [0, 1, 2, 63, 64, 127, 128, 129, L // 2, L - 129, L - 128, L - 2, L - 1]
    rnd = np.random.default_rng(seed).integers(0, L, size=n_rand).tolist()
    return np.array(sorted({r for r in fixed + rnd if 0 <= r < L}), dtype=np.int32)


def check_sampled(qb, kb, vb, gb, scale, slices, offsets=None, n_rand=8, gpu=None, rope_base=0.0,
                  fused_rope=False):
    """Full-size GPU run (or `gpu` results), oracle on sampled rows of (b, h) slices."""
    if gpu is None:
        gpu = run_cuda(qb, kb, vb, gb, scale, offsets, rope_base=rope_base, fused_rope=fused_rope)
    o, lse, dq, dk, dv = (to_f64(t) for t in gpu)
    B, L, H, d = qb.shape
    acc = {k: ([], []) for k in ("o", "lse", "dq", "dk", "dv")}
    for (b, h) in slices:
        sl = lambda x: bits_f64(x[b, :, h, :])
        q, k, v, g = sl(qb), sl(kb), sl(vb), sl(gb)
        if rope_base:
            q, k = (x[0, :, 0] for x in rope_inputs(q[None, :, None], k[None, :, None], rope_base))
        doc = orc.doc_ids(L, b, offsets)
        rows = sample_rows(L, n_rand, seed=b * 1000 + h)
        ro, rlse = orc.attn_fwd_rows(q, k, v, doc, scale, rows)
        rdq, rdk, rdv = orc.attn_bwd_rows(q, k, v, g, doc, scale, rows, rows)
        if rope_base:
            # R^T at the sampled positions: embed the rows at their positions of a zero slice
            full = np.zeros((2, L, d))
            full[0, rows], full[1, rows] = rdq, rdk
            un = rope.rope_unrotate(full[:, :, None], rope_base)[:, :, 0]
            rdq, rdk = un[0, rows], un[1, rows]
        acc["o"][0].append(o[b, rows, h]); acc["o"][1].append(ro)
        acc["lse"][0].append(lse[b, h, rows]); acc["lse"][1].append(rlse)
        acc["dq"][0].append(dq[b, rows, h]); acc["dq"][1].append(rdq)
        acc["dk"][0].append(dk[b, rows, h]); acc["dk"][1].append(rdk)
        acc["dv"][0].append(dv[b, rows, h]); acc["dv"][1].append(rdv)
    cat = {k: (np.concatenate(a), np.concatenate(r)) for k, (a, r) in acc.items()}
    errs = {
        "o_max": float(np.abs(cat["o"][0] - cat["o"][1]).max()),
        "o_rel": rel_l2(*cat["o"]),
        "lse_max": float(np.abs(cat["lse"][0] - cat["lse"][1]).max()),
        "dq_rel": rel_l2(*cat["dq"]),
        "dk_rel": rel_l2(*cat["dk"]),
        "dv_rel": rel_l2(*cat["dv"]),
    }
    assert errs["o_max"] <= TOL_O_MAX, errs
    assert errs["o_rel"] <= TOL_O_REL, errs
    assert errs["lse_max"] <= TOL_LSE_MAX, errs
    for key in ("dq_rel", "dk_rel", "dv_rel"):
        assert errs[key] <= TOL_GRAD_REL, errs
    assert all(np.isfinite(t).all() for t in (o, lse, dq, dk, dv))
    return errs


def doc_start_rows(B: int, L: int, offsets=None):
    """(b, row) of every first token of a document segment."""
    out = []
    for b in range(B):
        doc = orc.doc_ids(L, b, offsets)
        starts = [0] + [i for i in range(1, L) if doc[i] != doc[i - 1]]
        out += [(b, i) for i in starts]
    return out


def default_scale(d: int) -> float:
    return 1.0 / math.sqrt(d)
