"""Benchmark: causal attention fwd+bwd on GB300 through the C ABI (libddattn.so).

Headline workload: the 1B-model bucket sweep -- H=16, d=128, 65536 tokens per
call, L in {256, ..., 8192} with B = 65536 / L. One step = forward + backward
of one 65536-token batch of every bucket (6 calls of each). `value` is the
algorithmic TFLOP/s over the step (14 d H sum_seq L(L+1)/2 flops per call).
Also reported: per-bucket ms and TFLOP/s, the document-masked 8x8192
concat-and-chunk step (16 seeds), the Pack-8k+DM step, an Algorithm 1
stream (Grow-P2, 8 cycles) and every Table 2 curriculum, the sweep with RoPE
(f_b = 100k), the 3B (H=32, d=80) and 7B (H=32, d=128) head shapes, the
long-context bucket (B=4, L=16384, H=32), the roofline of the dominant kernel,
an end-to-end number through host buffers, and the fp64 oracle's throughput on
this host's cores.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
Multi-GPU: one process per GPU under torchrun; each rank runs its own
replica of the workload (attention has no exchange step), scaling "weak".
"""
from __future__ import annotations

import argparse
import json
import math
import os
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2405_13226_gb300 import workloads as wl  # noqa: E402

H, D = 16, 128
T = wl.TOKENS_PER_STEP
PEAKS_FALLBACK = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


def kernel_source_sha1() -> str:
    import hashlib
    h = hashlib.sha1()
    for f in ("attn_bwd_d128.cu", "attn_bwd_d128_persist.cu", "bwd_d128.cuh", "common.cuh", "ptx.cuh"):
        with open(os.path.join(ROOT, "paper_2405_13226_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()


def measured_traffic():
    """Mean DRAM bytes per launch of the backward main kernel over the sweep,
    from the committed ncu summary, if it was taken on the current sources."""
    p = os.path.join(ROOT, "profiles", "attn_kernels_sweep_traffic.md")
    if not os.path.exists(p):
        return None
    txt = open(p).read()
    if "source_sha1 (attn_bwd_d128.cu + attn_bwd_d128_persist.cu + bwd_d128.cuh + common.cuh + ptx.cuh): " + kernel_source_sha1() not in txt:
        return None
    vals = []
    for line in txt.splitlines():
        f = [x.strip() for x in line.split("|")]
        if len(f) > 5 and f[2] in ("attn_bwd_main_d128_kernel", "attn_bwd_main_d128_persist_kernel"):
            vals.append(float(f[5]))
    return sum(vals) / len(vals) if vals else None


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            return json.load(f), "measured"
    return PEAKS_FALLBACK, "fallback"


# ------------------------------------------------------------------ dist
def dist_setup(n_gpus, backend=None):
    """Rank, world size and local rank from the torchrun environment; for N > 1
    one process group over NCCL (one GPU per rank), or `backend` if given
    (the CPU tests use gloo)."""
    import torch
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    backend = backend or "nccl"
    if world > 1:
        import torch.distributed as dist
        if backend == "nccl":
            torch.cuda.set_device(local)
            dist.init_process_group("nccl", device_id=torch.device("cuda", local))
        else:
            dist.init_process_group(backend)
    elif backend == "nccl":
        torch.cuda.set_device(0)
    return rank, world, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x, world):
    """The slowest rank's time: every rank's CUDA-event time, reduced with MAX."""
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def replica_value(flops_per_step, steps, total_ms, world):
    """Whole-job TFLOP/s of N replicas: every rank runs the same per-rank
    workload (weak scaling), timed by the slowest rank."""
    return world * flops_per_step * steps / (total_ms * 1e-3) / 1e12


# ------------------------------------------------------------------ clocks
class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during a region."""

    Q = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), "--query-gpu=" + self.Q,
                                          "--format=csv,noheader,nounits", "-lms", "50"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *a):
        self.lines = []
        if self.proc is not None:
            self.proc.terminate()
            try:
                out, _ = self.proc.communicate(timeout=5)
            except Exception:
                self.proc.kill()
                out, _ = self.proc.communicate()
            self.lines = [l for l in out.splitlines() if l.strip()]

    def summary(self):
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for l in getattr(self, "lines", []):
            f = [x.strip() for x in l.split(",")]
            if len(f) < 7:
                continue
            try:
                sm.append(float(f[0]))
                mx = float(f[1])
            except ValueError:
                continue
            for n, v in zip(names, f[3:7]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": mx, "reasons": [], "samples": 0}
        return {"sm_mhz": float(np.median(sm)), "sm_max_mhz": mx, "reasons": sorted(reasons), "samples": len(sm)}


def smi_index(local: int) -> str:
    """nvidia-smi -i argument of this process's GPU (physical index or UUID)."""
    vis = os.environ.get("CUDA_VISIBLE_DEVICES")
    if vis:
        ent = [x.strip() for x in vis.split(",") if x.strip()]
        if local < len(ent):
            return ent[local]
    return str(local)


# ------------------------------------------------------------------ CPU oracle
def oracle_sample(max_seconds=15.0, rows_cap=None):
    """Time the fp64 oracle on slices of the bucket sweep: head h of sequence 0
    for every bucket, h = 0, 1, ..., until `max_seconds` of CPU work."""
    from oracle import oracle as orc
    orc.build()
    qb, kb, vb, gb = wl.attn_inputs(1, max(wl.BUCKETS), 4, D, seed=0)
    done_flops, spent, parts = 0, 0.0, []
    for h in range(4):
        for L in wl.BUCKETS:
            f64 = lambda x: wl.bf16_bits_to_f32(x[0, :L, h, :]).astype(np.float64)[None]
            q, k, v, g = f64(qb), f64(kb), f64(vb), f64(gb)
            doc = np.zeros((1, L), np.int32)
            t0 = time.perf_counter()
            orc.attn_fwd(q, k, v, doc, 1 / math.sqrt(D))
            orc.attn_bwd(q, k, v, g, doc, 1 / math.sqrt(D))
            spent += time.perf_counter() - t0
            done_flops += wl.attn_flops(1, L, 1, D)
            parts.append("L=%d h=%d" % (L, h))
            if spent >= max_seconds:
                break
        if spent >= max_seconds:
            break
    threads = int(os.environ.get("OMP_NUM_THREADS", os.cpu_count() or 1))
    return {"value": done_flops / spent / 1e12, "unit": "TFLOP/s", "cores": threads, "kind": "oracle",
            "sample": "fp64 oracle fwd+bwd on (seq 0, head h) slices of the bucket sweep, L=256..8192, "
                      "h=0.. until %.0f s: %d slices, %.1f s, %.3g algorithmic flops" % (
                          max_seconds, len(parts), spent, done_flops),
            "seconds": spent}


# ------------------------------------------------------------------ GPU helpers
def to_dev(bits, dev):
    import torch
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).to(dev)


class Bucket:
    """Buffers of one call shape; inputs are views of shared [T, H, D] tensors."""

    def __init__(self, ddattn, q, k, v, g, B, L, Hh, offsets=None, ws=None, rope_base=0.0, qk_rot=None, Dh=D):
        import torch
        self.dd = ddattn
        self.B, self.L = B, L
        self.rope_base = rope_base
        shape = (B, L, Hh, Dh)
        self.q, self.k, self.v, self.g = (x.view(shape) for x in (q, k, v, g))
        if rope_base:
            # the attention reads the rotated q, k, written each step by the forward
            # (dd_attn_fwd_rope) or, in the separate form, by rope_qk
            self.q_raw, self.k_raw = self.q, self.k
            self.q, self.k = (x.view(shape) for x in qk_rot)
        self.o = torch.empty_like(self.q)
        self.lse = torch.empty((B, Hh, L), dtype=torch.float32, device=q.device)
        self.dq, self.dk, self.dv = (torch.empty_like(self.q) for _ in range(3))
        self.off = offsets
        self.desc = ddattn.make_desc(B, L, Hh, Dh, None, offsets, rope_base)
        self.ws = ws if ws is not None else ddattn.new_workspace(self.desc, q.device)
        self.flops = wl.attn_flops(B, L, Hh, Dh, None if offsets is None else offsets.cpu().numpy())
        self.flops_fwd = wl.attn_flops(B, L, Hh, Dh, None if offsets is None else offsets.cpu().numpy(), bwd=False)
        self.flops_bwd = self.flops - self.flops_fwd

    def rope(self, stream):
        self.dd.rope_qk(self.q_raw, self.k_raw, self.rope_base, self.q, self.k, stream)

    def fwd(self, stream):
        if self.rope_base:
            self.dd.fwd_rope(self.q_raw, self.k_raw, self.v, self.rope_base, None, self.off, self.o, self.lse, self.q,
                             self.k, self.ws, stream)
        else:
            self.dd.fwd(self.q, self.k, self.v, None, self.off, self.o, self.lse, self.ws, stream)

    def fwd_separate(self, stream):
        """RoPE as its own pass (rope_qk), then the plain forward on the rotated q, k."""
        self.rope(stream)
        self.dd.fwd(self.q, self.k, self.v, None, self.off, self.o, self.lse, self.ws, stream)

    def bwd(self, stream, phases=None):
        self.dd.bwd(self.q, self.k, self.v, self.o, self.g, self.lse, None, self.off, self.dq, self.dk, self.dv,
                    self.ws, stream, phases if phases is not None else self.dd.DD_BWD_ALL, self.rope_base)


def run_ours(args):
    import torch
    from paper_2405_13226_gb300 import ddattn

    rank, world, local = dist_setup(args.gpus)
    dev = torch.device("cuda", local if world > 1 else 0)
    peaks, peak_src = load_peaks()
    ddattn.lib()
    stream = torch.cuda.current_stream()

    # inputs: [T, H, D] bf16 per tensor (256 MiB each, larger than L2), seeded
    qb, kb, vb, gb = wl.attn_inputs(1, T, H, D, seed=rank)
    q, k, v, g = (to_dev(x, dev) for x in (qb, kb, vb, gb))
    sweep = [args.only_L] if args.only_L else list(wl.BUCKETS)
    rb = args.rope_base
    # one workspace sized for the largest bucket (RoPE tables grow with L)
    ws = ddattn.new_workspace(max((ddattn.make_desc(T // L, L, H, D, None, None, rb) for L in sweep),
                                  key=ddattn.workspace_size), dev)
    qk_rot = (torch.empty_like(q), torch.empty_like(k)) if rb else None
    buckets = [Bucket(ddattn, q, k, v, g, T // L, L, H, ws=ws, rope_base=rb, qk_rot=qk_rot) for L in sweep]
    for bk in buckets:   # one correctness-agnostic pass so every instance is loaded
        bk.fwd(stream); bk.bwd(stream)
    torch.cuda.synchronize()

    E = lambda: torch.cuda.Event(enable_timing=True)
    nb = len(buckets)
    # events: per step, per bucket: [start, after fwd, after pre, after main, after post]
    ev = [[[E() for _ in range(5)] for _ in range(nb)] for _ in range(args.steps)]

    def step(evs=None):
        for i, bk in enumerate(buckets):
            if evs: evs[i][0].record(stream)
            bk.fwd(stream)
            if evs: evs[i][1].record(stream)
            bk.bwd(stream, ddattn.DD_BWD_PRE)
            if evs: evs[i][2].record(stream)
            bk.bwd(stream, ddattn.DD_BWD_MAIN)
            if evs: evs[i][3].record(stream)
            bk.bwd(stream, ddattn.DD_BWD_POST)
            if evs: evs[i][4].record(stream)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    barrier(world)
    t_start, t_end = E(), E()
    with ClockSampler(smi_index(local)) as clk:
        torch.cuda.synchronize()
        t_start.record(stream)
        for s in range(args.steps):
            step(ev[s])
        t_end.record(stream)
        torch.cuda.synchronize()
    barrier(world)
    total_ms = max_over_ranks(t_start.elapsed_time(t_end), world)
    st = ddattn.poll_status(ws)
    if st != 0:
        raise RuntimeError("device status %d (%s)" % (st, ddattn.status_string(st)))

    step_flops = sum(bk.flops for bk in buckets)
    ms_per_step = total_ms / args.steps
    value = replica_value(step_flops, args.steps, total_ms, world)

    per_bucket, fwd_t, main_t, main_flops = [], 0.0, 0.0, 0
    for i, bk in enumerate(buckets):
        ms = [ev[s][i][0].elapsed_time(ev[s][i][4]) for s in range(args.steps)]
        f_ms = [ev[s][i][0].elapsed_time(ev[s][i][1]) for s in range(args.steps)]
        m_ms = [ev[s][i][2].elapsed_time(ev[s][i][3]) for s in range(args.steps)]
        b_ms = [ev[s][i][1].elapsed_time(ev[s][i][4]) for s in range(args.steps)]
        fwd_t += sum(f_ms); main_t += sum(m_ms); main_flops += bk.flops_bwd * args.steps
        per_bucket.append({
            "L": bk.L, "B": bk.B, "ms": float(np.median(ms)), "fwd_ms": float(np.median(f_ms)),
            "bwd_ms": float(np.median(b_ms)), "bwd_main_ms": float(np.median(m_ms)),
            "tflops": bk.flops / (np.median(ms) * 1e-3) / 1e12,
            "fwd_tflops": bk.flops_fwd / (np.median(f_ms) * 1e-3) / 1e12,
            "bwd_main_tflops": bk.flops_bwd / (np.median(m_ms) * 1e-3) / 1e12,
            "frac_of_measured_sustained": bk.flops / (np.median(ms) * 1e-3) / 1e12 / peaks["bf16_tflops_sustained"],
            "min_hbm_GBps": wl.attn_min_bytes(bk.B, bk.L, H, D) / (np.median(ms) * 1e-3) / 1e9,
        })
    # dominant kernel over the timed region: the backward main kernel
    main_ach = main_flops / (main_t * 1e-3) / 1e12
    peak = peaks["bf16_tflops_sustained"]
    roofline = {"kernel": "attn_bwd_main (d=128: walking kernel for L <= 2048, per-key-tile kernel above)", "bound": "tensor", "achieved": main_ach, "peak": peak,
                "unit": "TFLOP/s", "frac": main_ach / peak, "traffic": measured_traffic(),
                "traffic_note": "read from profiles/attn_kernels_sweep_traffic.md, not measured in this run: "
                                "mean dram__bytes_read+write per launch over the six buckets from an ncu "
                                "capture of this kernel alone (its first six launches), taken on the sources "
                                "whose hash that file records; null if the sources changed since",
                "peak_kind": "bf16_tflops_sustained (%s)" % peak_src,
                "share_of_step": main_t / total_ms,
                "fwd_kernel_tflops": sum(bk.flops_fwd for bk in buckets) * args.steps / (fwd_t * 1e-3) / 1e12,
                "units": "10*d*H flops per live (q,k) pair per launch (backward algorithmic count)"}

    extras = {}
    if not args.quick:
        extras = extra_workloads(ddattn, q, k, v, g, buckets, ws, stream, peaks, dev)
    e2e = None if args.no_e2e else e2e_measure(ddattn, qb, kb, vb, gb, buckets, stream, dev, args, world)
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu:
        cpu = oracle_sample(args.cpu_seconds)

    line = {
        "metric": "causal attn fwd+bwd TFLOP/s (algorithmic, 14*d*H*sum L(L+1)/2 per call) over the bucket sweep",
        "value": value, "unit": "TFLOP/s", "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16 in, fp32 accumulate", "data": "synthetic (seeded N(0,1) bf16 q,k,v,dO)",
        "config": {"workload": "bucket sweep L=256..8192, 65536 tokens per call, H=16, d=128, causal; "
                               "step = fwd+bwd of every bucket (6 calls)",
                   "tokens_per_call": T, "H": H, "d": D, "buckets": sweep, "rope_base": args.rope_base,
                   "l2": "inputs larger than L2 (4 x 256 MiB bf16 tensors)", "parallelism": "replicas" if world > 1 else "1 GPU"},
        "ms_per_64k_token_step_by_bucket": {str(p["L"]): p["ms"] for p in per_bucket},
        "per_bucket": per_bucket,
        "roofline": roofline,
        "cpu_baseline": cpu,
        "e2e": e2e,
        # per bucket call: forward, backward pre / main / post; with RoPE the forward's and the
        # backward's (cos, sin) table fills and, above 512 tokens, the forward's k pass. For
        # L <= 256 the backward main kernel writes dq itself and post launches nothing.
        "gpu_launches": args.steps * sum(bwd_launches(bk.L, D) + 1
                                         + ((2 + (1 if bk.L > 512 else 0)) if args.rope_base else 0)
                                         for bk in buckets),
        "clocks": clk.summary(),
    }
    line.update(extras)
    if rank == 0:
        print(json.dumps(line))
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def bwd_launches(L: int, d: int) -> int:
    """Kernels one backward call launches: pre, main and post, except that for sequences of
    at most two 128-key tiles at d = 80 / 128 the main kernel writes dq itself (no post)."""
    return 2 if d != 64 and (L + 127) // 128 <= 2 else 3


def dm_pair_fractions(n_seeds: int) -> np.ndarray:
    """Live-pair fraction (vs plain causal) of the 8 x 8192 concat-and-chunk step for
    seeds 0 .. n_seeds - 1 (host only)."""
    full = wl.live_pairs(8, 8192)
    return np.array([wl.live_pairs(8, 8192, wl.concat_and_chunk_offsets(sd)) / full for sd in range(n_seeds)])


def time_calls(fn, reps, warm, stream):
    import torch
    for _ in range(warm):
        fn()
    s, e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    s.record(stream)
    for _ in range(reps):
        fn()
    e.record(stream)
    torch.cuda.synchronize()
    return s.elapsed_time(e) / reps


def extra_workloads(ddattn, q, k, v, g, buckets, ws, stream, peaks, dev):
    import torch
    out = {}
    # concat-and-chunk baseline with document masking, 16 seeds
    dm = []
    for seed in range(16):
        off_np = wl.concat_and_chunk_offsets(seed)
        off = torch.from_numpy(off_np).to(dev)
        bk = Bucket(ddattn, q, k, v, g, 8, 8192, H, offsets=off, ws=ws)
        ms = time_calls(lambda: (bk.fwd(stream), bk.bwd(stream)), 10, 3, stream)
        frac = wl.live_pairs(8, 8192, off_np) / wl.live_pairs(8, 8192)
        dm.append({"seed": seed, "ms": ms, "pair_fraction": frac, "tflops": bk.flops / (ms * 1e-3) / 1e12,
                   "segments": int(len(wl.segment_lengths(8, 8192, off_np)))})
    dm_mean = float(np.mean([x["ms"] for x in dm]))
    dm_flops = float(np.mean([wl.attn_flops(8, 8192, H, D, wl.concat_and_chunk_offsets(sd)) for sd in range(16)]))
    # the pair fraction's distribution over many seeds (host only): seeds 0..15 sit below its mean
    frac_many = dm_pair_fractions(1000)
    out["dm_baseline"] = {"workload": "8 chunks x 8192, H=16, d=128, document-masked, seeds 0..15; "
                                      "10 timed fwd+bwd calls after 3 warm-up calls per seed",
                          "ms_per_step_mean": dm_mean, "tflops": dm_flops / (dm_mean * 1e-3) / 1e12,
                          "pair_fraction_mean_16_seeds": float(np.mean([x["pair_fraction"] for x in dm])),
                          "pair_fraction_1000_seeds": {"mean": float(frac_many.mean()),
                                                       "median": float(np.median(frac_many)),
                                                       "min": float(frac_many.min()), "max": float(frac_many.max())},
                          "per_seed": dm}
    causal_8k = wl.attn_flops(8, 8192, H, D)
    # Algorithm 1 stream: Grow-P2 odds (Table 2), 8 cycles, bucket token counts
    # scaled to about 200 full steps of 65536 tokens (whole steps in every cycle)
    counts = wl.dd_bucket_tokens(0)
    tot = sum(counts.values())
    sched = {L: max(1, round(c / tot * 25)) * 8 * T for L, c in counts.items()}
    stream_L = wl.length_curriculum(sched, dict(zip(wl.BUCKETS, wl.CURRICULA["Grow-P2"])), 8, T, seed=0)
    by_L = {bk.L: bk for bk in buckets}
    torch.cuda.synchronize()
    s, e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    s.record(stream)
    for L in stream_L:
        by_L[L].fwd(stream)
        by_L[L].bwd(stream)
    e.record(stream)
    torch.cuda.synchronize()
    cur_ms = s.elapsed_time(e) / len(stream_L)
    cur_flops = sum(by_L[L].flops for L in stream_L) / len(stream_L)
    out["curriculum"] = {"workload": "Algorithm 1, Grow-P2 odds, 8 cycles: %d steps x 65536 tokens, H=16, d=128"
                                     % len(stream_L),
                         "bucket_steps": {str(L): stream_L.count(L) for L in sorted(sched)},
                         "ms_per_step_mean": cur_ms, "tflops": cur_flops / (cur_ms * 1e-3) / 1e12,
                         "dd_vs_dm_step_time_ratio": cur_ms / dm_mean, "dd_vs_dm_flop_ratio": cur_flops / dm_flops}
    # the curriculum step stream as stated for the DD-vs-DM comparison: 200 steps, each step's L
    # drawn i.i.d. with probability proportional to its bucket's token count (Sec. 2.2 sampling
    # with the natural mixture), one warm-up pass then the timed pass
    iid_L = wl.curriculum_stream(0, 200)
    for L in iid_L[:12]:
        by_L[L].fwd(stream)
        by_L[L].bwd(stream)
    torch.cuda.synchronize()
    s.record(stream)
    for L in iid_L:
        by_L[L].fwd(stream)
        by_L[L].bwd(stream)
    e.record(stream)
    torch.cuda.synchronize()
    iid_ms = s.elapsed_time(e) / len(iid_L)
    iid_flops = sum(by_L[L].flops for L in iid_L) / len(iid_L)
    bucket_frac = {L: c / sum(counts.values()) for L, c in counts.items()}
    expected_dd_flops = sum(f * wl.attn_flops(T // L, L, H, D) for L, f in bucket_frac.items())
    out["curriculum_iid"] = {
        "workload": "200 steps x 65536 tokens, H=16, d=128; each step's L drawn i.i.d. with probability "
                    "proportional to its bucket's token count (binary decomposition of 100k lognormal documents, "
                    "pieces < 256 dropped, > 8192 split), seed 0",
        "bucket_steps": {str(L): iid_L.count(L) for L in sorted(counts)},
        "ms_per_step_mean": iid_ms, "tflops": iid_flops / (iid_ms * 1e-3) / 1e12,
        "dd_vs_dm_step_time_ratio": iid_ms / dm_mean,
        "dd_vs_dm_flop_ratio": iid_flops / dm_flops,
        "dd_flop_fraction_of_causal_8192": iid_flops / causal_8k,
        "expected_dd_vs_dm_flop_ratio_1000_seeds": expected_dd_flops / (float(frac_many.mean()) * causal_8k)}
    # every curriculum of Table 2 with 1 and 8 cycles: each consumes the same bucket steps,
    # so the expected ms per step is fixed by the per-bucket times; measured = the stream run
    # in its own order
    per_L_ms = {bk.L: time_calls(lambda bk=bk: (bk.fwd(stream), bk.bwd(stream)), 5, 1, stream) for bk in buckets}
    expected = sum(per_L_ms[L] * stream_L.count(L) for L in set(stream_L)) / len(stream_L)
    curricula = {}
    for name, odds in wl.CURRICULA.items():
        for cyc in (1, 8):
            sl = wl.length_curriculum(sched, dict(zip(wl.BUCKETS, odds)), cyc, T, seed=0)
            torch.cuda.synchronize()
            s.record(stream)
            for L in sl:
                by_L[L].fwd(stream)
                by_L[L].bwd(stream)
            e.record(stream)
            torch.cuda.synchronize()
            curricula["%s/%d" % (name, cyc)] = {"measured_ms_per_step": s.elapsed_time(e) / len(sl),
                                                "first_8_L": sl[:8]}
    out["curricula"] = {"steps": len(stream_L), "expected_ms_per_step": expected, "per_curriculum": curricula}
    out["dd_vs_dm_step_time_ratio"] = iid_ms / dm_mean
    out["dd_vs_dm_flop_ratio"] = iid_flops / dm_flops
    # Pack-8k+DM: best-fit-decreasing packing into 8192-token sequences, pad tails masked
    pk = []
    for seed in range(4):
        off_np = wl.packed_dm_offsets(seed)
        off = torch.from_numpy(off_np).to(dev)
        bk = Bucket(ddattn, q, k, v, g, 8, 8192, H, offsets=off, ws=ws)
        ms = time_calls(lambda: (bk.fwd(stream), bk.bwd(stream)), 10, 3, stream)
        pk.append({"seed": seed, "ms": ms, "pair_fraction": wl.live_pairs(8, 8192, off_np) / wl.live_pairs(8, 8192),
                   "segments": int(len(wl.segment_lengths(8, 8192, off_np)))})
    out["pack8k_dm"] = {"workload": "8 best-fit-decreasing bins x 8192, H=16, d=128, document-masked, seeds 0..3; "
                                    "10 timed calls after 3 warm-up calls per seed",
                        "ms_per_step_mean": float(np.mean([x["ms"] for x in pk])), "per_seed": pk}
    # RoPE (f_b = 100k) on the bucket sweep: the forward that rotates q, k itself
    # (dd_attn_fwd_rope) + backward with R^T fused into the dq / dk outputs, against the
    # same step without RoPE and against the separate rotation pass (rope_qk + fwd + bwd)
    qr, kr = torch.empty_like(q), torch.empty_like(k)
    rdesc = [ddattn.make_desc(T // L, L, H, D, None, None, 1e5) for L in wl.BUCKETS]
    rws = ddattn.new_workspace(max(rdesc, key=lambda x: ddattn.workspace_size(x)), dev)
    rope_rows = []
    for bk0 in buckets:
        bk = Bucket(ddattn, q, k, v, g, bk0.B, bk0.L, H, ws=rws, rope_base=1e5, qk_rot=(qr, kr))
        ms = time_calls(lambda: (bk.fwd(stream), bk.bwd(stream)), 5, 2, stream)
        ms_sep = time_calls(lambda: (bk.fwd_separate(stream), bk.bwd(stream)), 5, 2, stream)
        ms_plain = time_calls(lambda: (bk0.fwd(stream), bk0.bwd(stream)), 5, 2, stream)
        fwd_ms = time_calls(lambda: bk.fwd(stream), 10, 2, stream)
        fwd_sep_ms = time_calls(lambda: bk.fwd_separate(stream), 10, 2, stream)
        rope_ms = time_calls(lambda: bk.rope(stream), 10, 2, stream)
        rope_rows.append({"L": bk.L, "ms": ms, "ms_separate_pass": ms_sep, "ms_without_rope": ms_plain,
                          "fwd_ms": fwd_ms, "fwd_separate_pass_ms": fwd_sep_ms, "rope_kernel_ms": rope_ms,
                          "rope_kernel_GBps": 4 * T * H * D * 2 / (rope_ms * 1e-3) / 1e9,
                          "tflops": bk.flops / (ms * 1e-3) / 1e12})
    st = ddattn.poll_status(rws)
    if st != 0:
        raise RuntimeError("device status %d (%s)" % (st, ddattn.status_string(st)))
    step_rope = sum(x["ms"] for x in rope_rows)
    step_sep = sum(x["ms_separate_pass"] for x in rope_rows)
    step_plain = sum(x["ms_without_rope"] for x in rope_rows)
    out["rope_sweep"] = {"workload": "bucket sweep with RoPE f_b=100k: dd_attn_fwd_rope (rotation in the forward "
                                     "kernel; k by a pass first above 512 tokens) + bwd per bucket; the separate "
                                     "form: dd_rope_qk + fwd + bwd",
                         "ms_per_step": step_rope, "ms_per_step_separate_pass": step_sep,
                         "ms_per_step_without_rope": step_plain,
                         "overhead": step_rope / step_plain - 1.0,
                         "overhead_separate_pass": step_sep / step_plain - 1.0,
                         "rope_kernel_frac_of_measured_hbm": float(np.median([x["rope_kernel_GBps"] for x in rope_rows]))
                         / peaks["hbm_gbs"],
                         "per_bucket": rope_rows}
    del qr, kr, rws
    # other model shapes of the Appendix model table at 65536 tokens per call:
    # 3B heads (H=32, d=2560/32=80) and 7B heads (H=32, d=4096/32=128)
    shapes = {}
    for name, Hh, Dh in (("3B", 32, 80), ("7B", 32, 128)):
        gen = torch.Generator(device=dev).manual_seed(Dh)
        xs = [torch.randn(T * Hh * Dh, device=dev, generator=gen).to(torch.bfloat16) for _ in range(4)]
        sws = ddattn.new_workspace(ddattn.make_desc(1, T, Hh, Dh), dev)
        rows = []
        for L in wl.BUCKETS:
            bk = Bucket(ddattn, *xs, T // L, L, Hh, ws=sws, Dh=Dh)
            ms = time_calls(lambda: (bk.fwd(stream), bk.bwd(stream)), 3, 1, stream)
            rows.append({"L": L, "ms": ms, "tflops": bk.flops / (ms * 1e-3) / 1e12})
        st = ddattn.poll_status(sws)
        if st != 0:
            raise RuntimeError("device status %d (%s)" % (st, ddattn.status_string(st)))
        shapes[name] = {"H": Hh, "d": Dh, "ms_per_step": sum(x["ms"] for x in rows),
                        "tflops": sum(wl.attn_flops(T // x["L"], x["L"], Hh, Dh) for x in rows)
                        / (sum(x["ms"] for x in rows) * 1e-3) / 1e12, "per_bucket": rows}
        del xs, sws
    torch.cuda.empty_cache()
    out["model_shapes"] = {"workload": "bucket sweep at 65536 tokens per call, inputs N(0,1) bf16 from a seeded "
                                       "torch generator", **shapes}
    # long-context bucket: B=4, L=16384, H=32, q/k x3
    qb, kb, vb, gb = wl.attn_inputs(4, 16384, 32, D, seed=0, qk_mult=3.0)
    lq, lk, lv, lg = (to_dev(x, dev) for x in (qb, kb, vb, gb))
    bk = Bucket(ddattn, lq, lk, lv, lg, 4, 16384, 32)
    ms = time_calls(lambda: (bk.fwd(stream), bk.bwd(stream)), 5, 2, stream)
    out["long_context"] = {"workload": "B=4 x L=16384, H=32, d=128, q/k x3", "ms": ms,
                           "tflops": bk.flops / (ms * 1e-3) / 1e12,
                           "frac_of_measured_sustained": bk.flops / (ms * 1e-3) / 1e12 / peaks["bf16_tflops_sustained"]}
    del lq, lk, lv, lg, bk
    torch.cuda.empty_cache()
    return out


def e2e_measure(ddattn, qb, kb, vb, gb, buckets, stream, dev, args, world):
    """Same step through the public API with host buffers: every bucket call
    copies its q, k, v, dO in from pinned host memory and its o, lse, dq, dk, dv
    out to pinned host memory inside the timed region. Copies in, compute and
    copies out run on three streams over two device buffer sets, so the copies
    of one call overlap the kernels of its neighbours (stream order guards
    every reuse of a buffer)."""
    import torch
    host_in = [torch.from_numpy(np.ascontiguousarray(x).view(np.int16)).view(torch.bfloat16).pin_memory()
               for x in (qb, kb, vb, gb)]
    outs = ["o", "dq", "dk", "dv"]
    host_out = {n: torch.empty((T, H, D), dtype=torch.bfloat16).pin_memory() for n in outs}
    host_lse = torch.empty(T * H, dtype=torch.float32).pin_memory()
    s_in, s_out = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
    s_c = stream
    sets = []
    for _ in range(2):
        dev_in = [torch.empty(x.shape, dtype=torch.bfloat16, device=dev) for x in host_in]
        calls = [Bucket(ddattn, *dev_in, bk.B, bk.L, H) for bk in buckets]   # own outputs + workspace
        sets.append((dev_in, calls))
    E = lambda: torch.cuda.Event()
    in_done, comp_done, out_done = [E(), E()], [E(), E()], [E(), E()]
    started = [False, False]

    def run(n_calls):
        for j in range(n_calls):
            st = j % 2
            dev_in, calls = sets[st]
            call = calls[j % len(buckets)]
            if started[st]:
                s_in.wait_event(comp_done[st])      # previous user of these inputs is done
            with torch.cuda.stream(s_in):
                for hsrc, d in zip(host_in, dev_in):
                    d.copy_(hsrc, non_blocking=True)
            in_done[st].record(s_in)
            s_c.wait_event(in_done[st])
            if started[st]:
                s_c.wait_event(out_done[st])        # previous outputs of this set copied out
            call.fwd(s_c)
            call.bwd(s_c)
            comp_done[st].record(s_c)
            s_out.wait_event(comp_done[st])
            with torch.cuda.stream(s_out):
                for n in outs:
                    host_out[n].copy_(getattr(call, n).view(T, H, D), non_blocking=True)
                host_lse.copy_(call.lse.view(-1), non_blocking=True)
            out_done[st].record(s_out)
            started[st] = True

    steps = max(2, min(args.steps, 5))
    run(2 * len(buckets))
    torch.cuda.synchronize()
    call0 = sets[0][1][-1]
    call_bytes = 4 * T * H * D * 2 + (4 * T * H * D * 2 + T * H * 4)

    def link_probe():
        """The host link alone: one call's input and output copies, concurrently."""
        e0, e1, e2 = (torch.cuda.Event(enable_timing=True) for _ in range(3))
        e0.record(s_in)
        s_out.wait_event(e0)
        with torch.cuda.stream(s_in):
            for hsrc, d in zip(host_in, sets[0][0]):
                d.copy_(hsrc, non_blocking=True)
        with torch.cuda.stream(s_out):
            for n in outs:
                host_out[n].copy_(getattr(call0, n).view(T, H, D), non_blocking=True)
            host_lse.copy_(call0.lse.view(-1), non_blocking=True)
        e1.record(s_in)
        e2.record(s_out)
        torch.cuda.synchronize()
        return max(e0.elapsed_time(e1), e0.elapsed_time(e2))

    # The host link is shared with the rest of the machine and its rate varies from second
    # to second (on one box whole trials ran at either ~40 or ~62 ms per step, builds and
    # copies-only steps alike), so the step is timed in several trials, each beside its own
    # link probe, and the median is reported.
    trial_ms, trial_link = [], []
    for _ in range(5):
        link_ms = link_probe()
        barrier(world)
        s, e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        s.record(s_in)
        run(steps * len(buckets))
        s_out.wait_stream(s_c)
        e.record(s_out)
        torch.cuda.synchronize()
        trial_ms.append(max_over_ranks(s.elapsed_time(e), world) / steps)
        trial_link.append(call_bytes / (link_ms * 1e-3) / 1e9)
    ms = float(np.median(trial_ms))
    link_gbps = float(np.median(trial_link))
    flops = sum(bk.flops for bk in buckets)
    h2d = len(buckets) * 4 * T * H * D * 2
    d2h = len(buckets) * (4 * T * H * D * 2 + T * H * 4)
    return {"value": world * flops / (ms * 1e-3) / 1e12, "unit": "TFLOP/s", "ms_per_step": ms,
            "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
            "host_link_GBps_in_plus_out": link_gbps,
            "copy_bound_ms_per_step": (h2d + d2h) / (link_gbps * 1e9) * 1e3,
            "trials_ms_per_step": trial_ms, "trials_host_link_GBps": trial_link,
            "steps_per_trial": steps,
            "how": "per bucket call: pinned host q,k,v,dO -> device, fwd+bwd via the C ABI, o,lse,dq,dk,dv -> "
                   "pinned host; copies in / kernels / copies out on 3 streams, 2 device buffer sets; median of 5 trials"}


# ------------------------------------------------------------------ reference arm
def run_reference(args):
    """The fp64 CPU oracle as the reference arm, on the same metric and workload
    (bounded sample per step), on this host's cores."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    per = max(0.5, 60.0 / max(1, args.steps + args.warmup))  # about a minute in all
    for _ in range(args.warmup):
        oracle_sample(per)
    vals, secs = [], 0.0
    for _ in range(args.steps):
        r = oracle_sample(per)
        vals.append(r["value"])
        secs += r["seconds"]
    value = float(np.mean(vals))
    cpu = dict(r)
    cpu["value"] = value
    line = {"impl": "reference",
            "metric": "causal attn fwd+bwd TFLOP/s (algorithmic, 14*d*H*sum L(L+1)/2 per call) over the bucket sweep",
            "value": value, "unit": "TFLOP/s", "n_gpus": int(os.environ.get("WORLD_SIZE", "1")),
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": secs / args.steps * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded N(0,1) bf16 q,k,v,dO)",
            "config": {"workload": "bucket sweep L=256..8192, 65536 tokens per call, H=16, d=128, causal; "
                                   "each step a bounded sample of (seq 0, head h) slices"},
            "cpu_baseline": cpu,
            "e2e": {"value": value, "unit": "TFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=60)  # ~1 s timed: ~20 clock samples
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--quick", action="store_true", help="headline sweep only")
    ap.add_argument("--no-cpu", action="store_true", help="skip the oracle CPU baseline")
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--no-e2e", action="store_true", help="skip the host-buffer end-to-end measurement")
    ap.add_argument("--only-L", type=int, default=0, help="run one bucket of the sweep (profiling)")
    ap.add_argument("--rope-base", type=float, default=0.0,
                    help="run the headline step with RoPE of this base frequency (rotation + fwd + bwd)")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
