#!/usr/bin/env python
"""Benchmark of the PHSA sparse-attention hot path on GB300.

One step = the whole hot path over one batch of the workload: block
representation (a), block selection (b), sparse attention forward (c1) and
its backward (c2-c5, with a synthetic upstream gradient dO). The default
workload is the 32k prefill: B=1, L=32768, 16 query / 8 KV heads, D=128,
blocks of 64 tokens, 14 blocks per query block (97.27% sparsity).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Prints one JSON line (rank 0). Multi-GPU runs (torchrun) shard independent
sequences across ranks (weak scaling, no data-path collective); the only
collectives are the barrier and the max-over-ranks of the elapsed time.
``--impl reference`` times the CPU oracle on bounded samples of the same
workload on this host's cores.
"""
from __future__ import annotations

import argparse
import dataclasses
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2601_02819_gb300 import inputs  # noqa: E402
from paper_2601_02819_gb300.sharding import max_over_ranks, rank_seed, shard_sequences  # noqa: E402

METRIC = ("sparse-attn prefill tokens/s + effective TFLOPS at 32k, 97.3% sparsity; "
          "% roofline")
DECODE_METRIC = ("sparse-attn decode tokens/s, 64 sequences x 32k cached tokens, top-k 14; "
                 "% HBM roofline")
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


# ---------------------------------------------------------------- helpers
def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            d = json.load(f)
        return d, "measured"
    except (OSError, ValueError):
        return dict(FALLBACK_PEAKS), "fallback"


def dist_env():
    return (int(os.environ.get("RANK", "0")), int(os.environ.get("WORLD_SIZE", "1")),
            int(os.environ.get("LOCAL_RANK", "0")))


def algorithmic(w, cnt: np.ndarray):
    """FLOPs and bytes the method must do/move, per stage and per kernel.

    pairs = sum over (b, kv head, query block) of the selected block count,
    times G query heads: every (query head, query block, selected block) pair
    is one 64x64 tile (the diagonal tile counted whole).
    """
    m, D, G = w.block_size, w.D, w.G
    pairs = float(cnt.astype(np.int64).sum()) * G
    bf = 2
    q = w.B * w.Hq * w.L * D * bf
    kv = w.B * w.Hkv * w.L * D * bf
    krepr = w.B * w.Hkv * w.T * D * bf
    idx = cnt.size * (w.topk + 1) * 4
    lse = w.B * w.Hq * w.L * 4
    # candidates actually scored: nC = qb - n_local - n_init + 1 when the budget
    # does not cover them all
    scored = 0
    for qb in range(w.NQB):
        n_c = max(0, qb - w.n_local - w.n_init + 1)
        n_f = min(w.n_init, qb + 1) + (qb - max(min(w.n_init, qb + 1), qb - w.n_local + 1) + 1)
        if w.topk - n_f < n_c:
            scored += n_c
    f_sel = 2.0 * D * m * scored * G * w.B * w.Hkv
    t = {
        "block_repr": {"flops": 0.0, "bytes": kv + w.B * w.L + krepr},
        "select_blocks": {"flops": f_sel, "bytes": q + krepr + idx},
        "attn_fwd": {"flops": 4.0 * m * m * D * pairs, "bytes": q + 2 * kv + q + lse + idx},
        "bwd_delta": {"flops": 0.0, "bytes": 2 * q + lse},
        "bwd_dkdv": {"flops": 8.0 * m * m * D * pairs,
                     "bytes": 2 * q + 2 * kv + 2 * lse + idx + 2 * kv},
        "bwd_dq": {"flops": 6.0 * m * m * D * pairs, "bytes": 2 * q + 2 * kv + 2 * lse + idx + q},
    }
    stages = {
        "fwd": {"flops": f_sel + 4.0 * m * m * D * pairs,
                "parts": ["block_repr", "select_blocks", "attn_fwd"]},
        # reads Q, K, V, O, dO, lse, idx; writes dQ, dK, dV; Delta written and read once
        "bwd": {"flops": 10.0 * m * m * D * pairs, "bytes": 4 * q + 4 * kv + 3 * lse + idx},
    }
    return t, stages, pairs


def roofline_time(t, P_tf, BW_gbs, parts):
    return sum(max(t[k]["flops"] / (P_tf * 1e12), t[k]["bytes"] / (BW_gbs * 1e9)) for k in parts)


class ClockSampler:
    """Samples nvidia-smi clocks/throttle reasons in the background."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, local_rank: int):
        self.proc = None
        self.path = None
        dev = os.environ.get("CUDA_VISIBLE_DEVICES", "").split(",")[0].strip()
        self.dev = dev if dev else str(local_rank)

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(prefix="phsa_clocks_", suffix=".csv")
            os.close(fd)
            self.t0 = time.time()
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu=timestamp,{self.FIELDS}", "--format=csv,noheader",
                 "-lms", "50", "-i", self.dev], stdout=open(self.path, "w"),
                stderr=subprocess.DEVNULL)
        except (OSError, ValueError):
            self.proc = None

    def stop(self, t_begin: float, t_end: float):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.12)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 10:
                    continue
                try:
                    ts = time.mktime(time.strptime(parts[0].split(".")[0], "%Y/%m/%d %H:%M:%S"))
                    ts += float("0." + parts[0].split(".")[1]) if "." in parts[0] else 0.0
                except (ValueError, IndexError):
                    ts = None
                rows.append((ts, parts))
        os.unlink(self.path)
        inside = [p for ts, p in rows if ts is not None and t_begin - 0.05 <= ts <= t_end + 0.05]
        window = "timed region" if inside else "whole run (no sample fell in the timed region)"
        rows = inside if inside else [p for _, p in rows]
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}

        def mhz(s):
            try:
                return float(s.split()[0])
            except (ValueError, IndexError):
                return None
        sm = [mhz(r[2]) for r in rows if mhz(r[2]) is not None]
        smax = [mhz(r[3]) for r in rows if mhz(r[3]) is not None]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = set()
        for r in rows:
            for k, name in enumerate(names):
                if r[6 + k].lower().startswith("active"):
                    reasons.add(name)
        power = [mhz(r[4]) for r in rows if mhz(r[4]) is not None]
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None,
                "reasons": sorted(reasons), "samples": len(rows), "window": window,
                "power_w_max": max(power) if power else None}


# ---------------------------------------------------------------- oracle sample
def oracle_sample_step(w, x, n_units: int, seed: int, aggregation: str = "softmax_sum",
                       fwd_only: bool = False):
    """Times the CPU oracle on a bounded sample of one step; returns estimated seconds
    for the whole step, the parts and a description.

    Sample: stage (a) in full; stages (b), (c) forward and dQ for `n_units` random
    (b, g, qb) units; dK/dV for `n_units` random KV blocks other than block 0. The
    attention parts use a fixed selection table (the forced blocks plus the most
    recent candidates). The oracle's cost per unit is linear in its work (scored
    candidates for (b), selected blocks for (c) and dQ, listed (query block,
    selected block) pairs for dK/dV), so each part is scaled by total work /
    sampled work. Block 0, listed by every query block, carries ~40 typical
    blocks' work; it is left out of the timed sample (one such unit would dominate
    a parallel sample's elapsed time) and counted in the total work."""
    import oracle
    rng = np.random.default_rng(seed)
    U = w.B * w.Hkv * w.NQB
    units = rng.choice(U, size=min(n_units, U), replace=False)
    scale = w.sm_scale
    idx = np.full((w.B, w.Hkv, w.NQB, w.topk), -1, np.int32)
    cnt = np.zeros((w.B, w.Hkv, w.NQB), np.int32)
    lists = np.zeros(w.NQB, np.int64)  # per KV block t: sum of cnt over the query blocks listing t
    for qb in range(w.NQB):
        s = sorted(set(range(min(w.n_init, qb + 1))) | set(range(max(0, qb - w.n_local + 1), qb + 1)))
        extra = [c for c in range(qb) if c not in s][::-1][: max(0, w.topk - len(s))]
        s = sorted(set(s) | set(extra))
        idx[:, :, qb, :len(s)] = s
        cnt[:, :, qb] = len(s)
        lists[s] += len(s)
    qbs = units % w.NQB
    t = {}
    t0 = time.perf_counter()
    Kr = oracle.block_repr(x["K"], x["mask"], w.block_size, w.lam)
    t["repr"] = time.perf_counter() - t0
    t0 = time.perf_counter()
    oracle.select_units(x["Q"], Kr, w.L, w.block_size, w.topk, w.n_init, w.n_local, scale, units,
                        aggregation=aggregation)
    cand_all = w.B * w.Hkv * float(np.sum(np.arange(1, w.NQB + 1)))
    t["select"] = (time.perf_counter() - t0) * cand_all / float(np.sum(qbs + 1))
    rows = []
    for u in units:
        qb = u % w.NQB
        bg = u // w.NQB
        b, g = bg // w.Hkv, bg % w.Hkv
        for hh in range(w.G):
            for i in range(qb * w.block_size, min((qb + 1) * w.block_size, w.L)):
                rows.append((b, g * w.G + hh, i))
    rows = np.array(rows, np.int32)
    frac = float(cnt.sum()) / float(cnt.reshape(-1)[units].sum())
    t0 = time.perf_counter()
    oracle.sparse_attn_rows(x["Q"], x["K"], x["V"], idx, cnt, w.block_size, scale, rows)
    t["fwd"] = (time.perf_counter() - t0) * frac
    if fwd_only:
        desc = (f"stage (a) in full; stages (b) and (c) fwd on {len(units)} of {U} (query block,"
                f" KV head) units; each part scaled by total / sampled work")
        return sum(t.values()), t, desc
    t0 = time.perf_counter()
    oracle.sparse_attn_bwd_dq_rows(x["Q"], x["K"], x["V"], x["dO"], idx, cnt, w.block_size, scale,
                                   rows)
    t["bwd_dq"] = (time.perf_counter() - t0) * frac
    kt = rng.integers(1, w.NQB, len(units)) if w.NQB > 1 else np.zeros(len(units), np.int64)
    kvb = np.stack([units // w.NQB // w.Hkv, (units // w.NQB) % w.Hkv, kt],
                   axis=1).astype(np.int32)
    t0 = time.perf_counter()
    oracle.sparse_attn_bwd_kv_blocks(x["Q"], x["K"], x["V"], x["dO"], idx, cnt, w.block_size,
                                     scale, kvb)
    t["bwd_dkdv"] = ((time.perf_counter() - t0) * w.B * w.Hkv * float(lists.sum())
                     / float(lists[kt].sum()))
    desc = (f"stage (a) in full; stages (b), (c) fwd and dQ on {len(units)}"
            f" of {U} (query block, KV head) units; dK/dV on {len(units)} of {U} KV blocks"
            f" (block 0 excluded); each part scaled by total / sampled work")
    return sum(t.values()), t, desc


def profiled_traffic(kernel: str, workload: str):
    """DRAM bytes per launch of `kernel` on `workload` from the committed ncu summary
    profiles/dram_<kernel>_<workload>.txt, or None when there is none or the kernel's
    sources (listed in it) no longer hash to the value it records."""
    path = os.path.join(ROOT, "profiles", f"dram_{kernel}_{workload}.txt")
    if not os.path.exists(path):
        return None
    fields = {}
    for line in open(path):
        key, sep, val = line.partition(":")
        if sep and key.strip() in ("dram_bytes_per_launch", "sources", "source_sha256"):
            fields[key.strip()] = val.strip()
    if len(fields) != 3:
        return None
    h = hashlib.sha256()
    for rel in fields["sources"].split():
        try:
            h.update(open(os.path.join(ROOT, rel), "rb").read())
        except OSError:
            return None
    return int(fields["dram_bytes_per_launch"]) if h.hexdigest() == fields["source_sha256"] else None


def oracle_threads():
    import oracle
    n = len(os.sched_getaffinity(0))
    oracle.set_threads(n)
    return oracle.max_threads()


# ---------------------------------------------------------------- GPU arm
def workload_of(args, table):
    """The named workload, with the paper's forced-set sizes when asked for."""
    w = table[args.workload]
    if args.forced == "paper":  # 128 initial + 512 local tokens at m = 64
        w = dataclasses.replace(w, name=w.name + "_paper_forced", n_init=2, n_local=8)
    return w


def run_ours(args):
    from paper_2601_02819_gb300 import phsa
    rank, world, local = dist_env()
    if not torch.cuda.is_available():
        raise SystemExit("bench.py needs a CUDA GPU")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    w = workload_of(args, inputs.WORKLOADS)
    # every block size runs the whole step (the backward at m < 64 needs two query
    # heads per KV head, as every workload here has)
    fwd_only = w.block_size != 64 and w.Hq != 2 * w.Hkv
    # weak scaling: every rank runs one batch of the workload on its own sequences
    mine = shard_sequences(world * w.B, world, rank)
    x = inputs.make_inputs(w, with_grad=not fwd_only, seed=rank_seed(w.seed, mine[0]))

    def dev_bf16(a):
        return torch.from_numpy(a.view(np.int16)).to(dev).view(torch.bfloat16)

    Q, K, V = (dev_bf16(x[k]) for k in ("Q", "K", "V"))
    dO = None if fwd_only else dev_bf16(x["dO"])
    mask = torch.from_numpy(x["mask"]).to(dev)
    Kr = torch.empty((w.B, w.Hkv, w.T, w.D), dtype=torch.bfloat16, device=dev)
    idx = torch.empty((w.B, w.Hkv, w.NQB, w.topk), dtype=torch.int32, device=dev)
    cnt = torch.empty((w.B, w.Hkv, w.NQB), dtype=torch.int32, device=dev)
    O = torch.empty_like(Q)
    lse = torch.empty((w.B, w.Hq, w.L), dtype=torch.float32, device=dev)
    if not fwd_only:
        dQ, dK, dV = torch.empty_like(Q), torch.empty_like(K), torch.empty_like(V)
        ws = torch.empty(phsa.phsa_sparse_attn_bwd_workspace(w.B, w.L, w.Hq, w.Hkv, w.topk,
                                                             block_size=w.block_size),
                         dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()
    bs = w.block_size

    def step():
        phsa.phsa_build_block_repr(K, mask, w.lam, Krepr=Kr, block_size=bs)
        phsa.phsa_select_blocks(Q, Kr, w.Hkv, w.topk, w.n_init, w.n_local, w.sm_scale,
                                block_idx=idx, block_cnt=cnt, aggregation=args.aggregation,
                                block_size=bs)
        phsa.phsa_sparse_attn_fwd(Q, K, V, idx, cnt, w.sm_scale, O=O, lse=lse, block_size=bs)
        if not fwd_only:
            phsa.phsa_sparse_attn_bwd(Q, K, V, O, dO, lse, idx, cnt, w.sm_scale, workspace=ws,
                                      dQ=dQ, dK=dK, dV=dV, block_size=bs)

    def barrier():
        if world > 1:
            import torch.distributed as dist
            dist.barrier()

    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    flush_read = torch.ones(256 << 20, dtype=torch.uint8, device=dev)

    def flush_l2():
        # 256 MB written, then 256 MB of another buffer read: every step starts
        # with none of its data in L2 and no dirty line of the flush to write back
        flush.zero_()
        flush_read.sum()

    for _ in range(args.warmup):
        flush_l2()
        step()
    torch.cuda.synchronize()
    status = phsa.phsa_get_device_status()
    if status != 0:
        raise SystemExit(f"device status after warm-up: {phsa.phsa_status_string(status)}")
    cnt_np = cnt.cpu().numpy()

    # Every timed step has its own event pair; L2 is flushed before it, outside
    # the events. ms_per_step is the median step (max over ranks).
    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.3)
    phsa.phsa_profile_read()
    phsa.phsa_profile_enable(True)
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in range(args.steps)]
    barrier()
    torch.cuda.synchronize()
    t_wall0 = time.time()
    for e0, e1 in evs:
        flush_l2()
        e0.record(stream)
        step()
        e1.record(stream)
    torch.cuda.synchronize()
    barrier()
    t_wall1 = time.time()
    phsa.phsa_profile_enable(False)
    prof = phsa.phsa_profile_read()
    clk = clocks.stop(t_wall0, t_wall1)
    step_ms = [a.elapsed_time(b) for a, b in evs]
    ms_step = max_over_ranks(statistics.median(step_ms), device=dev)
    ms_mean = max_over_ranks(statistics.mean(step_ms), device=dev)
    status = phsa.phsa_get_device_status()

    # ---- end to end through the C ABI's host-buffer call: every step copies its
    # inputs from pinned host memory and its results back, inside the timed region
    # (the host-buffer step includes the backward: m = 64 only)
    e2e = None
    if not args.no_e2e and not fwd_only and w.block_size == 64:  # the host-buffer step is m = 64
        pin = lambda a: torch.from_numpy(a).pin_memory()
        hQ, hK, hV, hdO = (pin(x[k].view(np.int16)) for k in ("Q", "K", "V", "dO"))
        hmask = pin(x["mask"])
        pinned = lambda shape, dt: torch.empty(shape, dtype=dt).pin_memory()
        outs = [{"O": pinned(Q.shape, torch.int16), "lse": pinned(lse.shape, torch.float32),
                 "dQ": pinned(Q.shape, torch.int16), "dK": pinned(K.shape, torch.int16),
                 "dV": pinned(K.shape, torch.int16)} for _ in range(2)]
        h2d = sum(t.numel() * t.element_size() for t in (hQ, hK, hV, hdO, hmask))
        d2h = sum(t.numel() * t.element_size() for t in outs[0].values())
        nbytes = phsa.phsa_step_host_workspace(w.B, w.L, w.Hq, w.Hkv, w.topk)
        wss = [torch.empty(nbytes, dtype=torch.uint8, device=dev) for _ in range(2)]
        evs = [torch.cuda.Event() for _ in range(2)]

        def e2e_step(i):
            # two workspaces alternate, so one step's copies overlap the other's kernels
            phsa.phsa_step_host(hQ, hK, hV, hdO, hmask, w.lam, w.topk, w.n_init, w.n_local,
                                w.sm_scale, workspace=wss[i % 2], done_event=evs[i % 2],
                                stream=stream, aggregation=args.aggregation, **outs[i % 2])

        for i in range(2):
            e2e_step(i)
        torch.cuda.synchronize()
        n_e2e = max(3, min(args.steps, 20))
        barrier()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for i in range(n_e2e):
            e2e_step(i)
        for ev in evs:
            stream.wait_event(ev)
        e1.record(stream)
        torch.cuda.synchronize()
        barrier()
        ms_e2e = max_over_ranks(e0.elapsed_time(e1) / n_e2e, device=dev)
        for ws in wss:
            phsa.phsa_step_host_release(ws)
        e2e = {"value": world * w.B * w.L / (ms_e2e / 1e3), "unit": "tokens/s",
               "ms_per_step": ms_e2e, "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
               "steps": n_e2e,
               "note": "phsa_step_host (C ABI) on pinned host buffers: Q, K, V, dO and the mask "
                       "copied in, O, lse, dQ, dK, dV copied back every step; the library "
                       "overlaps the copies with the kernels, two workspaces alternate"}

    if rank != 0:
        return None

    # ---- roofline and per-kernel accounting
    peaks, peak_src = load_peaks()
    P_burst, P_sus, BW = peaks["bf16_tflops"], peaks["bf16_tflops_sustained"], peaks["hbm_gbs"]
    kt, stages, pairs = algorithmic(w, cnt_np)
    kernels = {}
    for name, (ms, n) in prof.items():
        if n == 0:
            continue
        avg_s = ms / n / 1e3
        e = {"launches": n, "ms_total": round(ms, 4), "us_per_launch": round(avg_s * 1e6, 2),
             "share": None}
        if name in kt:
            a = kt[name]
            t_f = a["flops"] / (P_burst * 1e12)
            t_b = a["bytes"] / (BW * 1e9)
            e["bound"] = "tensor" if t_f >= t_b else "hbm"
            e["achieved_tflops"] = round(a["flops"] / avg_s / 1e12, 1)
            e["achieved_gbs"] = round(a["bytes"] / avg_s / 1e9, 1)
            e["frac"] = round(max(t_f, t_b) / avg_s, 4)
        kernels[name] = e
    tot = sum(v["ms_total"] for v in kernels.values()) or 1.0
    for v in kernels.values():
        v["share"] = round(v["ms_total"] / tot, 4)
    dom = max((k for k in kernels if k in kt), key=lambda k: kernels[k]["ms_total"])
    a = kt[dom]
    avg_s = kernels[dom]["ms_total"] / kernels[dom]["launches"] / 1e3
    if kernels[dom]["bound"] == "tensor":
        roof = {"kernel": dom, "bound": "tensor", "achieved": round(a["flops"] / avg_s / 1e12, 1),
                "peak": P_burst, "unit": "TFLOP/s",
                "frac": round(a["flops"] / avg_s / 1e12 / P_burst, 4),
                "peak_source": f"{peak_src} bf16 burst", "traffic": None,
                "algorithmic_per_launch": a["flops"]}
    else:
        roof = {"kernel": dom, "bound": "hbm", "achieved": round(a["bytes"] / avg_s / 1e9, 1),
                "peak": BW, "unit": "GB/s", "frac": round(a["bytes"] / avg_s / 1e9 / BW, 4),
                "peak_source": f"{peak_src} HBM copy", "traffic": None,
                "algorithmic_per_launch": a["bytes"]}
    roof["traffic"] = profiled_traffic(dom, w.name)
    fwd_ms = sum(kernels[k]["ms_total"] for k in ("block_repr", "select_blocks", "attn_fwd")
                 if k in kernels) / args.steps
    bwd_ms = sum(v["ms_total"] for k, v in kernels.items() if k.startswith("bwd")) / args.steps
    fwd_roof = roofline_time(kt, P_burst, BW, ["block_repr", "select_blocks", "attn_fwd"])
    bwd_roof = max(stages["bwd"]["flops"] / (P_burst * 1e12), stages["bwd"]["bytes"] / (BW * 1e9))
    tokens = world * w.B * w.L

    cpu = None
    if not args.no_cpu_baseline and world == 1:
        cores = oracle_threads()
        est_s, parts, desc = oracle_sample_step(w, x, args.cpu_units, seed=5,
                                                aggregation=args.aggregation, fwd_only=fwd_only)
        cpu = {"value": w.B * w.L / est_s, "unit": "tokens/s", "cores": cores, "kind": "oracle",
               "sample": desc, "est_s_per_step": round(est_s, 2),
               "parts_s": {k: round(v, 3) for k, v in parts.items()}}

    out = {
        "metric": METRIC, "value": tokens / (ms_step / 1e3), "unit": "tokens/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(ms_step, 4), "ms_per_step_mean": round(ms_mean, 4),
        "timing": "median of the per-step CUDA-event times; L2 flushed before every step",
        "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": w.name, "B": w.B, "L": w.L, "Hq": w.Hq, "Hkv": w.Hkv, "D": w.D,
                   "block_size": w.block_size, "topk": w.topk, "n_init": w.n_init,
                   "n_local": w.n_local, "lambda": w.lam, "aggregation": args.aggregation,
                   "sparsity": round(1 - w.topk * w.block_size / w.L, 5),
                   "step": ("fwd (repr + select + sparse attn)" if fwd_only else
                            "fwd (repr + select + sparse attn) + bwd (dQ, dK, dV)"),
                   "l2": ("flushed before every step, outside the timed events: 256 MB "
                          "written, then 256 MB of another buffer read; the inputs are also "
                          "larger than L2"),
                   "parallelism": f"dp{world} (independent sequences)"},
        "fwd": {"ms": round(fwd_ms, 4), "tokens_per_s": tokens / (fwd_ms / 1e3) if fwd_ms else None,
                "eff_tflops": round(stages["fwd"]["flops"] / (fwd_ms / 1e3) / 1e12, 1) if fwd_ms else None,
                "roofline_us": round(fwd_roof * 1e6, 1),
                "roofline_frac": round(fwd_roof / (fwd_ms / 1e3), 4) if fwd_ms else None},
        "bwd": None if fwd_only else {
            "ms": round(bwd_ms, 4),
            "eff_tflops": round(stages["bwd"]["flops"] / (bwd_ms / 1e3) / 1e12, 1) if bwd_ms else None,
            "roofline_us": round(bwd_roof * 1e6, 1),
            "roofline_frac": round(bwd_roof / (bwd_ms / 1e3), 4) if bwd_ms else None},
        "roofline": roof,
        "kernels": kernels,
        "gpu_launches": int(sum(v["launches"] for v in kernels.values())),
        "selected_pairs_per_step": int(pairs),
        "e2e": e2e,
        "cpu_baseline": cpu,
        "clocks": clk,
        "device_status": status,
        "peaks": {"source": peak_src, "hbm_gbs": BW, "bf16_tflops": P_burst,
                  "bf16_tflops_sustained": P_sus},
    }
    return out


# ---------------------------------------------------------------- decode
def decode_metric(w) -> str:
    if w.name == "decode_32k_b64":
        return DECODE_METRIC
    return (f"sparse-attn decode tokens/s, {w.B} sequences x {w.L // 1024}k cached tokens, "
            f"block size {w.block_size}, top-k {w.topk}; % HBM roofline")


def decode_algorithmic(w, lens: np.ndarray, cnt: np.ndarray):
    """Bytes each kernel of the fused decode step must move (both HBM-bound).

    select: the candidates' representative keys, q, the block lists; attn: q,
    the selected keys and values up to the new token, O and lse, the block
    lists, and for the refresh of a just-filled block its punctuation bytes and
    the representative key written (its keys are the local block's, already
    counted).
    """
    m, D, bf = w.block_size, w.D, 2
    filled = int(((lens > 0) & (lens % m == 0)).sum())
    rep = filled * w.Hkv * D * bf + filled * m
    n_c = np.maximum(0, (lens - 1) // m - w.n_local - w.n_init + 1)
    sel = int(n_c.sum()) * w.Hkv * D * bf + w.B * w.Hq * D * bf + cnt.size * (w.topk + 1) * 4
    keys = 0
    for b in range(w.B):
        qb = (lens[b] - 1) // m
        for g in range(w.Hkv):
            n = int(cnt[b, g])
            keys += n * m - ((qb + 1) * m - lens[b])  # the local block is filled up to p
    att = keys * 2 * D * bf + 2 * w.B * w.Hq * D * bf + w.B * w.Hq * 4 + cnt.size * (w.topk + 1) * 4
    return {"decode_select": {"flops": 2.0 * D * float(n_c.sum()) * w.Hq, "bytes": float(sel)},
            "decode_attn": {"flops": 4.0 * D * keys * w.G, "bytes": float(att + rep)}}


def oracle_decode_sample(w, x, n_units: int, seed: int, aggregation: str = "softmax_sum"):
    """Times the oracle on `n_units` random (sequence, KV head) units of one
    decode step (the just-filled block's repr, the selection, the attention)
    and scales to the whole batch. Representative keys of the cached blocks are
    computed beforehand (they belong to the cache, not to the step)."""
    import oracle
    rng = np.random.default_rng(seed)
    U = w.B * w.Hkv
    units = rng.choice(U, size=min(n_units, U), replace=False)
    bits = lambda t: t.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)
    m, secs = w.block_size, 0.0
    for u in units:
        b, g = int(u // w.Hkv), int(u % w.Hkv)
        Kbg, Vbg = bits(x["K"][b:b + 1, g:g + 1]), bits(x["V"][b:b + 1, g:g + 1])
        qbg = bits(x["q"][b:b + 1, w.G * g:w.G * (g + 1)])
        mb, lb = x["mask"][b:b + 1], x["lens"][b:b + 1]
        Kr = oracle.block_repr(Kbg, mb, m, w.lam)
        t0 = time.perf_counter()
        L = int(lb[0])
        if L % m == 0:
            oracle.block_repr(Kbg[:, :, L - m:L], mb[:, L - m:L], m, w.lam)
        idx, cnt = oracle.decode_select(qbg, Kr, lb, w.L, m, w.topk, w.n_init, w.n_local,
                                        w.sm_scale, aggregation=aggregation)
        oracle.decode_attn(qbg, Kbg, Vbg, idx, cnt, lb, m, w.sm_scale)
        secs += time.perf_counter() - t0
    est = secs * U / len(units)
    desc = (f"{len(units)} of {U} (sequence, KV head) units of one decode step (repr of the"
            f" filled block, selection, attention), scaled to the batch")
    return est, desc


def run_decode(args):
    from paper_2601_02819_gb300 import phsa
    rank, world, local = dist_env()
    if not torch.cuda.is_available():
        raise SystemExit("bench.py needs a CUDA GPU")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    w = workload_of(args, inputs.DECODE_WORKLOADS)
    x = inputs.make_decode_inputs(w, dev, seed=rank_seed(w.seed, rank * w.B))
    q, K, V, mask, lens = x["q"], x["K"], x["V"], x["mask_dev"], x["lens_dev"]
    # the cache's prefill: not part of a step
    Kr = phsa.phsa_build_block_repr(K, mask, w.lam, block_size=w.block_size)
    idx = torch.empty((w.B, w.Hkv, w.topk), dtype=torch.int32, device=dev)
    cnt = torch.empty((w.B, w.Hkv), dtype=torch.int32, device=dev)
    O = torch.empty_like(q)
    lse = torch.empty((w.B, w.Hq), dtype=torch.float32, device=dev)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    flush_read = torch.ones(256 << 20, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()

    def flush_l2():
        # 256 MB written, then 256 MB of another buffer read: the step finds none
        # of its data in L2, and no dirty line of the flush to write back
        flush.zero_()
        flush_read.sum()

    def step():  # selection; attention fused with the refresh of just-filled blocks
        phsa.phsa_decode_step(q, K, V, mask, lens, w.lam, Kr, w.topk, w.n_init, w.n_local,
                              w.sm_scale, block_idx=idx, block_cnt=cnt, O=O, lse=lse,
                              aggregation=args.aggregation, block_size=w.block_size)

    def barrier():
        if world > 1:
            import torch.distributed as dist
            dist.barrier()

    for _ in range(args.warmup):
        flush_l2()
        step()
    torch.cuda.synchronize()
    status = phsa.phsa_get_device_status()
    if status != 0:
        raise SystemExit(f"device status after warm-up: {phsa.phsa_status_string(status)}")
    cnt_np = cnt.cpu().numpy()

    # L2 is flushed before every step, outside the timed events.
    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.3)
    phsa.phsa_profile_read()
    phsa.phsa_profile_enable(True)
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in range(args.steps)]
    barrier()
    torch.cuda.synchronize()
    t_wall0 = time.time()
    for e0, e1 in evs:
        flush_l2()
        e0.record(stream)
        step()
        e1.record(stream)
    torch.cuda.synchronize()
    barrier()
    t_wall1 = time.time()
    phsa.phsa_profile_enable(False)
    prof = phsa.phsa_profile_read()
    clk = clocks.stop(t_wall0, t_wall1)
    step_ms = [a.elapsed_time(b) for a, b in evs]
    ms_step = max_over_ranks(statistics.median(step_ms), device=dev)
    ms_mean = max_over_ranks(sum(step_ms) / len(step_ms), device=dev)
    status = phsa.phsa_get_device_status()

    e2e = None
    if not args.no_e2e:
        # The caches stay on the device; each step uploads the new token's q, k, v
        # and id, marks the id against the resident punctuation set, appends k, v
        # and the flag at position L - 1, runs the step and reads O back.
        hq = torch.empty(q.shape, dtype=torch.int16).pin_memory()
        hk = torch.empty((w.B, w.Hkv, w.D), dtype=torch.int16).pin_memory()
        hv = torch.empty((w.B, w.Hkv, w.D), dtype=torch.int16).pin_memory()
        hid = torch.empty((w.B,), dtype=torch.int32).pin_memory()
        hq.copy_(q.view(torch.int16).cpu())
        hk.copy_(K[:, :, w.L - 1].contiguous().view(torch.int16).cpu())
        hv.copy_(V[:, :, w.L - 1].contiguous().view(torch.int16).cpu())
        hid.copy_(torch.from_numpy(np.ascontiguousarray(x["ids"][:, w.L - 1])))
        hO = torch.empty(O.shape, dtype=torch.int16).pin_memory()
        kn = torch.empty((w.B, w.Hkv, w.D), dtype=torch.bfloat16, device=dev)
        vn = torch.empty_like(kn)
        idn = torch.empty((w.B,), dtype=torch.int32, device=dev)
        mn = torch.empty((w.B,), dtype=torch.uint8, device=dev)
        pset = torch.from_numpy(x["punct_ids"]).to(dev)
        h2d = sum(t.numel() * t.element_size() for t in (hq, hk, hv, hid))
        d2h = hO.numel() * hO.element_size()

        def e2e_step():
            q.view(torch.int16).copy_(hq, non_blocking=True)
            kn.view(torch.int16).copy_(hk, non_blocking=True)
            vn.view(torch.int16).copy_(hv, non_blocking=True)
            idn.copy_(hid, non_blocking=True)
            phsa.phsa_punct_mask(idn, pset, mask=mn)
            phsa.phsa_decode_append(kn, vn, lens, K, V, flag_new=mn, punct_mask=mask)
            step()
            hO.copy_(O.view(torch.int16), non_blocking=True)

        for _ in range(3):
            e2e_step()
        n_e2e = max(3, min(args.steps, 50))
        barrier()
        torch.cuda.synchronize()
        a0, a1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a0.record(stream)
        for _ in range(n_e2e):
            e2e_step()
        a1.record(stream)
        torch.cuda.synchronize()
        barrier()
        ms_e2e = max_over_ranks(a0.elapsed_time(a1) / n_e2e, device=dev)
        e2e = {"value": world * w.B / (ms_e2e / 1e3), "unit": "tokens/s", "ms_per_step": ms_e2e,
               "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h), "steps": n_e2e,
               "note": "caches resident on the device; per step the new token's q, k, v and "
                       "id are uploaded, the id marked (phsa_punct_mask), k, v and the flag "
                       "appended (phsa_decode_append), the step run and O read back"}

    if rank != 0:
        return None
    peaks, peak_src = load_peaks()
    BW = peaks["hbm_gbs"]
    kt = decode_algorithmic(w, x["lens"], cnt_np)
    kernels = {}
    for name, (ms, n) in prof.items():
        if n == 0:
            continue
        avg_s = ms / n / 1e3
        e = {"launches": n, "ms_total": round(ms, 4), "us_per_launch": round(avg_s * 1e6, 2)}
        if name in kt:
            e["bound"] = "hbm"
            e["achieved_gbs"] = round(kt[name]["bytes"] / avg_s / 1e9, 1)
            e["frac"] = round(kt[name]["bytes"] / avg_s / 1e9 / BW, 4)
        kernels[name] = e
    tot = sum(v["ms_total"] for v in kernels.values()) or 1.0
    for v in kernels.values():
        v["share"] = round(v["ms_total"] / tot, 4)
    dom = max((k for k in kernels if k in kt), key=lambda k: kernels[k]["ms_total"])
    avg_s = kernels[dom]["ms_total"] / kernels[dom]["launches"] / 1e3
    roof = {"kernel": dom, "bound": "hbm", "achieved": round(kt[dom]["bytes"] / avg_s / 1e9, 1),
            "peak": BW, "unit": "GB/s", "frac": round(kt[dom]["bytes"] / avg_s / 1e9 / BW, 4),
            "peak_source": f"{peak_src} HBM copy", "traffic": None,
            "algorithmic_per_launch": kt[dom]["bytes"]}
    step_bytes = sum(v["bytes"] for v in kt.values())
    cpu = None
    if not args.no_cpu_baseline and world == 1:
        cores = oracle_threads()
        est, desc = oracle_decode_sample(w, x, args.cpu_units, seed=5,
                                         aggregation=args.aggregation)
        cpu = {"value": w.B / est, "unit": "tokens/s", "cores": cores, "kind": "oracle",
               "sample": desc, "est_s_per_step": round(est, 3)}
    return {
        "metric": decode_metric(w), "value": world * w.B / (ms_step / 1e3), "unit": "tokens/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(ms_step, 5), "ms_per_step_mean": round(ms_mean, 5),
        "timing": "median of the per-step CUDA-event times; L2 flushed before every step",
        "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": w.name, "B": w.B, "cache_len": w.L, "Hq": w.Hq, "Hkv": w.Hkv,
                   "D": w.D, "block_size": w.block_size, "topk": w.topk, "n_init": w.n_init,
                   "n_local": w.n_local, "lambda": w.lam, "aggregation": args.aggregation,
                   "step": "decode (phsa_decode_step): selection, then attention fused with the refresh of the just-filled block's representative key",
                   "l2": "flushed before every step, outside the timed events: 256 MB written, then 256 MB of another buffer read (no dirty flush line is written back inside the step)",
                   "parallelism": f"dp{world} (independent sequences)"},
        "step_roofline": {"bytes": step_bytes, "us": round(step_bytes / (BW * 1e9) * 1e6, 2),
                          "frac": round(step_bytes / (BW * 1e9) / (ms_step / 1e3), 4)},
        "roofline": roof,
        "kernels": kernels,
        "gpu_launches": int(sum(v["launches"] for v in kernels.values())),
        "e2e": e2e,
        "cpu_baseline": cpu,
        "clocks": clk,
        "device_status": status,
        "peaks": {"source": peak_src, "hbm_gbs": BW},
    }


# ---------------------------------------------------------------- chunked prefill
def run_chunked(args):
    """Prefill of the workload's K, V and punctuation flags into caches in chunks
    of args.chunked tokens through phsa_prefill_append (the representative keys
    of completed blocks from the same loads), against the same chunks copied in
    followed by one phsa_build_block_repr over the cache."""
    from paper_2601_02819_gb300 import phsa
    torch.cuda.set_device(0)
    dev = torch.device("cuda", 0)
    w = workload_of(args, inputs.WORKLOADS)
    if w.block_size != 64:
        raise SystemExit("--chunked runs at block size 64")
    x = inputs.make_inputs(w, with_grad=False, seed=w.seed)
    bf = lambda a: torch.from_numpy(a.view(np.int16)).to(dev).view(torch.bfloat16)
    Ksrc, Vsrc = bf(x["K"]), bf(x["V"])
    msrc = torch.from_numpy(x["mask"]).to(dev)
    C = args.chunked
    starts = list(range(0, w.L, C))
    chunks = [(Ksrc[:, :, p:p + C].contiguous(), Vsrc[:, :, p:p + C].contiguous(),
               msrc[:, p:p + C].contiguous(), torch.full((w.B,), min(p + C, w.L), dtype=torch.int32, device=dev))
              for p in starts]
    K, V = torch.empty_like(Ksrc), torch.empty_like(Vsrc)
    mask = torch.empty_like(msrc)
    Kr = torch.empty((w.B, w.Hkv, w.T, w.D), dtype=torch.bfloat16, device=dev)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)

    def fused():
        for kc, vc, fc, ln in chunks:
            phsa.phsa_prefill_append(kc, vc, ln, K, V, mask, Kr, w.lam, flag_chunk=fc)

    def unfused():
        for (kc, vc, fc, ln), p in zip(chunks, starts):
            n = kc.shape[2]
            K[:, :, p:p + n].copy_(kc)
            V[:, :, p:p + n].copy_(vc)
            mask[:, p:p + n].copy_(fc)
        phsa.phsa_build_block_repr(K, mask, w.lam, Krepr=Kr)

    def timed(fn):
        for _ in range(args.warmup):
            flush.zero_()
            fn()
        ts = []
        for _ in range(args.steps):
            flush.zero_()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            fn()
            e1.record()
            torch.cuda.synchronize()
            ts.append(e0.elapsed_time(e1))
        return statistics.median(ts)

    ms_f = timed(fused)
    assert phsa.phsa_get_device_status() == 0
    Kr_f = Kr.clone()
    ms_u = timed(unfused)
    same = bool(torch.equal(Kr_f.view(torch.int16), Kr.view(torch.int16)))
    peaks, peak_src = load_peaks()
    kv = w.B * w.Hkv * w.L * w.D * 2
    # algorithmic bytes of the fused path: chunks read, caches written, flags,
    # keys written, and the earlier rows of each block a chunk finishes (the
    # part of the block before the chunk, when C is not a multiple of 64)
    head = sum(p % 64 for p in starts[1:]) * w.B * w.Hkv * w.D * 2
    nbytes = 4 * kv + 2 * w.B * w.L + w.B * w.Hkv * w.T * w.D * 2 + head
    return {
        "metric": "chunked prefill into the KV caches with fused representative keys, GB/s",
        "value": nbytes / (ms_f / 1e3) / 1e9, "unit": "GB/s", "n_gpus": 1,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_f, 4),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic",
        "config": {"workload": w.name, "B": w.B, "L": w.L, "Hkv": w.Hkv, "D": w.D,
                   "chunk": C, "chunks": len(starts),
                   "step": "the whole sequence appended chunk by chunk (phsa_prefill_append)",
                   "l2": "flushed before every timed pass (256 MB written)"},
        "bytes_per_step": nbytes, "bytes_per_chunk": nbytes / len(starts),
        "hbm_frac": round(nbytes / (ms_f / 1e3) / 1e9 / peaks["hbm_gbs"], 4),
        "unfused_ms": round(ms_u, 4),
        "unfused_note": "the same chunks copied into the caches, then phsa_build_block_repr",
        "keys_bit_identical": same,
        "gpu_launches": len(starts),
        "peaks": {"source": peak_src, "hbm_gbs": peaks["hbm_gbs"]},
    }


# ---------------------------------------------------------------- reference arm
def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return None
    w = workload_of(args, inputs.WORKLOADS)
    fwd_only = w.block_size != 64 and w.Hq != 2 * w.Hkv  # the same step as our arm's
    x = inputs.make_inputs(w, with_grad=not fwd_only)
    cores = oracle_threads()
    n_units = max(args.ref_units, cores)  # at least one unit per thread
    for s in range(args.warmup):
        oracle_sample_step(w, x, n_units, seed=100 + s, aggregation=args.aggregation,
                           fwd_only=fwd_only)
    ests, descs = [], None
    t0 = time.perf_counter()
    for s in range(args.steps):
        est, _, descs = oracle_sample_step(w, x, n_units, seed=1000 + s,
                                           aggregation=args.aggregation, fwd_only=fwd_only)
        ests.append(est)
    wall = time.perf_counter() - t0
    est = statistics.mean(ests)
    value = w.B * w.L / est
    # A step runs a bounded sample: ms_per_step is its measured time, and the
    # tokens it stands for are the throughput times that time (the sample's
    # share of the whole step, the whole step taking est seconds).
    ms_sample = wall / max(1, args.steps) * 1e3
    return {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(ms_sample, 3), "tokens_per_step": round(value * ms_sample / 1e3, 3),
        "ms_per_full_step_estimate": round(est * 1e3, 1), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": w.name, "B": w.B, "L": w.L, "Hq": w.Hq, "Hkv": w.Hkv, "D": w.D,
                   "block_size": w.block_size, "topk": w.topk, "n_init": w.n_init,
                   "n_local": w.n_local, "lambda": w.lam, "aggregation": args.aggregation,
                   "step": ("fwd (repr + select + sparse attn)" if fwd_only else
                            "fwd (repr + select + sparse attn) + bwd (dQ, dK, dV)")},
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": cores, "kind": "oracle",
                         "sample": descs},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
        "wall_s": round(wall, 2),
    }


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="prefill_32k",
                    choices=sorted(inputs.WORKLOADS) + sorted(inputs.DECODE_WORKLOADS))
    ap.add_argument("--aggregation", choices=["softmax_sum", "max_logit"], default="softmax_sum",
                    help="how a unit's query rows are combined per candidate block")
    ap.add_argument("--forced", choices=["workload", "paper"], default="workload",
                    help="forced blocks: the workload's, or the paper's 2 initial + 8 local")
    ap.add_argument("--chunked", type=int, default=0,
                    help="time a chunked prefill of the workload's keys (chunk length) instead")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-units", type=int, default=48,
                    help="units in the oracle sample of the cpu_baseline")
    ap.add_argument("--ref-units", type=int, default=16,
                    help="units in each oracle sample step of --impl reference")
    args = ap.parse_args()
    if args.warmup < 3 and args.impl == "ours":
        args.warmup = 3
    if args.chunked > 0:
        out = run_chunked(args)
    elif args.workload in inputs.DECODE_WORKLOADS:
        if args.impl == "reference":
            raise SystemExit("--impl reference times the prefill workloads only")
        out = run_decode(args)
    else:
        out = run_reference(args) if args.impl == "reference" else run_ours(args)
    if out is not None:
        print(json.dumps(out), flush=True)
    if int(os.environ.get("WORLD_SIZE", "1")) > 1 and args.impl == "ours":
        import torch.distributed as dist
        if dist.is_initialized():
            dist.destroy_process_group()


if __name__ == "__main__":
    main()
