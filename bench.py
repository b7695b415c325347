#!/usr/bin/env python
"""Decode-step weight-streaming benchmark (A-IO, arxiv 2604.09752): weight-stream GB/s and
equivalent decode tokens/s on GB300.

A step is one pass of every projection of a decoder (Sec. 3.1: each generated token streams all
weights from HBM): 4 projections per layer plus the lm_head, streamed by one persistent
cooperative kernel launch (one CUDA graph node).  Default workload: the 7B-class decode step at M=1 in bf16
(32 layers, 129 projections, 13.21 GB of weights per token), synthetic seeded weights.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME] [--impl ours|reference]

Prints one JSON line (rank 0).  Multi-GPU: one process per GPU (torchrun); each rank runs an
independent replica (the path is replicated, not sharded) and ``value`` sums all ranks' bytes
over the slowest rank's time.  ``--impl reference`` times the fp64 CPU oracle on a bounded
sample of the same workload on the host cores.
"""
from __future__ import annotations

import argparse
import datetime as _dt
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "weight-stream GB/s (% of GB300 HBM peak); equivalent decode tokens/s at M=1"
NOMINAL_HBM_GBS = 8000.0
FALLBACK_HBM_GBS = 6800.0


def workload_by_name(name):
    from synth import workloads as swl
    if name in swl.WORKLOADS:
        return swl.WORKLOADS[name]
    if name.startswith("7b-pld-"):
        _, _, wt, m = name.split("-")
        return swl.pld_workload(int(m[1:]), wt)
    raise SystemExit(f"unknown workload {name}; choose from {sorted(swl.WORKLOADS)} or 7b-pld-<bf16|int8>-M<m>")


def measured_peak():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return float(d["hbm_gbs"]), "measured (MEASURED_PEAKS.json hbm_gbs: torch copy, read+write)"
    return FALLBACK_HBM_GBS, "fallback (no MEASURED_PEAKS.json)"


def kernel_source_hash():
    h = hashlib.sha256()
    for f in ("aio_stream.cuh", "aio_gemv.cu", "aio_chain.cu", "aio_internal.h"):
        path = os.path.join(ROOT, "paper_2604_09752_gb300", "csrc", f)
        if os.path.exists(path):
            h.update(open(path, "rb").read())
    return h.hexdigest()[:16]


def committed_traffic(workload_name, launches_per_step):
    """DRAM bytes per launch from the committed ncu summary, if it was taken on the current kernel.

    profiles/gemv_traffic.txt holds `kernel_src_sha <hash>` and one `dram_bytes_per_step.<workload>
    <bytes>` line per captured workload (read + write bytes of one whole-step launch)."""
    p = os.path.join(ROOT, "profiles", "gemv_traffic.txt")
    if not os.path.exists(p):
        return None, "no committed ncu traffic summary"
    kv = {}
    for line in open(p):
        line = line.strip()
        if line and not line.startswith("#") and " " in line:
            k, v = line.split(None, 1)
            kv[k] = v
    if kv.get("kernel_src_sha") != kernel_source_hash():
        return None, "kernel changed since the committed ncu capture"
    key = "dram_bytes_per_step." + workload_name
    if key not in kv:
        return None, f"no committed ncu capture for workload {workload_name}"
    return float(kv[key]) / launches_per_step, kv.get("note", "ncu dram__bytes_read.sum + dram__bytes_write.sum")


class ClockSampler:
    """nvidia-smi clocks / throttle reasons sampled every 200 ms in the background."""

    FIELDS = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
        try:
            self.p = subprocess.Popen(["nvidia-smi", f"--id={index}", f"--query-gpu={self.FIELDS}",
                                       "--format=csv,noheader,nounits", "-lms", "200"],
                                      stdout=self.f, stderr=subprocess.DEVNULL)
        except (FileNotFoundError, OSError):
            self.p = None

    def stop(self, t0, t1):
        if self.p is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0, "note": "nvidia-smi unavailable"}
        self.p.terminate()
        self.p.wait()
        self.f.seek(0)
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        sm, smax, reasons, n_all = [], [], set(), 0
        for line in self.f.read().splitlines():
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 10:
                continue
            n_all += 1
            try:
                ts = _dt.datetime.strptime(parts[0], "%Y/%m/%d %H:%M:%S.%f").timestamp()
            except ValueError:
                continue
            if not (t0 - 0.25 <= ts <= t1 + 0.25):
                continue
            try:
                sm.append(float(parts[2]))
                smax.append(float(parts[3]))
            except ValueError:
                continue
            for nm, v in zip(names, parts[6:10]):
                if v.lower().startswith("active"):
                    reasons.add(nm)
        os.unlink(self.f.name)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "reasons": sorted(reasons), "samples": len(sm)}


def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


# Replica bookkeeping across ranks (pg: torch.distributed or None for one process; device: where
# the reduction tensor lives, "cuda" under NCCL, "cpu" under gloo).
def barrier(pg):
    if pg is not None:
        pg.barrier()


def max_over_ranks(pg, v, device="cuda"):
    if pg is None:
        return v
    import torch
    t = torch.tensor([float(v)], dtype=torch.float64, device=device)
    pg.all_reduce(t, op=pg.ReduceOp.MAX)
    return float(t.item())


def sum_over_ranks(pg, v, device="cuda"):
    if pg is None:
        return v
    import torch
    t = torch.tensor([float(v)], dtype=torch.float64, device=device)
    pg.all_reduce(t, op=pg.ReduceOp.SUM)
    return float(t.item())


def replica_throughput(pg, bytes_rank, ms_rank, device="cuda"):
    """Whole-job GB/s of independent replicas: every rank's bytes over the slowest rank's time."""
    ms_max = max_over_ranks(pg, ms_rank, device)
    total = sum_over_ranks(pg, bytes_rank, device)
    return total / (ms_max / 1e3) / 1e9, ms_max


# ---------------------------------------------------------------------------------------------
def oracle_sample(wl, seed, frac):
    """The first ceil(frac*N) rows of every projection, regenerated on the host: [(x, W, s)], bytes."""
    from synth import workloads as swl
    items, nbytes = [], 0
    for p in wl.projs:
        rows = max(1, math.ceil(frac * p.N))
        x = swl.gen_x(seed, wl, p, wl.M).reshape(wl.M, p.K)
        if wl.wtype == "int8":
            W = swl.gen_codes(seed, wl, p, 0, rows).reshape(rows, p.K)
            s = swl.gen_scales(seed, wl, p, 0, rows)
            nbytes += rows * p.K + 2 * rows
        else:
            W = swl.gen_w_bf16(seed, wl, p, 0, rows).reshape(rows, p.K)
            s = None
            nbytes += rows * p.K * 2
        items.append((x, W, s))
    return items, nbytes


def time_oracle(items):
    """Seconds for one pass of the fp64 oracle over a sample, and the threads it used."""
    import oracle
    t0 = time.perf_counter()
    for x, W, s in items:
        if s is None:
            oracle.linear_bf16(x, W)
        else:
            oracle.linear_i8(x, W, s)
    return time.perf_counter() - t0, oracle.threads()


def cpu_oracle_sample(wl, seed, frac, min_seconds=0.0):
    """Time the oracle over a row sample, repeating whole passes until min_seconds have elapsed."""
    items, nbytes = oracle_sample(wl, seed, frac)
    dt, cores = time_oracle(items)
    passes = 1
    while dt < min_seconds:
        d, cores = time_oracle(items)
        dt += d
        passes += 1
    return dt, nbytes * passes, cores, passes


def oracle_single_layer_ms():
    """The oracle on the single 2048 x 2048 bf16 layer (M = 1), best of 5, with every host thread and
    with one (a child process with OMP_NUM_THREADS=1): {"threads": n, "ms": t, "single_thread_ms": t1}."""
    code = ("import sys, time; sys.path.insert(0, %r)\n"
            "import oracle\n"
            "from synth import workloads as swl\n"
            "wl = swl.WORKLOADS['linear-2048']; p = wl.projs[0]\n"
            "x = swl.gen_x(0, wl, p, 1).reshape(1, p.K); W = swl.gen_w_bf16(0, wl, p).reshape(p.N, p.K)\n"
            "best = 1e9\n"
            "for _ in range(5):\n"
            "    t0 = time.perf_counter(); oracle.linear_bf16(x, W); best = min(best, time.perf_counter() - t0)\n"
            "print(oracle.threads(), best * 1e3)\n") % ROOT
    out = {}
    for key, env in (("all", dict(os.environ)), ("one", dict(os.environ, OMP_NUM_THREADS="1"))):
        r = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, env=env, timeout=120)
        threads, ms = r.stdout.split()
        out[key] = (int(threads), float(ms))
    return {"threads": out["all"][0], "ms": round(out["all"][1], 3), "single_thread_ms": round(out["one"][1], 3)}


def run_reference(args, wl):
    world, rank, _ = dist_setup()
    if rank != 0:
        return 0
    # calibrate: a 1/512 sample, then size each step to about 1 s of oracle work
    dt0, b0, cores, _ = cpu_oracle_sample(wl, args.seed, 1.0 / 512)
    per_byte = dt0 / b0
    full = wl.weight_bytes()
    budget_s = max(0.2, min(2.0, 150.0 / max(1, args.steps + args.warmup)))
    frac = min(1.0, budget_s / (per_byte * full))
    items, nbytes = oracle_sample(wl, args.seed, frac)
    dts = []
    for i in range(args.warmup + args.steps):
        dt, cores = time_oracle(items)
        if i >= args.warmup:
            dts.append(dt)
    t = sum(dts) / len(dts)
    gbs = nbytes / t / 1e9
    sample = f"first {frac:.4%} of the rows of all {len(wl.projs)} projections ({nbytes} weight bytes) per step"
    line = {
        "impl": "reference", "metric": METRIC, "value": round(gbs, 3), "unit": "GB/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(t * 1000, 3), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": wl.name, "M": wl.M, "wtype": wl.wtype, "projections": len(wl.projs),
                   "weight_bytes_per_token": full},
        "tokens_per_s_equivalent": round(gbs * 1e9 / full, 4),
        "cpu_baseline": {"value": round(gbs, 3), "unit": "GB/s", "cores": cores, "kind": "oracle", "sample": sample},
        "e2e": {"value": round(gbs, 3), "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        "gpu_launches": 0,
        "oracle_linear_2048": oracle_single_layer_ms(),
    }
    print(json.dumps(line), flush=True)
    return 0


# ---------------------------------------------------------------------------------------------
# ---------------------------------------------------------------------------------------------
def time_calls(fn, stream, steps, warmup):
    """Milliseconds per call of fn(stream handle): warmup untimed calls, then steps calls timed with
    CUDA events on stream, with a device synchronize on both sides."""
    import torch
    sh = stream.cuda_stream
    with torch.cuda.stream(stream):
        for _ in range(warmup):
            fn(sh)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    with torch.cuda.stream(stream):
        for _ in range(steps):
            fn(sh)
    e1.record(stream)
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / steps


def step_record(name, M, wtype, wbytes, ms, peak, launches, **extra):
    """One sub-record of the configs block: a whole decode step of `name` at width M."""
    gbs = wbytes / (ms / 1e3) / 1e9
    r = {"workload": name, "M": M, "wtype": wtype, "weight_bytes_per_token": wbytes, "ms_per_step": round(ms, 4),
         "GB/s": round(gbs, 2), "frac_of_measured_peak": round(gbs / peak, 4), "tokens_per_s": round(1000.0 / ms, 2),
         "launches_per_step": launches}
    if M > 1:
        r["verified_tokens_per_s_upper_bound"] = round(1000.0 * M / ms, 2)
    r.update(extra)
    return r


def bench_single_linear(args, peak):
    """The single 2048 x 2048 bf16 layer at M = 1 (8.39 MB: it would sit in the 129 MB L2 if timed
    alone), timed over 64 distinct seeded copies (537 MB, over 4x L2) so that every launch streams
    from HBM.  Each copy is one standalone launch of the small-projection kernel (what
    aio_linear_run enqueues for this shape: one CTA per row group), the 64 chained with programmatic
    dependent launch in one CUDA graph; the time per layer is the graph's time / 64."""
    from paper_2604_09752_gb300 import aio
    from paper_2604_09752_gb300.workload import DeviceWorkload
    from synth import workloads as swl
    import torch
    copies = 64
    base = swl.WORKLOADS["linear-2048"].projs[0]
    wl = swl.Workload("linear-2048-x64", 0, "bf16", 1, [swl.Proj(i, base.index, base.K, base.N) for i in range(copies)],
                      "64 distinct copies of the single 2048 x 2048 layer")
    dw = DeviceWorkload(wl, seed=args.seed, max_M=1)
    dw.fill_x(1)
    step = dw.step_handle(1, aio.AIO_STEP_GRAPH | aio.AIO_STEP_PDL)
    stream = torch.cuda.Stream()
    ms = time_calls(lambda sh: aio.aio_decode_step(step, sh), stream, args.steps, args.warmup)
    assert aio.aio_decode_step_check(step) == 0
    dw.close()
    layer = base.N * base.K * 2
    per = ms / copies
    gbs = layer / (per / 1e3) / 1e9
    return {"workload": "linear-2048", "baseline_config": 1, "M": 1, "wtype": "bf16", "weight_bytes_per_layer": layer,
            "ms_per_layer": round(per, 5), "GB/s": round(gbs, 2), "frac_of_measured_peak": round(gbs / peak, 4),
            "copies": copies, "rotating_weight_bytes": copies * layer, "launches_per_layer": 1,
            "kernel": "aio_small_kernel<1, bf16> (one CTA per row group)",
            "l2": "64 distinct copies, 537 MB, over 4x the 129 MB L2"}


def bench_steps(args, peak, wl, widths, name_of, **extra):
    """Whole decode steps of one weight set at each width M (one persistent launch per step)."""
    from paper_2604_09752_gb300 import aio
    from paper_2604_09752_gb300.workload import DeviceWorkload
    import torch
    flags = aio.AIO_STEP_GRAPH | aio.AIO_STEP_PERSISTENT
    dw = DeviceWorkload(wl, seed=args.seed, max_M=max(widths))
    wbytes = dw.weight_bytes()
    stream = torch.cuda.Stream()
    out = {}
    for M in widths:
        dw.fill_x(M)
        step = dw.step_handle(M, flags)
        ms = time_calls(lambda sh: aio.aio_decode_step(step, sh), stream, args.steps, args.warmup)
        assert aio.aio_decode_step_check(step) == 0
        out[name_of(M)] = step_record(name_of(M), M, wl.wtype, wbytes, ms, peak, aio.aio_decode_step_kernels(step),
                                      **extra)
    dw.close()
    return out


def bench_chain(args, peak):
    """The chained 7B-class decoder step (every x computed on the device from earlier outputs:
    RMSNorm with residual adds, V of QKV, SwiGLU), M = 1, one persistent launch per step."""
    from paper_2604_09752_gb300 import aio
    from paper_2604_09752_gb300.workload import DeviceWorkload
    from synth import workloads as swl
    import torch
    flags = aio.AIO_STEP_GRAPH | aio.AIO_STEP_PERSISTENT
    out = {}
    # (workload, M, context): context None = attention over one position (O reads the V third of
    # QKV); else attention over a KV cache of that many positions in every layer (2K, Sec. 5.1)
    for name, M, ctx in (("7b-bf16", 1, None), ("7b-int8", 1, None), ("7b-bf16", 1, 2048), ("7b-int8", 1, 2048),
                         ("7b-bf16", 3, 2048)):
        wl = swl.WORKLOADS[name]
        dw = DeviceWorkload(wl, seed=args.seed, max_M=M, chained=True, kv_len=ctx)
        dw.fill_chain(M)
        if ctx:
            dw.fill_kv(ctx - M)
        step = dw.step_handle(M, flags)
        stream = torch.cuda.Stream()
        ms = time_calls(lambda sh: aio.aio_decode_step(step, sh), stream, args.steps, args.warmup)
        assert aio.aio_decode_step_check(step) == 0
        wbytes = dw.weight_bytes()
        if ctx:
            kv_bytes = len(dw.attn_layers) * 2 * dw.n_heads * ctx * swl.HEAD_DIM * 2
            key = f"7b-chain-attn{ctx // 1024}k-{wl.wtype}" + (f"-M{M}" if M > 1 else "")
            out[key] = step_record(key, M, wl.wtype, wbytes + kv_bytes, ms, peak, aio.aio_decode_step_kernels(step),
                                   weight_bytes=wbytes, kv_bytes_per_step=kv_bytes, context=ctx,
                                   note="GB/s over weight + KV-cache bytes")
        else:
            key = f"7b-chain-{wl.wtype}"
            out[key] = step_record(key, M, wl.wtype, wbytes, ms, peak, aio.aio_decode_step_kernels(step))
        dw.close()
    return out


def bench_attention(args, peak):
    """Decode attention over KV caches of the 7B-class shapes (32 heads x 128) at the paper's 2K and
    32K contexts, M = 1 and 3 (PLD look-ahead L = 2): one call per layer, over enough distinct layer
    caches (seeded bf16 N(0, 1)) that a step streams more than 1 GB, well above L2; a step's calls
    are captured in one CUDA graph.  Metric: KV bytes per step / time."""
    import torch
    from paper_2604_09752_gb300 import aio
    n_heads, d = 32, 128
    gen = torch.Generator(device="cuda").manual_seed(args.seed)
    stream = torch.cuda.Stream()
    out = {}
    for L, layers in ((2048, 32), (32768, 4)):
        caches = [(torch.randn(n_heads * L * d, device="cuda", generator=gen).to(torch.bfloat16),
                   torch.randn(n_heads * L * d, device="cuda", generator=gen).to(torch.bfloat16)) for _ in range(layers)]
        for M in (1, 3):
            q = torch.randn(M, n_heads * d, device="cuda", generator=gen)
            o = torch.empty(M, n_heads * d, device="cuda")
            wsb = aio.aio_attention_workspace_bytes(M)
            ws = torch.zeros(wsb, dtype=torch.uint8, device="cuda")

            def one_step(sh):
                for kc, vc in caches:
                    aio.aio_attention_decode(q.data_ptr(), n_heads * d, kc.data_ptr(), vc.data_ptr(), n_heads, d, L, L, M,
                                             o.data_ptr(), ws.data_ptr(), wsb, sh)
            torch.cuda.synchronize()
            one_step(stream.cuda_stream)
            torch.cuda.synchronize()
            graph = torch.cuda.CUDAGraph()            # one replay per step: no host gaps between layers
            with torch.cuda.graph(graph, stream=stream):
                one_step(stream.cuda_stream)
            torch.cuda.synchronize()
            ms = time_calls(lambda sh: graph.replay(), stream, args.steps, args.warmup)
            assert aio.aio_attention_check(ws.data_ptr()) == 0
            kv_bytes = layers * 2 * n_heads * L * d * 2
            gbs = kv_bytes / (ms / 1e3) / 1e9
            key = f"7b-attention-L{L}-M{M}"
            out[key] = {"workload": key, "L": L, "M": M, "layers": layers, "ms_per_step": round(ms, 4),
                        "ms_per_layer": round(ms / layers, 5), "kv_bytes_per_step": kv_bytes, "GB/s": round(gbs, 2),
                        "frac_of_measured_peak": round(gbs / peak, 4), "launches_per_layer": 2}
        del caches
        torch.cuda.empty_cache()
    return out


def bench_pld_ops(args):
    """Latency of the work around a PLD verification pass (Sec. 4.2, N = 6, L = 2): drafting over a
    2K and a 32K token history, the argmax of 3 rows of 32000 logits, and the acceptance check;
    each captured in a CUDA graph and replayed, so the figure is device time per call."""
    import torch
    from paper_2604_09752_gb300 import aio
    gen = torch.Generator(device="cuda").manual_seed(args.seed)
    stream = torch.cuda.Stream()
    res = {}
    for name, T in (("draft_2k", 2048), ("draft_32k", 32768)):
        toks = torch.randint(0, 32000, (T,), dtype=torch.int32, device="cuda", generator=gen)
        out = torch.zeros(5, dtype=torch.int32, device="cuda")
        res[name] = (lambda t=toks, o=out, n=T: aio.aio_pld_draft(t.data_ptr(), n, 6, 2, o.data_ptr(), stream.cuda_stream))
    logits = torch.randn(3, 32000, device="cuda", generator=gen)
    am = torch.zeros(3, dtype=torch.int32, device="cuda")
    res["argmax_3x32000"] = lambda: aio.aio_argmax_rows(logits.data_ptr(), 3, 32000, 32000, am.data_ptr(), stream.cuda_stream)
    dbuf = torch.tensor([2, 2, 0, 1, 2], dtype=torch.int32, device="cuda")
    acc = torch.zeros(2, dtype=torch.int32, device="cuda")
    res["accept"] = lambda: aio.aio_pld_accept(am.data_ptr(), dbuf.data_ptr(), acc.data_ptr(), stream.cuda_stream)
    line = {"unit": "us per call"}
    for name, fn in res.items():
        reps = 50
        fn()
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            for _ in range(reps):
                fn()
        g.replay()
        torch.cuda.synchronize()
        line[name] = round(time_calls(lambda sh: g.replay(), stream, 3, 1) * 1e3 / reps, 2)
    return line


def configs_block(args, peak, local, main_rec):
    """Every named workload in one object (the single 2048 x 2048 layer, the 1B and 7B bf16 steps, the
    7B int8 step and the PLD widths), then the later rows of the path (chained step, decode
    attention, PLD drafting and acceptance), with the clocks seen meanwhile."""
    from synth import workloads as swl
    clocks = ClockSampler(local)
    t0 = time.time()
    out = {"linear-2048": bench_single_linear(args, peak)}
    out.update(bench_steps(args, peak, swl.WORKLOADS["1b-bf16"], (1,), lambda M: "1b-bf16", baseline_config=2))
    out["7b-bf16"] = dict(main_rec, baseline_config=3, measured_in="the main line above")
    for wt in ("bf16", "int8"):
        out.update(bench_steps(args, peak, swl.pld_workload(8, wt), swl.PLD_WIDTHS,
                               lambda M, wt=wt: f"7b-pld-{wt}-M{M}", baseline_config=5))
    m1 = out["7b-pld-int8-M1"]
    out["7b-int8"] = dict(m1, workload="7b-int8", baseline_config=4,
                          measured_in="the int8 weight set of the PLD sweep at M = 1 (the same kernel and launch)")
    if args.configs == "all":
        nxt = {}
        nxt.update(bench_chain(args, peak))
        nxt.update(bench_attention(args, peak))
        nxt["pld_ops"] = bench_pld_ops(args)
        out["next_rows"] = nxt
    out["clocks"] = clocks.stop(t0, time.time())
    out["steps"], out["warmup"] = args.steps, args.warmup
    return out


# ---------------------------------------------------------------------------------------------
def run_ours(args, wl):
    import torch
    world, rank, local = dist_setup()
    if not torch.cuda.is_available():
        raise SystemExit("bench.py needs a CUDA GPU (libaio is sm_103a only); no CPU fallback")
    torch.cuda.set_device(local)
    pg = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
        pg = dist
    from paper_2604_09752_gb300 import aio
    from paper_2604_09752_gb300.workload import DeviceWorkload

    M = wl.M
    t_setup = time.perf_counter()
    dw = DeviceWorkload(wl, seed=args.seed + rank, max_M=M)
    x_host = dw.fill_x(M)
    setup_s = time.perf_counter() - t_setup
    stream = torch.cuda.Stream()
    sh = stream.cuda_stream
    flags = {"persistent": aio.AIO_STEP_GRAPH | aio.AIO_STEP_PERSISTENT,
             "chain": aio.AIO_STEP_GRAPH | aio.AIO_STEP_PDL}[args.step_mode]
    step = dw.step_handle(M, flags)
    n_kernels = aio.aio_decode_step_kernels(step)
    wbytes = dw.weight_bytes()

    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            aio.aio_decode_step(step, sh)
    torch.cuda.synchronize()
    assert aio.aio_decode_step_check(step) == 0

    # ---- device-resident timed region
    clocks = ClockSampler(local)
    time.sleep(0.4)
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier(pg)
    torch.cuda.synchronize()
    w0 = time.time()
    ev0.record(stream)
    for _ in range(args.steps):
        aio.aio_decode_step(step, sh)
    ev1.record(stream)
    torch.cuda.synchronize()
    w1 = time.time()
    barrier(pg)
    ms = ev0.elapsed_time(ev1) / args.steps
    clk = clocks.stop(w0, w1)
    value, ms_max = replica_throughput(pg, wbytes, ms)
    assert aio.aio_decode_step_check(step) == 0

    # ---- end to end through the public API: aio_decode_step_host copies the step's x from pinned
    # host memory, runs the step and copies its y back to pinned host memory, every step
    y_host = torch.empty(dw.y_arena.numel(), dtype=torch.uint8, pin_memory=True)
    xb, yb = x_host.numel(), y_host.numel()

    def e2e_step(s):
        aio.aio_decode_step_host(step, x_host.data_ptr(), dw.x_arena.data_ptr(), xb, dw.y_arena.data_ptr(),
                                 y_host.data_ptr(), yb, s)
    e_steps = max(10, args.steps // 4)
    barrier(pg)
    e_ms_rank = time_calls(e2e_step, stream, e_steps, 3)
    barrier(pg)
    e2e_gbs, e_ms = replica_throughput(pg, wbytes, e_ms_rank)
    assert torch.equal(y_host, dw.y_arena.cpu()), "host copy of y differs from the device's"

    # ---- largest projection alone (standalone kernel, same stream)
    big = max(range(len(dw.bufs)), key=lambda i: dw.bufs[i].proj.N * dw.bufs[i].proj.K)
    bp = dw.bufs[big].proj
    big_ms = time_calls(lambda s: dw.run_proj(big, M, s), stream, 50, 5)
    esize = 1 if dw.i8 else 2
    big_bytes = bp.N * bp.K * esize + (2 * bp.N if dw.i8 else 0)

    # ---- read ceiling of the same bulk-copy ring (4 GiB, well above L2)
    pbuf = torch.empty(4 << 30, dtype=torch.uint8, device="cuda")
    pout = torch.zeros(1, dtype=torch.int32, device="cuda")
    probe_ms = time_calls(lambda s: aio.aio_probe_read(pbuf.data_ptr(), pbuf.numel(), pout.data_ptr(), s), stream, 10, 3)
    probe_gbs = pbuf.numel() / (probe_ms / 1e3) / 1e9
    del pbuf

    peak, peak_src = measured_peak()
    gbs_rank = wbytes / (ms / 1e3) / 1e9
    tokens = world * 1000.0 / ms_max
    traffic, traffic_note = committed_traffic(wl.name, n_kernels)
    dw.close()
    del dw
    torch.cuda.empty_cache()

    line = None
    if rank == 0:
        main_rec = step_record(wl.name, M, wl.wtype, wbytes, ms, peak, n_kernels)
        configs = None
        if world == 1 and args.configs != "none":
            configs = configs_block(args, peak, local, main_rec)
        cpu = None
        if world == 1 and not args.no_cpu_baseline:
            dt, nbytes, cores, passes = cpu_oracle_sample(wl, args.seed, args.cpu_frac, args.cpu_seconds)
            cpu = {"value": round(nbytes / dt / 1e9, 3), "unit": "GB/s", "cores": cores, "kind": "oracle",
                   "sample": f"first {args.cpu_frac:.2%} of the rows of all {len(wl.projs)} projections, "
                             f"{passes} passes ({nbytes} weight bytes, {dt:.1f} s of fp64 oracle work)"}
        line = {
            "metric": METRIC,
            "value": round(value, 2),
            "unit": "GB/s",
            "n_gpus": world,
            "steps": args.steps,
            "warmup": args.warmup,
            "ms_per_step": round(ms_max, 4),
            "higher_is_better": True,
            "scaling": "weak",
            "vs_baseline": None,
            "dtype": "int8" if wl.wtype == "int8" else "bf16",
            "data": "synthetic",
            "config": {
                "workload": wl.name,
                "description": wl.description,
                "M": M, "wtype": wl.wtype, "projections": len(wl.projs),
                "weight_bytes_per_token": wbytes,
                "parallelism": f"replicas x{world}" if world > 1 else "single GPU",
                "l2": "inputs larger than L2 (every step streams all weights, >= 2.39 GB)",
                "step_mode": args.step_mode,
            },
            "tokens_per_s": round(tokens, 2),
            "verified_tokens_per_s_upper_bound": round(tokens * M, 2),
            "pct_of_measured_peak": round(100 * gbs_rank / peak, 2),
            "pct_of_nominal_8tbs": round(100 * gbs_rank / NOMINAL_HBM_GBS, 2),
            "roofline": {
                "bound": "hbm",
                "kernel": f"aio_stream_kernel<M={M}, {wl.wtype}>",
                "achieved": round(gbs_rank, 2),
                "peak": peak,
                "unit": "GB/s",
                "frac": round(gbs_rank / peak, 4),
                "traffic": traffic,
                "traffic_note": traffic_note,
                "peak_source": peak_src,
                "algorithmic_bytes_per_launch": round(wbytes / n_kernels, 1),
                "avg_launch_ms": round(ms / n_kernels, 5),
                "launches_per_step": n_kernels,
            },
            "kernel_alone": {"projection": bp.name, "K": bp.K, "N": bp.N, "ms": round(big_ms, 4),
                             "GB/s": round(big_bytes / (big_ms / 1e3) / 1e9, 2)},
            "probe_read_gbs": round(probe_gbs, 1),
            "e2e": {"value": round(e2e_gbs, 2), "unit": "GB/s", "ms_per_step": round(e_ms, 4),
                    "h2d_bytes_per_step": int(xb), "d2h_bytes_per_step": int(yb),
                    "path": "aio_decode_step_host: pinned host x -> device, the step, device y -> pinned host, "
                            "one stream"},
            "gpu_launches": args.steps * n_kernels,
            "clocks": clk,
            "setup_s": round(setup_s, 1),
            "cpu_baseline": cpu,
            "configs": configs,
            # The paper's own decode rates on Ascend 910B, FP16 at 2K context (Tab. 3, Tab. 4): context only.
            "paper_context": {"hardware": "Ascend 910B", "tokens_per_s_1b": 21.58, "tokens_per_s_7b": 17.18,
                              "tokens_per_s_a_io_scenario_a": 19.80},
        }
        print(json.dumps(line), flush=True)
    if pg is not None:
        pg.barrier()
        pg.destroy_process_group()
    return 0


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=500)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="7b-bf16")
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--cpu-frac", type=float, default=0.125)
    ap.add_argument("--cpu-seconds", type=float, default=12.0,
                    help="repeat oracle passes over the row sample for at least this long")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--configs", choices=["all", "baseline", "none"], default="all",
                    help="the configs block (N = 1 only): every named workload (baseline), plus the chained step, "
                         "decode attention and PLD drafting (all), or nothing (none)")
    ap.add_argument("--step-mode", choices=["persistent", "chain"], default="persistent",
                    help="one cooperative launch per step (default) or one launch per projection")
    args = ap.parse_args()
    if args.warmup < 3:
        raise SystemExit("--warmup must be >= 3")
    wl = workload_by_name(args.workload)
    if args.impl == "reference":
        return run_reference(args, wl)
    return run_ours(args, wl)


if __name__ == "__main__":
    sys.exit(main())
