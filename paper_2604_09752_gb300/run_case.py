"""Run one projection (or one whole step) of a workload a few times: the small, self-contained case
that profilers capture.

  python -m paper_2604_09752_gb300.run_case --workload 7b-bf16 --proj lm_head --reps 3
  python -m paper_2604_09752_gb300.run_case --workload 1b-bf16 --step --reps 3

Prints the mean time per repetition from CUDA events.
"""
from __future__ import annotations

import argparse
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--workload", default="7b-bf16")
    ap.add_argument("--proj", default="lm_head", help="qkv, o, gate_up, down or lm_head (layer 0 / last)")
    ap.add_argument("--M", type=int, default=1)
    ap.add_argument("--step", action="store_true", help="run the whole decode step instead of one projection")
    ap.add_argument("--layers", type=int, default=0, help="with --step: keep only this many layers (0 = all)")
    ap.add_argument("--mode", choices=["persistent", "chain"], default="persistent")
    ap.add_argument("--reps", type=int, default=3)
    ap.add_argument("--attention", type=int, default=0, metavar="L",
                    help="run decode attention over a 7B-shaped KV cache of L positions (32 heads x 128) instead")
    args = ap.parse_args()

    import torch
    from paper_2604_09752_gb300 import aio
    from paper_2604_09752_gb300.workload import DeviceWorkload
    from synth import workloads as swl

    if args.attention:
        return attention_case(args)
    wl = swl.WORKLOADS[args.workload]
    if args.step:
        L = max(p.layer for p in wl.projs)
        projs = [p for p in wl.projs if args.layers == 0 or p.layer < args.layers or p.layer == L]
    else:
        idx = swl.PROJ_NAMES.index(args.proj)
        projs = [next(p for p in wl.projs if p.index == idx)]
    dw = DeviceWorkload(wl, seed=0, max_M=args.M, projs=projs)
    dw.fill_x(args.M)
    flags = (aio.AIO_STEP_GRAPH | aio.AIO_STEP_PERSISTENT) if args.mode == "persistent" else \
        (aio.AIO_STEP_GRAPH | aio.AIO_STEP_PDL)
    run = (lambda: dw.step(args.M, flags)) if args.step else (lambda: dw.run_proj(0, args.M))
    run()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(args.reps):
        run()
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / args.reps
    gb = dw.weight_bytes() / 1e9
    print(f"{args.workload} {'step' if args.step else args.proj} M={args.M}: {ms:.4f} ms, {gb / ms * 1e3:.1f} GB/s")
    dw.close()


def attention_case(args):
    """One layer's decode attention (32 heads x 128, seeded bf16 N(0, 1) caches), reps calls."""
    import torch
    from paper_2604_09752_gb300 import aio
    n_heads, d, L, M = 32, 128, args.attention, args.M
    gen = torch.Generator(device="cuda").manual_seed(0)
    k = torch.randn(n_heads * L * d, device="cuda", generator=gen).to(torch.bfloat16)
    v = torch.randn(n_heads * L * d, device="cuda", generator=gen).to(torch.bfloat16)
    q = torch.randn(M, n_heads * d, device="cuda", generator=gen)
    out = torch.empty(M, n_heads * d, device="cuda")
    wsb = aio.aio_attention_workspace_bytes(M)
    ws = torch.zeros(wsb, dtype=torch.uint8, device="cuda")

    def run():
        aio.aio_attention_decode(q.data_ptr(), n_heads * d, k.data_ptr(), v.data_ptr(), n_heads, d, L, L, M, out.data_ptr(),
                                 ws.data_ptr(), wsb, torch.cuda.current_stream().cuda_stream)
    run()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(args.reps):
        run()
    e1.record()
    torch.cuda.synchronize()
    assert aio.aio_attention_check(ws.data_ptr()) == 0
    ms = e0.elapsed_time(e1) / args.reps
    kv = 2 * n_heads * L * d * 2
    print(f"attention L={L} M={M}: {ms:.4f} ms per call, {kv / ms / 1e6:.1f} GB/s of KV")


if __name__ == "__main__":
    main()
