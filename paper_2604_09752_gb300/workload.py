"""Device-resident decode-step workloads on top of the C ABI.

PyTorch only provides memory (device tensors, pinned host staging) and streams;
every byte of arithmetic runs in libaio.  Synthetic inputs come from ``synth``
(seeded, counter-based) and are copied host -> device once; the packer then
tiles each weight matrix on the device.

Buffers: one bf16 x arena and one fp32 y arena hold every projection's x [M, K]
and y [M, N] back to back (each slice 256-byte aligned), so a whole step's
inputs and outputs move with one host<->device copy each.

A chained workload (``chained=True``) wires the projections into decoder layers
(synth.workloads.chain_links): the device computes every projection's x from
earlier outputs, so the step's only inputs are the residual stream h0 and the
norm weights.  With ``kv_len=L_max`` each layer also gets a KV cache of L_max
positions, and O's x is attention of the new tokens over it (the step's L_past
is a device int set by ``fill_chain``).
"""
from __future__ import annotations

import math
from dataclasses import dataclass
from typing import Dict, List, Optional, Tuple

import torch

from . import aio
from synth import workloads as swl

_ALIGN = 256


def _round(v: int, a: int = _ALIGN) -> int:
    return (v + a - 1) // a * a


@dataclass
class _ProjBuf:
    proj: swl.Proj
    handle: int
    W: torch.Tensor            # packed (or row-major) weight bytes
    scales: Optional[torch.Tensor]
    x_off: int                 # byte offsets into the arenas
    y_off: int


class DeviceWorkload:
    """All weights of a workload resident on the current CUDA device, plus x / y arenas.

    ``M`` is the number of token rows of the step (the workload's own M by default);
    ``max_M`` sizes the handles so one set of packed weights serves several widths.
    """

    def __init__(self, wl: swl.Workload, seed: int = 0, max_M: int = 8, layout: str = "packed",
                 device: Optional[torch.device] = None, projs: Optional[List[swl.Proj]] = None,
                 chained: bool = False, kv_len: Optional[int] = None):
        assert layout in ("packed", "rowmajor")
        self.wl = wl
        self.seed = seed
        self.max_M = max_M
        self.layout = layout
        self.device = device or torch.device("cuda", torch.cuda.current_device())
        self.projs = list(projs if projs is not None else wl.projs)
        self.i8 = wl.wtype == "int8"
        self._handles: Dict[Tuple[int, int], int] = {}
        self._steps: Dict[Tuple[int, int], int] = {}
        flags = aio.AIO_FLAG_ROWMAJOR if layout == "rowmajor" else 0
        wt = aio.AIO_W_INT8_PERCHANNEL if self.i8 else aio.AIO_W_BF16
        for p in self.projs:
            if (p.K, p.N) not in self._handles:
                self._handles[(p.K, p.N)] = aio.aio_linear_create(p.K, p.N, wt, max_M, flags)
        # arenas sized for max_M rows
        x_bytes = y_bytes = 0
        offs = []
        for p in self.projs:
            offs.append((x_bytes, y_bytes))
            x_bytes += _round(max_M * p.K * 2)
            y_bytes += _round(max_M * p.N * 4)
        self.x_arena = torch.zeros(x_bytes, dtype=torch.uint8, device=self.device)
        self.y_arena = torch.zeros(y_bytes, dtype=torch.uint8, device=self.device)
        self.bufs: List[_ProjBuf] = []
        self._load_weights(offs)
        self.chained = chained
        self.kv_len = kv_len if chained else None
        if chained:
            self.links = swl.chain_links(swl.Workload(wl.name, wl.family, wl.wtype, wl.M, self.projs),
                                         attention=self.kv_len is not None)
            H = self.projs[0].K
            hb = _round(max_M * H * 4)
            # h0, the two residual buffers, then the norm weights [n_norms, H] bf16
            self.n_norms = max(l.gamma for l in self.links) + 1
            self.h_arena = torch.zeros(3 * hb + _round(self.n_norms * H * 2), dtype=torch.uint8, device=self.device)
            self._hb = hb
        if self.kv_len is not None:
            self.n_heads = H // swl.HEAD_DIM
            self.attn_layers = sorted({l.layer for l in self.links if l.op == swl.XOP_ATTENTION})
            self._kvb = _round(2 * self.n_heads * self.kv_len * swl.HEAD_DIM * 2)
            self.kv_arena = torch.zeros(len(self.attn_layers) * self._kvb, dtype=torch.uint8, device=self.device)
            self.lpast = torch.zeros(64, dtype=torch.int32, device=self.device)

    # ------------------------------------------------------------------ loading
    def _load_weights(self, offs):
        esize = 1 if self.i8 else 2
        max_elems = max(p.N * p.K for p in self.projs)
        stage = torch.empty(max_elems * esize, dtype=torch.uint8, pin_memory=True)
        raw = torch.empty(max_elems * esize, dtype=torch.uint8, device=self.device) if self.layout == "packed" else None
        sstage = torch.empty(max(p.N for p in self.projs) * 2, dtype=torch.uint8, pin_memory=True)
        stream = torch.cuda.current_stream(self.device)
        for p, (xo, yo) in zip(self.projs, offs):
            h = self._handles[(p.K, p.N)]
            nbytes = p.N * p.K * esize
            torch.cuda.synchronize(self.device)   # the staging buffers are reused
            if self.i8:
                swl.gen_codes(self.seed, self.wl, p, out=stage.data_ptr())
            else:
                swl.gen_w_bf16(self.seed, self.wl, p, out=stage.data_ptr())
            W = torch.empty(nbytes, dtype=torch.uint8, device=self.device)
            scales = None
            if self.i8:
                swl.gen_scales(self.seed, self.wl, p, out=sstage.data_ptr())
                scales = torch.empty(p.N * 2, dtype=torch.uint8, device=self.device)
                scales.copy_(sstage[: p.N * 2], non_blocking=True)
            if self.layout == "packed":
                raw[:nbytes].copy_(stage[:nbytes], non_blocking=True)
                aio.aio_linear_pack(h, raw.data_ptr(), scales.data_ptr() if self.i8 else None, W.data_ptr(),
                                    scales.data_ptr() if self.i8 else None, stream.cuda_stream)
            else:
                W.copy_(stage[:nbytes], non_blocking=True)
            self.bufs.append(_ProjBuf(p, h, W, scales, xo, yo))
        torch.cuda.synchronize(self.device)
        del raw

    def fill_x(self, M: Optional[int] = None):
        """Write every projection's seeded x [M, K] into the x arena (host generation, one copy)."""
        M = M or self.wl.M
        host = torch.zeros(self.x_arena.numel(), dtype=torch.uint8, pin_memory=True)
        for b in self.bufs:
            swl.gen_x(self.seed, self.wl, b.proj, M, out=host.data_ptr() + b.x_off)
        self.x_arena.copy_(host)
        torch.cuda.synchronize(self.device)
        return host

    def fill_chain(self, M: Optional[int] = None):
        """Write the chained step's inputs: h0 [M, H] (fp32) and every norm weight [H] (bf16)."""
        assert self.chained
        M = M or self.wl.M
        H = self.projs[0].K
        host = torch.zeros(self.h_arena.numel(), dtype=torch.uint8, pin_memory=True)
        h0 = swl.gen_h0(self.seed, self.wl, M)
        host[: M * H * 4].copy_(torch.from_numpy(h0.view("uint8").reshape(-1)))
        g = host[3 * self._hb:].view(torch.int16)
        for j in range(self.n_norms):
            swl.gen_gamma(self.seed, self.wl, j, out=g.data_ptr() + j * H * 2)
        self.h_arena.copy_(host)
        torch.cuda.synchronize(self.device)
        return h0

    def fill_kv(self, L_past: int):
        """Every layer's seeded KV cache (synth.workloads.gen_kv_cache) and the step's L_past."""
        assert self.kv_len is not None
        n = 2 * self.n_heads * self.kv_len * swl.HEAD_DIM
        host = torch.empty(n * 2, dtype=torch.uint8, pin_memory=True)
        for i, layer in enumerate(self.attn_layers):
            torch.cuda.synchronize(self.device)   # the staging buffer is reused
            swl.gen_kv_cache(self.seed, self.wl, layer, self.kv_len, out=host.data_ptr())
            self.kv_arena[i * self._kvb: i * self._kvb + n * 2].copy_(host, non_blocking=True)
        self.set_lpast(L_past)
        torch.cuda.synchronize(self.device)

    def set_lpast(self, L_past: int):
        self.lpast[0] = L_past

    def kv_ptr(self, layer: int) -> int:
        return self.kv_arena.data_ptr() + self.attn_layers.index(layer) * self._kvb

    def kv(self, layer: int) -> torch.Tensor:
        """Layer `layer`'s cache as int16 bf16 bits [2, n_heads, L_max, 128]."""
        o = self.attn_layers.index(layer) * self._kvb
        n = 2 * self.n_heads * self.kv_len * swl.HEAD_DIM
        return self.kv_arena[o: o + n * 2].view(torch.int16).view(2, self.n_heads, self.kv_len, swl.HEAD_DIM)

    def h_ptr(self, j: int) -> int:
        """-1: the input h0; 0 / 1: the residual buffers."""
        return self.h_arena.data_ptr() + (j + 1) * self._hb

    def h(self, j: int, M: int) -> torch.Tensor:
        H = self.projs[0].K
        o = (j + 1) * self._hb
        return self.h_arena[o: o + M * H * 4].view(torch.float32).view(M, H)

    def gamma_ptr(self, j: int) -> int:
        return self.h_arena.data_ptr() + 3 * self._hb + j * self.projs[0].K * 2

    def gamma(self, j: int) -> torch.Tensor:
        H = self.projs[0].K
        o = 3 * self._hb + j * H * 2
        return self.h_arena[o: o + H * 2].view(torch.int16)

    def _preps(self):
        out = []
        for i, (b, l) in enumerate(zip(self.bufs, self.links)):
            src = self.y_ptr(l.src) if l.src >= 0 else None
            if l.op == swl.XOP_RMSNORM:
                out.append((l.op, src, b.proj.K, 0, self.h_ptr(l.h_in), self.h_ptr(l.h_out) if l.h_out >= 0 else None,
                            self.gamma_ptr(l.gamma), swl.RMS_EPS))
            elif l.op == swl.XOP_ATTENTION:
                out.append((l.op, src, self.bufs[l.src].proj.N, 0, None, None, None, 0.0, self.kv_ptr(l.layer),
                            self.lpast.data_ptr(), self.n_heads, self.kv_len))
            else:
                out.append((l.op, src, self.bufs[l.src].proj.N, l.src_off, None, None, None, 0.0))
        return out

    # ------------------------------------------------------------------ views and calls
    def x_ptr(self, i: int) -> int:
        return self.x_arena.data_ptr() + self.bufs[i].x_off

    def y_ptr(self, i: int) -> int:
        return self.y_arena.data_ptr() + self.bufs[i].y_off

    def y(self, i: int, M: int) -> torch.Tensor:
        b = self.bufs[i]
        return self.y_arena[b.y_off: b.y_off + M * b.proj.N * 4].view(torch.float32).view(M, b.proj.N)

    def x(self, i: int, M: int) -> torch.Tensor:
        b = self.bufs[i]
        return self.x_arena[b.x_off: b.x_off + M * b.proj.K * 2].view(torch.int16).view(M, b.proj.K)

    def run_proj(self, i: int, M: int, stream: Optional[int] = None):
        b = self.bufs[i]
        s = torch.cuda.current_stream(self.device).cuda_stream if stream is None else stream
        aio.aio_linear_run(b.handle, self.x_ptr(i), M, b.proj.K, b.proj.N, b.W.data_ptr(),
                           b.scales.data_ptr() if b.scales is not None else None, self.y_ptr(i), s)

    def step_handle(self, M: int, flags: int = aio.AIO_STEP_GRAPH | aio.AIO_STEP_PERSISTENT) -> int:
        """The step over every projection: chained (x computed on the device) for a chained
        workload, else with every x an input."""
        key = (M, flags)
        if key not in self._steps:
            projs = [(b.handle, self.x_ptr(i), b.W.data_ptr(),
                      b.scales.data_ptr() if b.scales is not None else None, self.y_ptr(i))
                     for i, b in enumerate(self.bufs)]
            if self.chained:
                self._steps[key] = aio.aio_decode_step_create_chained(projs, self._preps(), M, flags)
            else:
                self._steps[key] = aio.aio_decode_step_create(projs, M, flags)
        return self._steps[key]

    def step(self, M: int, flags: int = aio.AIO_STEP_GRAPH | aio.AIO_STEP_PERSISTENT, stream: Optional[int] = None):
        s = torch.cuda.current_stream(self.device).cuda_stream if stream is None else stream
        aio.aio_decode_step(self.step_handle(M, flags), s)

    def weight_bytes(self) -> int:
        esize = 1 if self.i8 else 2
        return sum(p.N * p.K * esize + (2 * p.N if self.i8 else 0) for p in self.projs)

    def close(self):
        torch.cuda.synchronize(self.device)
        for s in self._steps.values():
            aio.aio_decode_step_destroy(s)
        self._steps.clear()
        for h in self._handles.values():
            aio.aio_linear_destroy(h)
        self._handles.clear()
        self.bufs.clear()

    def __del__(self):
        try:
            if self._handles:
                self.close()
        except Exception:
            pass
