"""Decode-step workloads: projection shapes and the input recipe.

The paper streams every weight of a 1B-class and a 7B-class decoder from HBM
for each generated token (Sec. 2.1, Sec. 3.1); it does not print the models'
architecture, so the shapes below are LLaMA-style 1B-class and 7B-class
decoders whose fp16 weight totals (2.39 GB, 13.21 GB) sit near the paper's
"~2GB" and "~14GB" footprints (Sec. 3.1).  Prompt-lookup verification (Sec. 4.2,
N=6, L=2) runs the same projections on several token rows at once (M > 1).

Recipe (all seeded, all synthetic; nothing here is the linear-layer arithmetic):
  * x   [M, K]  bf16 ~ N(0, 1)            key(seed, tag(layer), proj, KIND_X)
  * W   [N, K]  bf16 ~ N(0, 1/K)          key(seed, tag(layer), proj, KIND_W)
  * q   [N, K]  int8 uniform on [-127,127] key(seed, tag(layer), proj, KIND_Q)
  * s   [N]     bf16 ~ U(1e-3, 1e-2)      key(seed, tag(layer), proj, KIND_S)
  where tag(layer) = family * 1000 + layer, the lm_head is layer = n_layers,
  element (m, k) of x is index m*K + k, element (n, k) of W or q is n*K + k.

Chained step (the projections wired into decoder layers, see chain_links):
  * h0  [M, H]  fp32 holding bf16 ~ N(0, 1) values (an embedding row)
                                           key(seed, family * 1000, 0, KIND_H0)
  * g   [H]     bf16 ~ U(0.5, 1.5), one per norm: 2l (before QKV of layer l),
                2l + 1 (before gate+up), 2L (before lm_head)
                                           key(seed, family * 1000 + norm, 0, KIND_GAMMA)
  * RMSNorm epsilon RMS_EPS = 1e-5.

Chained step with attention over a KV cache (chain_links(..., attention=True)): O takes its x from
attention of the new tokens over layer l's cache instead of the one-position V slice.
  * cache [2][n_heads][L_max][128] bf16 ~ N(0, 1) (K then V; positions >= L_past are overwritten by
    the step)                              key(seed, family * 1000 + layer, 0, KIND_KV)
  * n_heads = H / 128, the new tokens at positions L_past .. L_past + M - 1.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from typing import List, Optional

import numpy as np

from . import codes_i8, key, normal_bf16, uniform_bf16

KIND_W, KIND_X, KIND_Q, KIND_S, KIND_GAMMA, KIND_H0, KIND_KV = 0, 1, 2, 3, 4, 5, 6
HEAD_DIM = 128
RMS_EPS = 1e-5

# How a projection of a chained step gets its x (the values of the C ABI's AIO_X_* constants).
XOP_GIVEN, XOP_RMSNORM, XOP_SWIGLU, XOP_SLICE, XOP_ATTENTION = 0, 1, 2, 3, 4
PROJ_NAMES = ("qkv", "o", "gate_up", "down", "lm_head")


@dataclass(frozen=True)
class Proj:
    layer: int
    index: int      # 0 qkv, 1 o, 2 gate_up, 3 down, 4 lm_head
    K: int
    N: int

    @property
    def name(self) -> str:
        return f"L{self.layer}.{PROJ_NAMES[self.index]}"


@dataclass(frozen=True)
class Workload:
    name: str
    family: int          # 0 single linear, 1 1B-class, 7 7B-class
    wtype: str           # "bf16" or "int8"
    M: int
    projs: List[Proj] = field(default_factory=list)
    description: str = ""

    def weight_bytes(self) -> int:
        """Algorithmic HBM bytes streamed per step: every weight byte once, plus int8 scales."""
        esize = 2 if self.wtype == "bf16" else 1
        total = sum(p.N * p.K * esize for p in self.projs)
        if self.wtype == "int8":
            total += sum(2 * p.N for p in self.projs)
        return total

    def io_bytes(self) -> int:
        """Activation bytes per step: x (bf16) in, y (fp32) out."""
        return sum(self.M * p.K * 2 + self.M * p.N * 4 for p in self.projs)

    def macs(self) -> int:
        return sum(self.M * p.N * p.K for p in self.projs)

    def with_M(self, M: int, wtype: Optional[str] = None) -> "Workload":
        wt = wtype or self.wtype
        return Workload(f"{self.name.split('@')[0]}@{wt}-M{M}", self.family, wt, M, list(self.projs),
                        self.description)


def decoder(layers: int, H: int, I: int, qkv: int, vocab: int) -> List[Proj]:
    """The projections of a decoder in step order: per layer QKV (H -> qkv), O (H -> H), gate+up
    (H -> 2I), down (I -> H), then the lm_head (H -> vocab)."""
    projs = []
    for l in range(layers):
        projs.append(Proj(l, 0, H, qkv))
        projs.append(Proj(l, 1, H, H))
        projs.append(Proj(l, 2, H, 2 * I))
        projs.append(Proj(l, 3, I, H))
    projs.append(Proj(layers, 4, H, vocab))
    return projs


def _build():
    w = {}
    w["linear-2048"] = Workload(
        "linear-2048", 0, "bf16", 1, [Proj(0, 1, 2048, 2048)],
        "single linear y = x W^T, M=1, K=N=2048, bf16 (8 MB of weights)")
    w["1b-bf16"] = Workload(
        "1b-bf16", 1, "bf16", 1, decoder(22, 2048, 5632, 6144, 32000),
        "1B-class decode step, M=1, bf16: 22 layers, hidden 2048, QKV 2048->6144, O 2048->2048, "
        "gate+up 2048->11264, down 5632->2048, lm_head 2048->32000")
    w["7b-bf16"] = Workload(
        "7b-bf16", 7, "bf16", 1, decoder(32, 4096, 11008, 12288, 32000),
        "7B-class decode step, M=1, bf16: 32 layers, hidden 4096, QKV 4096->12288, O 4096->4096, "
        "gate+up 4096->22016, down 11008->4096, lm_head 4096->32000")
    w["7b-int8"] = Workload(
        "7b-int8", 7, "int8", 1, decoder(32, 4096, 11008, 12288, 32000),
        "7B-class decode step, M=1, int8 weight-only codes with per-output-channel bf16 scales")
    return w


WORKLOADS = _build()
PLD_WIDTHS = (1, 2, 4, 8)


def pld_workload(M: int, wtype: str) -> Workload:
    """Prompt-lookup verification width M on the 7B-class shapes."""
    base = WORKLOADS["7b-bf16"]
    return Workload(f"7b-pld-{wtype}-M{M}", 7, wtype, M, list(base.projs),
                    f"7B-class decode step, M={M} verification rows, {wtype}")


def tensor_key(seed: int, family: int, proj: Proj, kind: int) -> int:
    return key(seed, family * 1000 + proj.layer, proj.index, kind)


def gen_x(seed: int, wl: Workload, proj: Proj, M: Optional[int] = None, out=None):
    M = wl.M if M is None else M
    return normal_bf16(tensor_key(seed, wl.family, proj, KIND_X), 1.0, M * proj.K, 0, out)


def gen_w_bf16(seed: int, wl: Workload, proj: Proj, row0: int = 0, nrows: Optional[int] = None, out=None):
    nrows = proj.N - row0 if nrows is None else nrows
    return normal_bf16(tensor_key(seed, wl.family, proj, KIND_W), 1.0 / math.sqrt(proj.K),
                       nrows * proj.K, row0 * proj.K, out)


def gen_codes(seed: int, wl: Workload, proj: Proj, row0: int = 0, nrows: Optional[int] = None, out=None):
    nrows = proj.N - row0 if nrows is None else nrows
    return codes_i8(tensor_key(seed, wl.family, proj, KIND_Q), nrows * proj.K, row0 * proj.K, out)


def gen_scales(seed: int, wl: Workload, proj: Proj, row0: int = 0, nrows: Optional[int] = None, out=None):
    nrows = proj.N - row0 if nrows is None else nrows
    return uniform_bf16(tensor_key(seed, wl.family, proj, KIND_S), 1e-3, 1e-2, nrows, row0, out)


def gen_rows(seed: int, wl: Workload, proj: Proj, rows: np.ndarray):
    """Weights (and scales) of an arbitrary set of rows, regenerated one row at a time."""
    rows = np.asarray(rows, dtype=np.int64)
    if wl.wtype == "bf16":
        W = np.empty((len(rows), proj.K), dtype=np.uint16)
        for i, r in enumerate(rows):
            gen_w_bf16(seed, wl, proj, int(r), 1, out=W[i])
        return W, None
    Q = np.empty((len(rows), proj.K), dtype=np.int8)
    S = np.empty(len(rows), dtype=np.uint16)
    for i, r in enumerate(rows):
        gen_codes(seed, wl, proj, int(r), 1, out=Q[i])
        gen_scales(seed, wl, proj, int(r), 1, out=S[i:i + 1])
    return Q, S


@dataclass(frozen=True)
class ChainLink:
    """Where projection i of a chained step takes its x from (structure only, no arithmetic).

    op      XOP_RMSNORM: x = RMSNorm(h_in + y[src]) with norm weight `gamma`, the sum stored in
            residual buffer h_out; XOP_SWIGLU: x = SwiGLU of y[src] (gate | up halves);
            XOP_SLICE: x = columns [src_off, src_off + K) of y[src]; XOP_ATTENTION: x = attention
            of the new tokens over layer `layer`'s KV cache, q, k and v the thirds of y[src].
    src     index of the projection whose y feeds x (-1: none).
    h_in    residual buffer read (-1: the step's input h0, 0 / 1: the two residual buffers).
    h_out   residual buffer written (-1: none).
    """
    op: int
    K: int
    src: int = -1
    src_off: int = 0
    h_in: int = -1
    h_out: int = -1
    gamma: int = -1
    layer: int = -1


def chain_links(wl: Workload, attention: bool = False) -> List[ChainLink]:
    """Pre-norm decoder layers over the workload's projections (qkv, o, gate_up, down per layer,
    then lm_head).  Residual adds ride on the next RMSNorm; the two residual buffers alternate so
    that no buffer is written while another CTA may still read it (two grid barriers apart).
    attention: O's x is attention over the layer's KV cache (else the one-position V slice)."""
    links: List[ChainLink] = []
    base = {}
    for i, p in enumerate(wl.projs):
        base[(p.layer, p.index)] = i
    L = max(p.layer for p in wl.projs if p.index != 4) + 1
    for i, p in enumerate(wl.projs):
        l = p.layer
        if p.index == 0:      # qkv: x = RMSNorm(h), h = h_mid(l-1) + y_down(l-1)
            if l == 0:
                links.append(ChainLink(XOP_RMSNORM, p.K, gamma=0))
            else:
                links.append(ChainLink(XOP_RMSNORM, p.K, src=base[(l - 1, 3)], h_in=1, h_out=0, gamma=2 * l))
        elif p.index == 1 and attention:   # o: attention over the layer's KV cache
            links.append(ChainLink(XOP_ATTENTION, p.K, src=base[(l, 0)], layer=l))
        elif p.index == 1:    # o: attention over one position = the V third of qkv
            q = wl.projs[base[(l, 0)]]
            links.append(ChainLink(XOP_SLICE, p.K, src=base[(l, 0)], src_off=2 * q.N // 3))
        elif p.index == 2:    # gate_up: x = RMSNorm(h + y_o)
            links.append(ChainLink(XOP_RMSNORM, p.K, src=base[(l, 1)], h_in=-1 if l == 0 else 0, h_out=1,
                                   gamma=2 * l + 1))
        elif p.index == 3:    # down: x = SwiGLU(y_gate_up)
            links.append(ChainLink(XOP_SWIGLU, p.K, src=base[(l, 2)]))
        else:                 # lm_head: x = RMSNorm(h_mid(L-1) + y_down(L-1))
            links.append(ChainLink(XOP_RMSNORM, p.K, src=base[(L - 1, 3)], h_in=1, h_out=0, gamma=2 * L))
    return links


def hidden(wl: Workload) -> int:
    return wl.projs[0].K


def gen_h0(seed: int, wl: Workload, M: int):
    """The step's input residual stream [M, H] as fp32 (bf16-valued)."""
    H = hidden(wl)
    b = normal_bf16(key(seed, wl.family * 1000, 0, KIND_H0), 1.0, M * H)
    return (b.astype(np.uint32) << 16).view(np.float32).reshape(M, H)


def gen_gamma(seed: int, wl: Workload, norm: int, out=None):
    return uniform_bf16(key(seed, wl.family * 1000 + norm, 0, KIND_GAMMA), 0.5, 1.5, hidden(wl), 0, out)


def n_heads(wl: Workload) -> int:
    return hidden(wl) // HEAD_DIM


def gen_kv_cache(seed: int, wl: Workload, layer: int, L_max: int, out=None):
    """Layer `layer`'s KV cache [2][n_heads][L_max][128] as bf16 bits (K then V), N(0, 1)."""
    n = 2 * n_heads(wl) * L_max * HEAD_DIM
    return normal_bf16(key(seed, wl.family * 1000 + layer, 0, KIND_KV), 1.0, n, 0, out)


def n_norms(wl: Workload) -> int:
    return 2 * (max(p.layer for p in wl.projs if p.index != 4) + 1) + 1


def truncated(wl: Workload, layers: int) -> Workload:
    """The first `layers` decoder layers of wl plus its lm_head (small chained cases)."""
    L = max(p.layer for p in wl.projs)
    projs = [p for p in wl.projs if p.layer < layers or p.layer == L]
    return Workload(f"{wl.name}-{layers}layer", wl.family, wl.wtype, wl.M, projs, wl.description)
