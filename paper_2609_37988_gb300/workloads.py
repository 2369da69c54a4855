"""Seeded synthetic decode workloads shaped like the paper's models.

This module only draws random numbers: it holds none of the method's
arithmetic, and it is the one module both the GPU path's tests/bench and the
oracle's inputs come from.  Shapes follow Tab. backbones (Qwen2.5-7B:
28 layers, 4 KV heads; Qwen2.5-14B: 48 layers, 8 KV heads; head_dim 128) and
the MLA conversion of Appendix B (latent 512 + positional key 64).  The
paper's own evaluation data (IFEval, GSM8K, RULER, real checkpoints) are not
used; these tensors stand in for them.

Five workloads (``config(n)``):
 1  single-layer GQA toy: B=1, 8 q / 2 kv heads, d_h 64, T=512, fp32 K/V/q,
    int8 per-token groups of 64, sigma = 1/8.
 2  Qwen2.5-7B-shaped step: 28 layers, 28 q / 4 kv heads, B=16, T=8192, bf16
    q; layers (2i, 2i+1) share one cache; per-anchor precision drawn from
    {bf16, int8 g64, int4 g32} (1/3 each); keys per-channel, values per-token;
    K/V ~ N(0,1) x lognormal(0, 0.5) per (layer, head, channel).
 3  Qwen2.5-14B-shaped step: 48 layers, 40 q / 8 kv heads, B=32, T=8192
    (8191 cached + 1 appended per step); 16 inheritors drawn among layers
    1..47, the 32 anchors split 12 bf16 + 20 int4 g32 at random; per-token
    groups; K, V, q ~ N(0,1) bf16.
 4  MLA latent cache: 27 layers, 16 heads, latent 512 + k^R 64, head_dim 128,
    B=64, T=4096, bf16; per-layer kept width from {512, 256, 128, 64};
    latent coordinate k ~ N(0, 1/(k+1)); W_UK, W_UV ~ N(0, 1/512) (std
    512^-1/2); k^R, q_nope, q_pe ~ N(0,1).
 5  long context on 14B shapes: 48 layers, B=4, T=131072, pairs share, all
    anchors int4 g32 per-token, each (anchor, sequence) keeps a sorted uniform
    sample of T/8 positions.
"""
from __future__ import annotations

import math
import re
from dataclasses import dataclass, field

import numpy as np
import torch


@dataclass
class Workload:
    name: str
    kind: str                      # "gqa" or "mla"
    n_layers: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    batch: int
    context: int                   # positions read per step
    layers: list                   # per-layer dicts (inherit, bits, group, key_axis, width, evict_capacity, scheme)
    sigma: float
    q_dtype: torch.dtype
    kv_dtype: torch.dtype
    seed: int
    latent_dim: int = 0
    rope_dim: int = 0
    append_per_step: bool = False  # one appended position per anchor per step
    keep: int = 0                  # kept positions per (anchor, sequence), 0 = all
    kv_scale: dict = field(default_factory=dict)  # layer -> (k_scale[H,D], v_scale[H,D])

    @property
    def anchors(self):
        return [l for l, a in enumerate(self.layers) if not a["inherit"]]

    def sources(self):
        src, last = [], 0
        for l, a in enumerate(self.layers):
            if not a["inherit"]:
                last = l
            src.append(last)
        return src


def _layer(inherit=False, bits=16, group=64, key_axis="token", width=0, evict_capacity=0,
           scheme="grouped"):
    return dict(inherit=inherit, bits=bits, group=group, key_axis=key_axis, width=width,
                evict_capacity=evict_capacity, scheme=scheme)


def config(n: int, seed: int = None, *, batch: int = None, context: int = None,
           n_layers: int = None, sym_bits: int = None, mla_bits: int = None,
           mla_scheme: str = "symmetric") -> Workload:
    """Workload ``n`` (1..5).  ``batch``/``context``/``n_layers`` shrink it
    for oracle-sized tests while keeping the per-layer draws.  ``sym_bits``
    (8, 4 or 2) stores every quantised anchor with the paper's symmetric
    per-vector quantiser at that bit-width instead (per-token rows; the
    plan, shapes and inputs are otherwise unchanged).  ``mla_bits`` (8, 4 or
    2; MLA workload only) stores every latent layer quantised as well (all
    three axes), each position's kept latent and positional key one vector
    each, with ``mla_scheme`` ``"symmetric"`` or ``"grouped"``."""
    seed = n if seed is None else seed
    rng = np.random.default_rng(seed)
    if n == 1:
        w = Workload("gqa-toy-b1-h8kv2-d64-t512-int8g64", "gqa", 1, 8, 2, 64, 1, 512,
                     [_layer(bits=8, group=64)], 1.0 / 8.0, torch.float32, torch.float32, seed)
    elif n == 2:
        L = 28
        layers = []
        for i in range(L // 2):
            bits = int(rng.choice([16, 8, 4]))
            grp = {16: 64, 8: 64, 4: 32}[bits]
            layers.append(_layer(bits=bits, group=grp, key_axis="channel" if bits != 16 else "token"))
            layers.append(_layer(inherit=True))
        w = Workload("qwen2.5-7b-b16-t8192-mixed-pairs", "gqa", L, 28, 4, 128, 16, 8192, layers,
                     1.0 / math.sqrt(128), torch.bfloat16, torch.bfloat16, seed)
        for l in w.anchors:
            w.kv_scale[l] = (rng.lognormal(0.0, 0.5, (4, 128)).astype(np.float32),
                             rng.lognormal(0.0, 0.5, (4, 128)).astype(np.float32))
    elif n == 3:
        L = 48
        inh = set((rng.choice(47, 16, replace=False) + 1).tolist())
        anchors = [l for l in range(L) if l not in inh]
        kinds = rng.permutation([16] * 12 + [4] * 20)
        bits_of = dict(zip(anchors, kinds.tolist()))
        layers = [_layer(inherit=True) if l in inh else
                  _layer(bits=int(bits_of[l]), group=32 if bits_of[l] == 4 else 64) for l in range(L)]
        w = Workload("qwen2.5-14b-b32-t8192-12bf16-20int4-16inherit", "gqa", L, 40, 8, 128, 32,
                     8192, layers, 1.0 / math.sqrt(128), torch.bfloat16, torch.bfloat16, seed,
                     append_per_step=True)
    elif n == 4:
        L = 27
        widths = rng.choice([512, 256, 128, 64], L).tolist()
        layers = [_layer(bits=16, width=int(d)) for d in widths]
        w = Workload("mla-l27-h16-r512-b64-t4096", "mla", L, 16, 1, 128, 64, 4096, layers,
                     1.0 / math.sqrt(128 + 64), torch.bfloat16, torch.bfloat16, seed,
                     latent_dim=512, rope_dim=64)
    elif n == 5:
        L, T = 48, 131072
        layers = []
        for i in range(L // 2):
            layers.append(_layer(bits=4, group=32, evict_capacity=T // 8))
            layers.append(_layer(inherit=True))
        w = Workload("qwen2.5-14b-b4-t131072-keep1of8-int4-pairs", "gqa", L, 40, 8, 128, 4, T,
                     layers, 1.0 / math.sqrt(128), torch.bfloat16, torch.bfloat16, seed, keep=T // 8)
    else:
        raise ValueError(f"no workload {n}")
    if sym_bits is not None:
        if sym_bits not in (8, 4, 2) or w.kind != "gqa" or w.head_dim != 128:
            raise ValueError("symmetric anchors: 8, 4 or 2 bits on a head_dim-128 GQA workload")
        for a in w.layers:
            if not a["inherit"] and a["bits"] != 16:
                a.update(bits=sym_bits, scheme="symmetric", key_axis="token")
        if re.search(r"int\d", w.name):
            w.name = re.sub(r"int\d", f"sym{sym_bits}", w.name)
        else:
            w.name += f"-sym{sym_bits}"
    if mla_bits is not None:
        if mla_bits not in (8, 4, 2) or w.kind != "mla" or mla_scheme not in ("symmetric", "grouped") \
                or (mla_bits == 2 and mla_scheme == "grouped"):
            raise ValueError("quantised latents: symmetric 8/4/2 or grouped 8/4 bits on the MLA workload")
        for a in w.layers:
            a.update(bits=mla_bits, scheme=mla_scheme)
        w.name += f"-{'sym' if mla_scheme == 'symmetric' else 'int'}{mla_bits}"
    if batch is not None:
        w.batch = batch
    if n_layers is not None:
        w.layers = w.layers[:n_layers]
        w.n_layers = n_layers
    if context is not None:
        w.context = context
        if w.keep:
            w.keep = max(1, context // 8)
            for a in w.layers:
                if not a["inherit"]:
                    a["evict_capacity"] = w.keep
    return w


def _gen(seed: int, ids, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed((seed * 1_000_003 + sum((i + 1) * 7919 ** k for k, i in enumerate(ids))) % (2 ** 63))
    return g


def randn(shape, seed: int, *ids, dtype=torch.float32, device="cpu", std=1.0) -> torch.Tensor:
    """N(0, std^2) tensor from a generator keyed by (seed, ids), drawn on
    ``device`` in float32 and then cast.  The values depend on the device's
    generator; tests hand the oracle the very tensors the GPU received."""
    dev = torch.device(device)
    t = torch.randn(shape, generator=_gen(seed, ids, dev), dtype=torch.float32, device=dev)
    if std != 1.0:
        t = t * std
    return t.to(dtype=dtype)


def kv_inputs(w: Workload, layer: int, t0: int, t1: int, device="cpu"):
    """Keys and values written to anchor ``layer`` for positions [t0, t1):
    ``[B, t1-t0, H_kv, D]`` in the workload's K/V dtype.  Generated per
    position block so any range reproduces the same values."""
    B, H, D = w.batch, w.n_kv_heads, w.head_dim
    ks, vs = [], []
    blk = 1024
    for p0 in range(t0 - t0 % blk, t1, blk):
        k = randn((B, blk, H, D), w.seed, layer, 0, p0 // blk, device=device)
        v = randn((B, blk, H, D), w.seed, layer, 1, p0 // blk, device=device)
        lo, hi = max(t0, p0) - p0, min(t1, p0 + blk) - p0
        ks.append(k[:, lo:hi]); vs.append(v[:, lo:hi])
    k = torch.cat(ks, 1); v = torch.cat(vs, 1)
    if layer in w.kv_scale:
        sk, sv = w.kv_scale[layer]
        k = k * torch.from_numpy(sk).to(k.device)[None, None]
        v = v * torch.from_numpy(sv).to(v.device)[None, None]
    return k.to(dtype=w.kv_dtype), v.to(dtype=w.kv_dtype)


def queries(w: Workload, layer: int, step: int = 0, device="cpu") -> torch.Tensor:
    """Query ``[B, H_q, D]`` of ``layer`` at decode step ``step``."""
    return randn((w.batch, w.n_q_heads, w.head_dim), w.seed, layer, 2, step,
                 dtype=w.q_dtype, device=device)


def window_queries(w: Workload, layer: int, n_win: int, device="cpu") -> torch.Tensor:
    """Queries of each sequence's last ``n_win`` positions (the eviction
    observation window) ``[B, n_win, H_q, D]``."""
    return randn((w.batch, n_win, w.n_q_heads, w.head_dim), w.seed, layer, 10,
                 dtype=w.q_dtype, device=device)


def kept_positions(w: Workload, layer: int, lens, device="cpu"):
    """Sorted uniform samples of ``w.keep`` positions per sequence:
    (idx ``[B, keep]`` int32, n_kept ``[B]`` int32)."""
    rng = np.random.default_rng([w.seed, layer, 5])
    idx = np.zeros((w.batch, w.keep), np.int32)
    n = np.zeros(w.batch, np.int32)
    for b in range(w.batch):
        k = min(w.keep, int(lens[b]))
        idx[b, :k] = np.sort(rng.choice(int(lens[b]), k, replace=False))
        n[b] = k
    return torch.from_numpy(idx).to(device), torch.from_numpy(n).to(device)


def mla_inputs(w: Workload, layer: int, t0: int, t1: int, device="cpu"):
    """Latent ``[B, t1-t0, r]`` (coordinate k scaled by (k+1)^-1/2) and
    positional key ``[B, t1-t0, d_R]``, bf16."""
    B, r, dR = w.batch, w.latent_dim, w.rope_dim
    cs, ks = [], []
    blk = 1024
    decay = torch.arange(r, dtype=torch.float32, device=device).add(1.0).rsqrt()
    for p0 in range(t0 - t0 % blk, t1, blk):
        c = randn((B, blk, r), w.seed, layer, 3, p0 // blk, device=device) * decay
        k = randn((B, blk, dR), w.seed, layer, 4, p0 // blk, device=device)
        lo, hi = max(t0, p0) - p0, min(t1, p0 + blk) - p0
        cs.append(c[:, lo:hi]); ks.append(k[:, lo:hi])
    return torch.cat(cs, 1).to(torch.bfloat16), torch.cat(ks, 1).to(torch.bfloat16)


def mla_weights(w: Workload, layer: int, device="cpu"):
    """W_UK, W_UV ``[H, 128, r]`` bf16 with std r^-1/2 (r = 512)."""
    H, r = w.n_q_heads, w.latent_dim
    std = 1.0 / math.sqrt(512)
    wk = randn((H, w.head_dim, r), w.seed, layer, 6, std=std, dtype=torch.bfloat16, device=device)
    wv = randn((H, w.head_dim, r), w.seed, layer, 7, std=std, dtype=torch.bfloat16, device=device)
    return wk, wv


def mla_queries(w: Workload, layer: int, step: int = 0, device="cpu"):
    """q_nope ``[B, H, 128]`` and post-RoPE q_pe ``[B, H, 64]``, bf16."""
    qn = randn((w.batch, w.n_q_heads, w.head_dim), w.seed, layer, 8, step, dtype=torch.bfloat16,
               device=device)
    qp = randn((w.batch, w.n_q_heads, w.rope_dim), w.seed, layer, 9, step, dtype=torch.bfloat16,
               device=device)
    return qn, qp
