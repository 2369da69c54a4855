"""Thin PyTorch-facing wrapper of the C ABI (include/kvk.h).

PyTorch provides device memory (arenas, workspace, outputs) and the current
CUDA stream; every computation runs in ``libkvk.so``.  A :class:`Cache`
holds one per-layer plan (Sec. 2.2 of the paper: inherit, or a cache at some
bit-width / kept width) for a fixed model geometry.
"""
from __future__ import annotations

import ctypes
from dataclasses import dataclass

import torch

from . import _lib
from ._lib import (AXIS_CHANNEL, AXIS_TOKEN, DTYPE_BF16, DTYPE_F32, KIND_GQA, KIND_MLA,
                   QUANT_GROUPED, QUANT_SYMMETRIC, KVKError, LayerCfg, ModelDesc, check, load)

__all__ = ["Layer", "Cache", "splitk_reduce", "KVKError"]


@dataclass
class Layer:
    """One plan action.  ``inherit=True`` is the depth action; otherwise a
    cache at ``bits`` (16, 8, 4, 2) quantised with ``scheme`` ``"grouped"``
    (asymmetric, ``group`` elements per scale/zero pair, key axis
    ``"token"``/``"channel"``) or ``"symmetric"`` (one bf16 scale per
    token-head row), MLA kept ``width``, optional eviction list capacity."""
    inherit: bool = False
    bits: int = 16
    group: int = 64
    key_axis: str = "token"
    width: int = 0
    evict_capacity: int = 0
    scheme: str = "grouped"

    def to_c(self) -> LayerCfg:
        if self.scheme not in ("grouped", "symmetric"):
            raise ValueError(f"unknown quantisation scheme {self.scheme!r}")
        return LayerCfg(int(self.inherit), self.bits, self.group,
                        AXIS_CHANNEL if self.key_axis == "channel" else AXIS_TOKEN,
                        AXIS_TOKEN, self.width, self.evict_capacity,
                        QUANT_SYMMETRIC if self.scheme == "symmetric" else QUANT_GROUPED)


def _ptr(t):
    return ctypes.c_void_p(0 if t is None else t.data_ptr())


def _stream(stream=None):
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.float32:
        return DTYPE_F32
    if t.dtype == torch.bfloat16:
        return DTYPE_BF16
    raise TypeError(f"unsupported dtype {t.dtype}")


def _need(t: torch.Tensor, name: str):
    if not (t.is_cuda and t.is_contiguous()):
        raise ValueError(f"{name} must be a contiguous CUDA tensor")


class Cache:
    """A compressed KV cache for one model geometry and one plan."""

    def __init__(self, *, kind: str = "gqa", n_layers: int, n_q_heads: int, n_kv_heads: int = 1,
                 head_dim: int = 128, latent_dim: int = 0, rope_dim: int = 0, max_batch: int,
                 max_ctx: int, layers, max_splits: int = 64, device=None):
        self.lib = load()
        self.desc = ModelDesc(KIND_MLA if kind == "mla" else KIND_GQA, n_layers, n_q_heads,
                              n_kv_heads, head_dim, latent_dim, rope_dim, max_batch, max_ctx)
        self.kind = kind
        self.layers = list(layers)
        if len(self.layers) != n_layers:
            raise ValueError("one Layer per model layer")
        cfg = (LayerCfg * n_layers)(*[l.to_c() for l in self.layers])
        self._cfg = cfg
        sizes = (ctypes.c_size_t * n_layers)()
        check(self.lib.kvk_cache_plan(ctypes.byref(self.desc), cfg, sizes))
        ws = ctypes.c_size_t()
        check(self.lib.kvk_workspace_size(ctypes.byref(self.desc), max_splits, ctypes.byref(ws)))
        dev = torch.device(device) if device is not None else torch.device("cuda", torch.cuda.current_device())
        self.device = dev
        self.arena_bytes = [int(s) for s in sizes]
        # torch's caching allocator returns 512-byte aligned blocks
        self.arenas = [torch.empty(n, dtype=torch.uint8, device=dev) if n else None
                       for n in self.arena_bytes]
        self.workspace = torch.empty(int(ws.value), dtype=torch.uint8, device=dev)
        ptrs = (ctypes.c_void_p * n_layers)(*[0 if a is None else a.data_ptr() for a in self.arenas])
        h = ctypes.c_void_p()
        with torch.cuda.device(dev):
            check(self.lib.kvk_cache_create(ctypes.byref(self.desc), cfg, ptrs,
                                            _ptr(self.workspace), ws.value, max_splits,
                                            ctypes.byref(h)))
        self.handle = h
        self.max_splits = max_splits
        self.reset()

    # -- lifetime ------------------------------------------------------------
    def close(self):
        if getattr(self, "handle", None):
            self.lib.kvk_cache_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def reset(self, stream=None):
        check(self.lib.kvk_cache_reset(self.handle, _stream(stream)))

    WAIT_LIMIT_DEFAULT = 4194304

    def set_wait_limit(self, polls: int):
        """Polls a decode kernel's bounded wait makes in its tile loop before
        giving up (0: at the first poll, setting the timeout error)."""
        check(self.lib.kvk_set_wait_limit(self.handle, int(polls)))

    SCHEDULE_AUTO, SCHEDULE_SPLITS, SCHEDULE_RUNS = 0, 1, 2

    def set_decode_schedule(self, schedule: int, run_ctas: int = 0, run_setup: int = -1):
        """How automatic GQA decodes partition the work: SCHEDULE_SPLITS (equal
        context splits per unit), SCHEDULE_RUNS (equal runs of the flattened
        unit x tile grid, where the format has them) or SCHEDULE_AUTO;
        run_ctas: CTAs of a run decode (0: whole waves of resident CTAs);
        run_setup: planned tiles charged to each unit's start (-1: default)."""
        check(self.lib.kvk_set_decode_schedule(self.handle, int(schedule), int(run_ctas),
                                               int(run_setup)))

    # -- plan ----------------------------------------------------------------
    def source(self, layer: int) -> int:
        out = ctypes.c_int32()
        check(self.lib.kvk_layer_source(self.handle, layer, ctypes.byref(out)))
        return out.value

    def lengths(self, layer: int) -> torch.Tensor:
        """Device int32[max_batch] lengths of the anchor ``layer`` reads (a view)."""
        src = self.source(layer)
        return self.arenas[src][: 4 * self.desc.max_batch].view(torch.int32)

    def cost(self):
        b, s, r = ctypes.c_double(), ctypes.c_double(), ctypes.c_double()
        check(self.lib.kvk_cost(self.handle, ctypes.byref(b), ctypes.byref(s), ctypes.byref(r)))
        return {"bits_per_token_model": b.value, "bytes_per_token_stored": s.value, "rho": r.value}

    # -- writes --------------------------------------------------------------
    def append(self, layer: int, k: torch.Tensor, v: torch.Tensor, n_per_seq: torch.Tensor = None,
               stream=None):
        """GQA: k, v ``[B, n, H_kv, D]`` (fp32/bf16).  MLA: k = latent
        ``[B, n, r]`` bf16, v = positional key ``[B, n, d_R]`` bf16."""
        _need(k, "k"); _need(v, "v")
        n = int(k.shape[1])
        if n_per_seq is not None:
            _need(n_per_seq, "n_per_seq")
        check(self.lib.kvk_append(self.handle, layer, _ptr(k), _ptr(v), _dtype_code(k), n,
                                  _ptr(n_per_seq), _stream(stream)))

    def set_kept(self, layer: int, idx: torch.Tensor = None, n_kept: torch.Tensor = None,
                 stream=None):
        if n_kept is not None:
            _need(idx, "idx"); _need(n_kept, "n_kept")
        check(self.lib.kvk_set_kept(self.handle, layer, _ptr(idx), _ptr(n_kept), _stream(stream)))

    def evict_window(self, layer: int, q_win: torch.Tensor, scale: float, budget: int,
                     stream=None):
        """Attention-scored eviction: ``q_win`` ``[B, n_win, H_q, head_dim]``,
        the queries of each sequence's last ``n_win`` positions; installs
        per-(sequence, KV head) kept lists of ``budget`` positions.  Returns
        the votes, a float32 view ``[max_batch, H_kv, C]`` of the scratch
        (valid before each window of the sequences longer than ``budget``,
        once the stream has run the call)."""
        _need(q_win, "q_win")
        d = self.desc
        if q_win.dim() != 4 or (q_win.shape[0], q_win.shape[2], q_win.shape[3]) != (
                d.max_batch, d.n_q_heads, d.head_dim):
            raise ValueError("q_win must be [max_batch, n_win, n_q_heads, head_dim]")
        n_win = q_win.shape[1]
        nbytes = ctypes.c_size_t()
        check(self.lib.kvk_evict_scratch_size(self.handle, layer, n_win, ctypes.byref(nbytes)))
        scratch = torch.empty(nbytes.value, dtype=torch.uint8, device=self.device)
        check(self.lib.kvk_evict_window(self.handle, layer, _ptr(q_win), _dtype_code(q_win), n_win,
                                        float(scale), budget, _ptr(scratch), nbytes.value,
                                        _stream(stream)))
        self._evict_scratch = scratch  # kept alive until the stream is done with it
        C = (d.max_ctx + 63) // 64 * 64
        return scratch[: 4 * d.max_batch * d.n_kv_heads * C].view(torch.float32).view(
            d.max_batch, d.n_kv_heads, C)

    def prefill(self, layer: int, q: torch.Tensor, scale: float, out: torch.Tensor = None,
                stream=None) -> torch.Tensor:
        """Causal chunk attention of ``q`` ``[B, n_q, H_q, head_dim]``, the
        queries of each sequence's last ``n_q`` positions (appended first),
        over the compressed cache; returns float32 ``[B, n_q, H_q, head_dim]``."""
        _need(q, "q")
        d = self.desc
        if q.dim() != 4 or (q.shape[0], q.shape[2], q.shape[3]) != (d.max_batch, d.n_q_heads, d.head_dim):
            raise ValueError("q must be [max_batch, n_q, n_q_heads, head_dim]")
        n_q = q.shape[1]
        if out is None:
            out = torch.empty(q.shape, dtype=torch.float32, device=q.device)
        nbytes = ctypes.c_size_t()
        check(self.lib.kvk_prefill_scratch_size(self.handle, layer, n_q, ctypes.byref(nbytes)))
        scratch = torch.empty(nbytes.value, dtype=torch.uint8, device=self.device)
        check(self.lib.kvk_prefill_attention(self.handle, layer, _ptr(q), _dtype_code(q), n_q,
                                             float(scale), _ptr(out), _ptr(scratch), nbytes.value,
                                             _stream(stream)))
        self._prefill_scratch = scratch  # kept alive until the stream is done with it
        return out

    def prefill_mla(self, layer: int, q_nope: torch.Tensor, q_pe: torch.Tensor, w_uk: torch.Tensor,
                    w_uv: torch.Tensor, scale: float, out: torch.Tensor = None, stream=None) -> torch.Tensor:
        """MLA causal chunk attention: ``q_nope`` ``[B, n_q, H, head_dim]`` and
        ``q_pe`` ``[B, n_q, H, rope_dim]`` (bf16), the queries of each
        sequence's last ``n_q`` positions (appended first); returns float32
        ``[B, n_q, H, head_dim]``."""
        for t, n in ((q_nope, "q_nope"), (q_pe, "q_pe"), (w_uk, "w_uk"), (w_uv, "w_uv")):
            _need(t, n)
        d = self.desc
        if q_nope.dim() != 4 or (q_nope.shape[0], q_nope.shape[2], q_nope.shape[3]) != \
                (d.max_batch, d.n_q_heads, d.head_dim) or q_pe.shape != q_nope.shape[:3] + (d.rope_dim,):
            raise ValueError("q_nope must be [max_batch, n_q, n_q_heads, head_dim], q_pe [.., rope_dim]")
        n_q = q_nope.shape[1]
        if out is None:
            out = torch.empty(q_nope.shape, dtype=torch.float32, device=q_nope.device)
        nbytes = ctypes.c_size_t()
        check(self.lib.kvk_prefill_scratch_size(self.handle, layer, n_q, ctypes.byref(nbytes)))
        scratch = torch.empty(nbytes.value, dtype=torch.uint8, device=self.device)
        check(self.lib.kvk_prefill_attention_mla(self.handle, layer, _ptr(q_nope), _ptr(q_pe), _ptr(w_uk),
                                                 _ptr(w_uv), n_q, float(scale), _ptr(out), _ptr(scratch),
                                                 nbytes.value, _stream(stream)))
        self._prefill_scratch = scratch  # kept alive until the stream is done with it
        return out

    def kept_lists(self, layer: int, stream=None):
        """Installed kept lists: ``(idx, n, per_head)`` device tensors shaped
        per head ``[B, H_kv, cap]`` / ``[B, H_kv]`` (or per sequence), or
        ``None`` when no list is installed."""
        d = self.desc
        cap = self.layers[layer].evict_capacity
        idx = torch.empty((d.max_batch, d.n_kv_heads, max(cap, 1)), dtype=torch.int32,
                          device=self.device)
        n = torch.empty((d.max_batch, d.n_kv_heads), dtype=torch.int32, device=self.device)
        ph = ctypes.c_int32()
        check(self.lib.kvk_export_kept(self.handle, layer, _ptr(idx), _ptr(n), ctypes.byref(ph),
                                       _stream(stream)))
        if ph.value < 0:
            return None
        if ph.value == 0:
            flat_i = idx.view(-1)[: d.max_batch * cap].view(d.max_batch, cap)
            return flat_i, n.view(-1)[: d.max_batch].clone(), False
        return idx, n, True

    def rewind(self, n: int, stream=None):
        """Drop the last ``n`` positions of every sequence of every anchor."""
        check(self.lib.kvk_rewind(self.handle, n, _stream(stream)))

    # -- reads ---------------------------------------------------------------
    def plan_splits(self, layer: int) -> int:
        out = ctypes.c_int32()
        check(self.lib.kvk_decode_plan_splits(self.handle, layer, ctypes.byref(out)))
        return out.value

    def decode(self, layer: int, q: torch.Tensor, scale: float, out: torch.Tensor = None,
               n_splits: int = 0, stream=None) -> torch.Tensor:
        _need(q, "q")
        if out is None:
            out = torch.empty(q.shape, dtype=torch.float32, device=q.device)
        check(self.lib.kvk_decode_attention(self.handle, layer, _ptr(q), _dtype_code(q),
                                            float(scale), _ptr(out), n_splits, _stream(stream)))
        return out

    def decode_partial(self, layer: int, q: torch.Tensor, scale: float, n_splits: int,
                       partials: torch.Tensor = None, stream=None) -> torch.Tensor:
        _need(q, "q")
        B, Hq, D = q.shape
        if partials is None:
            n = n_splits if n_splits > 0 else self.plan_splits(layer)
            partials = torch.empty((n, B * Hq, D + 2), dtype=torch.float32, device=q.device)
        check(self.lib.kvk_decode_partial(self.handle, layer, _ptr(q), _dtype_code(q), float(scale),
                                          _ptr(partials), n_splits, _stream(stream)))
        return partials

    def decode_mla(self, layer: int, q_nope, q_pe, w_uk, w_uv, scale: float, out=None,
                   n_splits: int = 0, stream=None) -> torch.Tensor:
        for t, nm in ((q_nope, "q_nope"), (q_pe, "q_pe"), (w_uk, "w_uk"), (w_uv, "w_uv")):
            _need(t, nm)
        if out is None:
            out = torch.empty(q_nope.shape, dtype=torch.float32, device=q_nope.device)
        check(self.lib.kvk_decode_attention_mla(self.handle, layer, _ptr(q_nope), _ptr(q_pe),
                                                _ptr(w_uk), _ptr(w_uv), float(scale), _ptr(out),
                                                n_splits, _stream(stream)))
        return out

    def export(self, layer: int, stream=None) -> dict:
        """Stored state of anchor ``layer`` in canonical order (device tensors)."""
        d = self.desc
        L = self.layers[layer]
        B, T = d.max_batch, d.max_ctx
        dev = self.device
        res = {}
        if self.kind == "mla":
            if L.bits == 16:
                res["c"] = torch.empty((B, T, L.width), dtype=torch.bfloat16, device=dev)
                res["k_r"] = torch.empty((B, T, d.rope_dim), dtype=torch.bfloat16, device=dev)
                check(self.lib.kvk_export_layer(self.handle, layer, _ptr(res["c"]), _ptr(res["k_r"]),
                                                None, None, None, None, None, _stream(stream)))
                return res
            # quantised latents: codes (signed for the symmetric scheme) and
            # per-position scales (and zeros) of the latent and of k^R
            ct = torch.int8 if L.scheme == "symmetric" else torch.uint8
            res["c_codes"] = torch.empty((B, T, L.width), dtype=ct, device=dev)
            res["kr_codes"] = torch.empty((B, T, d.rope_dim), dtype=ct, device=dev)
            for k in ("c_scale", "c_zero", "kr_scale", "kr_zero"):
                res[k] = torch.empty((B, T), dtype=torch.float32, device=dev)
            check(self.lib.kvk_export_layer(self.handle, layer, _ptr(res["c_codes"]),
                                            _ptr(res["kr_codes"]), _ptr(res["c_scale"]),
                                            _ptr(res["c_zero"]), _ptr(res["kr_scale"]),
                                            _ptr(res["kr_zero"]), None, _stream(stream)))
            return res
        H, D = d.n_kv_heads, d.head_dim
        if L.bits == 16:
            res["k"] = torch.empty((B, H, T, D), dtype=torch.bfloat16, device=dev)
            res["v"] = torch.empty((B, H, T, D), dtype=torch.bfloat16, device=dev)
            check(self.lib.kvk_export_layer(self.handle, layer, _ptr(res["k"]), _ptr(res["v"]),
                                            None, None, None, None, None, _stream(stream)))
            return res
        if L.scheme == "symmetric":
            res["k_codes"] = torch.empty((B, H, T, D), dtype=torch.int8, device=dev)
            res["v_codes"] = torch.empty((B, H, T, D), dtype=torch.int8, device=dev)
            res["k_scale"] = torch.empty((B, H, T), dtype=torch.float32, device=dev)
            res["v_scale"] = torch.empty((B, H, T), dtype=torch.float32, device=dev)
            check(self.lib.kvk_export_layer(self.handle, layer, _ptr(res["k_codes"]),
                                            _ptr(res["v_codes"]), _ptr(res["k_scale"]), None,
                                            _ptr(res["v_scale"]), None, None, _stream(stream)))
            return res
        g = L.group
        res["k_codes"] = torch.empty((B, H, T, D), dtype=torch.uint8, device=dev)
        res["v_codes"] = torch.empty((B, H, T, D), dtype=torch.uint8, device=dev)
        res["v_scale"] = torch.empty((B, H, T, D // g), dtype=torch.float32, device=dev)
        res["v_zero"] = torch.empty((B, H, T, D // g), dtype=torch.float32, device=dev)
        if L.key_axis == "channel":
            res["k_scale"] = torch.empty((B, H, T // g, D), dtype=torch.float32, device=dev)
            res["k_zero"] = torch.empty((B, H, T // g, D), dtype=torch.float32, device=dev)
            res["k_residual"] = torch.empty((B, H, g, D), dtype=torch.bfloat16, device=dev)
        else:
            res["k_scale"] = torch.empty((B, H, T, D // g), dtype=torch.float32, device=dev)
            res["k_zero"] = torch.empty((B, H, T, D // g), dtype=torch.float32, device=dev)
            res["k_residual"] = None
        check(self.lib.kvk_export_layer(self.handle, layer, _ptr(res["k_codes"]), _ptr(res["v_codes"]),
                                        _ptr(res["k_scale"]), _ptr(res["k_zero"]), _ptr(res["v_scale"]),
                                        _ptr(res["v_zero"]), _ptr(res["k_residual"]), _stream(stream)))
        return res

    def device_error(self, stream=None) -> int:
        """Synchronise, read and clear the device error word (0 = none)."""
        code = ctypes.c_int32()
        st = self.lib.kvk_get_device_error(self.handle, _stream(stream), ctypes.byref(code))
        if st not in (0, 7):
            check(st)
        return code.value


def splitk_reduce(partials: torch.Tensor, out: torch.Tensor = None, stream=None) -> torch.Tensor:
    """Merge ``[n_splits, rows, dim + 2]`` partials into ``[rows, dim]``."""
    _need(partials, "partials")
    S, R, W = partials.shape
    if out is None:
        out = torch.empty((R, W - 2), dtype=torch.float32, device=partials.device)
    check(load().kvk_splitk_reduce(_ptr(partials), S, R, W - 2, _ptr(out), _stream(stream)))
    return out
