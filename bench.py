"""Decode-step benchmark of the compressed-KV path on GB300.

Default workload: the Qwen2.5-14B-shaped mixed plan (48 layers, 40 q / 8 kv
heads, head_dim 128, batch 32, 8191 cached positions + 1 appended per step,
12 bf16 + 20 int4 g32 anchors, 16 inheriting layers).  One step = append one
position to every anchor, decode attention for all 48 layers (inheritors
read their source anchor with their own query), then roll the appended
position back so every step reads exactly 8192 positions.

Metric: achieved HBM GB/s of algorithmic bytes (compressed cache bytes every
layer reads, plus query/output/append traffic) per step, and ms per step.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]

Prints one JSON line (rank 0).  Under torchrun each rank runs its own
replica of the workload (independent sequences; no collective on the data
path) and the line reports the sum over ranks divided by the slowest rank.
"""
from __future__ import annotations

import argparse
import dataclasses
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "decode-attention achieved HBM GB/s and % of GB300 peak; per-step latency (us)"
UNIT = "GB/s"


# ---------------------------------------------------------------------------
def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


def _record_bytes(w, l):
    """Bytes stored per (position, kv head) by anchor l: one record, with the
    group metadata (per-token formats) or the two bf16 scales (symmetric)."""
    return _rec_bytes(w.layers[l], w.head_dim)


def _rec_bytes(a, D):
    if a["bits"] == 16:
        return 4 * D
    if a.get("scheme") == "symmetric":
        return 2 * D * a["bits"] // 8 + 2 * 2
    return 2 * D * a["bits"] // 8 + 2 * 8 * D // a["group"]


def algorithmic_bytes(w, lens_after_append):
    """Bytes one step must move: each layer reads its source anchor's records
    at the current length (per-token formats: rec bytes per (position, kv
    head)); queries read, outputs written; appended rows read and written."""
    B, H, D = w.batch, w.n_kv_heads, w.head_dim
    src = w.sources()
    total = 0
    per_layer = []
    for l in range(w.n_layers):
        a = w.layers[src[l]]
        rec = _record_bytes(w, src[l])
        n = w.keep if w.keep else lens_after_append
        cache = B * H * n * rec
        qo = B * w.n_q_heads * D * (2 + 4)
        per_layer.append(cache)
        total += cache + qo
        if not a["inherit"] and w.append_per_step and not w.layers[l]["inherit"]:
            total += B * H * D * 2 * 2 + B * H * rec
    return total, per_layer


def mla_position_bytes(w, l):
    """Stored bytes of one position of MLA layer l: [c[:d] | k^R] in bf16,
    or their codes plus the two vectors' scales (and zeros)."""
    a = w.layers[l]
    n = a["width"] + w.rope_dim
    if a["bits"] == 16:
        return 2 * n
    return n * a["bits"] // 8 + (4 if a.get("scheme") == "symmetric" else 16)


def algorithmic_bytes_mla(w, T):
    """MLA step: every layer reads its latent cache [c[:d] | k^R] at length
    T (bf16, or codes and per-position metadata), the absorbed /
    up-projection weight slices W_UK[:, :, :d] and W_UV[:, :, :d], its
    queries, and writes its output."""
    B, H = w.batch, w.n_q_heads
    total, per_layer = 0, []
    for l in range(w.n_layers):
        d = w.layers[l]["width"]
        cache = B * T * mla_position_bytes(w, l)
        per_layer.append(cache)
        total += cache + 2 * H * w.head_dim * d * 2 + B * H * (w.head_dim + w.rope_dim) * 2 + \
            B * H * w.head_dim * 4
    return total, per_layer


class Clocks:
    """nvidia-smi sampler running during the timed region."""

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.path = None

    def __enter__(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index),
                 "--query-gpu=timestamp,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
                 "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
                 "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap",
                 "--format=csv,noheader,nounits", "-lms", "10"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
            # the timed region starts once the sampler is producing rows
            t0 = time.perf_counter()
            while time.perf_counter() - t0 < 10.0 and self.proc.poll() is None:
                if os.path.getsize(self.path) > 0:
                    break
                time.sleep(0.01)
        except Exception:
            self.proc = None
        return self

    def mark(self, which):
        """Host wall-clock time of the start or end of the timed region."""
        setattr(self, "t_" + which, time.time())

    def __exit__(self, *exc):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        if not self.proc or not self.path:
            return None
        import datetime
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) >= 9:
                    try:
                        ts = datetime.datetime.strptime(parts[0], "%Y/%m/%d %H:%M:%S.%f").timestamp()
                    except ValueError:
                        ts = None
                    rows.append((ts, parts[1:]))
        os.unlink(self.path)
        # rows sampled inside the timed region (all rows if none carry a
        # usable time stamp or the region was too short to hold one)
        t0, t1 = getattr(self, "t_start", None), getattr(self, "t_end", None)
        inside = [r for ts, r in rows if ts is not None and t0 is not None and t1 is not None
                  and t0 <= ts <= t1]
        rows = inside or [r for _, r in rows]
        if not rows:
            return None
        sm = [float(r[0]) for r in rows if r[0].replace(".", "").isdigit()]
        mx = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({n for r in rows for n, v in zip(names, r[4:8]) if v.lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons, "samples": len(rows),
                "samples_in_timed_region": len(inside), "interval_ms": 10}


def reduce_max(x: float, dist=None, device=None) -> float:
    """Maximum of ``x`` over ranks (the slowest rank sets the job time)."""
    if dist is None:
        return x
    import torch
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(step_bytes: int, steps: int, world: int, seconds: float) -> float:
    """Whole-job GB/s: every rank moves ``step_bytes`` per step (weak
    scaling), divided by the slowest rank's time."""
    return step_bytes * steps * world / seconds / 1e9


# ---------------------------------------------------------------------------
def cpu_baseline(w, seconds=12.0):
    """The oracle (NumPy/fp64, as it stands) on a bounded sample of the same
    workload: one (sequence, kv head) unit of a bf16 anchor and one of an
    int4 anchor, each a full decode over the context (dequantise + softmax
    attention for the G heads).  Returns (GB/s, sample text, cores)."""
    import numpy as np
    import torch
    from oracle import attention as oatt
    from oracle import quant as oq
    from paper_2609_37988_gb300 import workloads as W

    T, D, G = w.context, w.head_dim, w.n_q_heads // w.n_kv_heads
    kinds = {}
    for a in w.anchors:
        kinds.setdefault(w.layers[a]["bits"], a)
    units = []
    w1 = dataclasses.replace(w, batch=1)  # one sequence's inputs: the sample needs one unit
    for bits, a in sorted(kinds.items()):
        k, v = W.kv_inputs(w1, a, 0, T, device="cpu")
        kk = k[0, :, 0].float().numpy()
        vv = v[0, :, 0].float().numpy()
        q = W.queries(w1, a)[0, :G].float().numpy()
        if bits == 16:
            units.append((bits, q, kk, vv, None))
        elif w.layers[a].get("scheme") == "symmetric":
            units.append((bits, q, oq.quantise_symmetric(kk, bits), oq.quantise_symmetric(vv, bits), 0))
        else:
            g = w.layers[a]["group"]
            units.append((bits, q, oq.quantise_per_token(kk, bits, g), oq.quantise_per_token(vv, bits, g), g))
    nbytes = 0
    n = 0
    t0 = time.perf_counter()
    while True:
        for bits, q, kq, vq, g in units:
            if bits == 16:
                kh, vh = kq, vq
                nbytes += T * 4 * D
            elif g == 0:  # symmetric: codes + one bf16 scale per row
                kh = oq.dequantise_symmetric(*kq)
                vh = oq.dequantise_symmetric(*vq)
                nbytes += T * (2 * D * bits // 8 + 4)
            else:
                kh = oq.dequantise_per_token(*kq, g)
                vh = oq.dequantise_per_token(*vq, g)
                nbytes += T * (2 * D * bits // 8 + 16 * D // g)
            oatt.gqa_decode(q[None], kh[None, None], vh[None, None], [T], w.sigma)
        n += 1
        if time.perf_counter() - t0 >= seconds:
            break
    dt = time.perf_counter() - t0
    cores = len(os.sched_getaffinity(0))
    sample = (f"{n} passes over one (sequence, kv head) unit of each anchor format "
              f"({', '.join(str(b) + '-bit' for b, *_ in units)}), {T} positions, G={G} heads")
    return nbytes / dt / 1e9, sample, cores


def cpu_baseline_mla(w, seconds=12.0):
    """The oracle's unabsorbed MLA decode (as it stands) on one sequence of
    the widest and of the narrowest latent layer of the workload (inputs
    drawn for a batch of one).  Bytes counted as on the GPU: the sequence's
    latent cache [c[:d] | k^R] in bf16.  Returns (GB/s, sample text, cores)."""
    from oracle import attention as oatt
    from paper_2609_37988_gb300 import workloads as W

    w1 = W.config(4, batch=1, mla_bits=w.layers[0]["bits"] if w.layers[0]["bits"] != 16 else None,
                  mla_scheme=w.layers[0].get("scheme", "symmetric"))
    T = w1.context
    widths = {}
    for l, a in enumerate(w1.layers):
        widths.setdefault(a["width"], l)
    units = []
    for d in sorted({max(widths), min(widths)}):
        l = widths[d]
        cl, kr = W.mla_inputs(w1, l, 0, T)
        wk, wv = W.mla_weights(w1, l)
        qn, qp = W.mla_queries(w1, l)
        cl, kr = cl.float().numpy(), kr.float().numpy()
        if w1.layers[l]["bits"] != 16:  # the oracle's stored state (outside the timed loop)
            from oracle import cache as ocache
            st = ocache.mla_anchor_state(cl, kr, [T], d, w1.layers[l]["bits"], w1.layers[l]["scheme"])
            cl, kr = st["c_hat"], st["kr_hat"]
        units.append((l, d, qn.float().numpy(), qp.float().numpy(), cl, kr, wk.float().numpy(),
                      wv.float().numpy()))
    nbytes, n = 0, 0
    t0 = time.perf_counter()
    while True:
        for l, d, qn, qp, cl, kr, wk, wv in units:
            oatt.mla_decode_unabsorbed(qn, qp, cl, kr, wk, wv, d, [T], w1.sigma)
            nbytes += T * mla_position_bytes(w1, l)
        n += 1
        if time.perf_counter() - t0 >= seconds:
            break
    dt = time.perf_counter() - t0
    cores = len(os.sched_getaffinity(0))
    sample = (f"{n} passes over one sequence of a d={max(widths)} and a d={min(widths)} latent "
              f"layer, {T} positions, {w1.n_q_heads} heads (unabsorbed oracle)")
    return nbytes / dt / 1e9, sample, cores


def run_reference(args):
    """--impl reference: the oracle as it stands, on the host cores."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    from paper_2609_37988_gb300 import workloads as W
    w = W.config(args.config, sym_bits=args.sym_bits, mla_bits=args.mla_bits,
                 mla_scheme=args.mla_scheme)
    base = cpu_baseline if w.kind == "gqa" else cpu_baseline_mla
    per = max(2.0, 60.0 / max(1, args.steps + args.warmup))
    for _ in range(args.warmup):
        base(w, seconds=min(per, 3.0))
    vals = []
    for _ in range(args.steps):
        g, sample, cores = base(w, seconds=per)
        vals.append(g)
    v = statistics.median(vals)
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": v, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": w.name},
        "cpu_baseline": {"value": v, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": sample},
        "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }))


# ---------------------------------------------------------------------------
def _layer_kind(w, l, src):
    if w.kind == "mla":
        a = w.layers[l]
        q = "" if a["bits"] == 16 else f"_{'sym' if a.get('scheme') == 'symmetric' else 'int'}{a['bits']}"
        return f"mla_d{a['width']}{q}"
    a = w.layers[src[l]]
    if a["bits"] == 16:
        return "bf16"
    return f"{'sym' if a.get('scheme') == 'symmetric' else 'int'}{a['bits']}"


def kernel_durations(w, cache, stream, new_kv, qs, outs, splits, per_layer, src, layer_call, dev,
                     splitk_reduce, reps=5):
    """Per-layer decode-kernel durations (ms) grouped by kind, with the
    algorithmic bytes of each layer: ``{kind: [(ms, bytes), ...]}``; for
    GQA steps also the appends and the split-K merges in ``aux`` (same
    form, kinds "append" and "merge").  Returns (kt, aux, how)."""
    import torch
    L = w.n_layers
    aux = {}
    parts = {}
    if w.kind == "gqa":
        for l in range(L):
            if splits[l] > 1:
                parts[l] = torch.empty((splits[l], w.batch * w.n_q_heads, w.head_dim + 2),
                                       device=dev)

    def run_layer(l):
        if w.kind == "mla":
            layer_call(l)  # the whole MLA call (4 launches)
        elif splits[l] > 1:
            # the automatic schedule, as the step's decode (splits or runs;
            # splits[l] partial slots either way)
            cache.decode_partial(l, qs[l], w.sigma, 0, partials=parts[l])
        else:
            cache.decode(l, qs[l], w.sigma, out=outs[l], n_splits=1)

    def merge(l):
        if w.kind == "gqa" and splits[l] > 1:
            splitk_reduce(parts[l], out=outs[l].view(-1, w.head_dim))

    def append_bytes(l):
        # the new rows read (bf16 keys and values) and one record written per
        # (sequence, new position, kv head)
        k, v = new_kv[l]
        rows = k.shape[0] * k.shape[1] * k.shape[2]
        return k.numel() * k.element_size() + v.numel() * v.element_size() + rows * _record_bytes(w, l)

    def merge_bytes(l):
        rows = w.batch * w.n_q_heads
        return splits[l] * rows * (w.head_dim + 2) * 4 + rows * w.head_dim * 4

    kt = {}
    try:
        def ev():
            return (torch.cuda.Event(enable_timing=True, external=True),
                    torch.cuda.Event(enable_timing=True, external=True))
        evs = [ev() for _ in range(L)]
        aev = {l: ev() for l in new_kv}
        mev = {l: ev() for l in range(L) if w.kind == "gqa" and splits[l] > 1}

        def tstep():
            for l in range(L):
                if l in new_kv:
                    aev[l][0].record(stream)
                    cache.append(l, *new_kv[l])
                    aev[l][1].record(stream)
                evs[l][0].record(stream)
                run_layer(l)
                evs[l][1].record(stream)
                if l in mev:
                    mev[l][0].record(stream)
                merge(l)
                if l in mev:
                    mev[l][1].record(stream)
            if w.append_per_step:
                cache.rewind(1)

        with torch.cuda.stream(stream):
            tstep()
            stream.synchronize()
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                tstep()
            for r in range(reps + 1):
                g.replay()
                stream.synchronize()
                if r == 0:
                    continue
                for l in range(L):
                    kt.setdefault(_layer_kind(w, l, src), []).append(
                        (evs[l][0].elapsed_time(evs[l][1]), per_layer[l]))
                for l, (e0, e1) in aev.items():
                    aux.setdefault("append", []).append((e0.elapsed_time(e1), append_bytes(l)))
                for l, (e0, e1) in mev.items():
                    aux.setdefault("merge", []).append((e0.elapsed_time(e1), merge_bytes(l)))
        del g
        return kt, aux, "event nodes in a graph replay of the step"
    except (TypeError, RuntimeError):
        torch.cuda.synchronize()
        kt, aux = {}, {}
    with torch.cuda.stream(stream):
        for l in range(L):
            if l in new_kv:
                cache.append(l, *new_kv[l])
            for _ in range(reps):
                s0, s1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                s0.record(stream)
                run_layer(l)
                s1.record(stream)
                s1.synchronize()
                kt.setdefault(_layer_kind(w, l, src), []).append((s0.elapsed_time(s1), per_layer[l]))
            merge(l)
        if w.append_per_step:
            cache.rewind(1)
        torch.cuda.synchronize()
    return kt, aux, "eager launches between events (includes host launch gaps)"



def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--config", type=int, default=3)
    ap.add_argument("--impl", default="kvk")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--e2e-steps", type=int, default=10)
    ap.add_argument("--mla-bits", type=int, choices=[8, 4, 2], default=None,
                    help="MLA workload (--config 4): store every latent layer quantised at this "
                         "bit-width (the kept latent and k^R one vector each)")
    ap.add_argument("--mla-scheme", choices=["symmetric", "grouped"], default="symmetric")
    ap.add_argument("--sym-bits", type=int, choices=[8, 4, 2], default=None,
                    help="store the quantised anchors with the symmetric per-vector "
                         "quantiser at this bit-width")
    ap.add_argument("--schedule", choices=["auto", "splits", "runs"], default="auto",
                    help="partition of the GQA decodes over CTAs (kvk_set_decode_schedule)")
    ap.add_argument("--run-ctas", type=int, default=0,
                    help="CTAs of a run-schedule decode (0: whole waves of resident CTAs)")
    ap.add_argument("--run-setup", type=int, default=-1,
                    help="planned tiles charged to each unit's start in a run decode (-1: default)")
    ap.add_argument("--profile-case",
                    choices=["gqa", "kpc", "mla", "mla64", "gather", "sym", "evict", "evict-small",
                             "prefill", "prefill-small", "append", "mlaq", "mlaq64"],
                    default=None,
                    help="small ncu case: decode (or eviction) launches only, no timing line")
    ap.add_argument("--prefill", action="store_true",
                    help="time causal chunk attention (pre-fill) over one compressed 14B anchor "
                         "instead of the decode step (one JSON line of its own)")
    ap.add_argument("--prefill-mla", action="store_true",
                    help="time MLA pre-fill (a 1024-query chunk over B=4 x 4096 positions) at every "
                         "kept width instead of the decode step (one JSON line of its own)")
    ap.add_argument("--append", action="store_true",
                    help="time bulk appends (quantise on write) at the 14B shape instead of the "
                         "decode step (one JSON line of its own)")
    ap.add_argument("--evict", action="store_true",
                    help="time the window-vote evictor at the long-context 14B shape instead "
                         "of the decode step (one JSON line of its own)")
    args = ap.parse_args()
    if args.impl == "reference":
        run_reference(args)
        return
    if args.profile_case:
        profile_case(args.profile_case)
        return
    if args.evict:
        evict_bench(args)
        return
    if args.prefill:
        prefill_bench(args)
        return
    if args.append:
        append_bench(args)
        return
    if args.prefill_mla:
        prefill_mla_bench(args)
        return

    import torch
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)

    from __graft_entry__ import build
    build()
    from paper_2609_37988_gb300 import workloads as W
    from paper_2609_37988_gb300.cache import Cache, Layer

    w = W.config(args.config, sym_bits=args.sym_bits, mla_bits=args.mla_bits,
                 mla_scheme=args.mla_scheme)
    T = w.context
    src = w.sources()
    new_kv = {}
    if w.kind == "mla":
        cache = Cache(kind="mla", n_layers=w.n_layers, n_q_heads=w.n_q_heads, head_dim=w.head_dim,
                      latent_dim=w.latent_dim, rope_dim=w.rope_dim, max_batch=w.batch, max_ctx=T,
                      layers=[Layer(**a) for a in w.layers], max_splits=64, device=dev)
        for l in range(w.n_layers):
            cl, kr = W.mla_inputs(w, l, 0, T, device=dev)
            cache.append(l, cl, kr)
            del cl, kr
        mq = [W.mla_queries(w, l, device=dev) for l in range(w.n_layers)]
        mw = [W.mla_weights(w, l, device=dev) for l in range(w.n_layers)]
        qs = [torch.cat([a.flatten(), b.flatten()]) for a, b in mq]  # host copies for e2e
        outs = [torch.empty((w.batch, w.n_q_heads, w.head_dim), dtype=torch.float32, device=dev)
                for _ in range(w.n_layers)]

        def layer_call(l, q_nope=None, q_pe=None):
            qn, qp = (mq[l] if q_nope is None else (q_nope, q_pe))
            cache.decode_mla(l, qn, qp, mw[l][0], mw[l][1], w.sigma, out=outs[l])

        def step():
            for l in range(w.n_layers):
                layer_call(l)
    else:
        pre = T - 1 if w.append_per_step else T
        cache = Cache(n_layers=w.n_layers, n_q_heads=w.n_q_heads, n_kv_heads=w.n_kv_heads,
                      head_dim=w.head_dim, max_batch=w.batch, max_ctx=T,
                      layers=[Layer(**a) for a in w.layers], max_splits=64, device=dev)
        cache.set_decode_schedule({"auto": 0, "splits": 1, "runs": 2}[args.schedule], args.run_ctas,
                                  args.run_setup)
        for a in w.anchors:
            k, v = W.kv_inputs(w, a, 0, pre, device=dev)
            cache.append(a, k, v)
            del k, v
        if w.keep:
            import numpy as np
            for a in w.anchors:
                idx, n = W.kept_positions(w, a, np.full(w.batch, T), device=dev)
                cache.set_kept(a, idx, n)
        qs = [W.queries(w, l, device=dev) for l in range(w.n_layers)]
        outs = [torch.empty((w.batch, w.n_q_heads, w.head_dim), dtype=torch.float32, device=dev)
                for _ in range(w.n_layers)]
        if w.append_per_step:
            for a in w.anchors:
                new_kv[a] = W.kv_inputs(w, a, pre, T, device=dev)

        def step():
            for l in range(w.n_layers):
                if l in new_kv:
                    cache.append(l, *new_kv[l])
                cache.decode(l, qs[l], w.sigma, out=outs[l])
            if w.append_per_step:
                cache.rewind(1)
    torch.cuda.synchronize()

    stream = torch.cuda.Stream(device=dev)
    with torch.cuda.stream(stream):
        step()  # eager: sets kernel attributes, occupancy queries
        stream.synchronize()
        splits = [cache.plan_splits(l) if w.kind == "gqa" else 1 for l in range(w.n_layers)]
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=stream):
            step()
    torch.cuda.synchronize()
    if w.kind == "mla":
        launches = 4 * w.n_layers  # absorb, latent decode, merge, up-projection
        step_bytes, per_layer = algorithmic_bytes_mla(w, T)
    else:
        launches = sum(1 + (splits[l] > 1) for l in range(w.n_layers))
        launches += len(new_kv) + (1 if w.append_per_step else 0)
        step_bytes, per_layer = algorithmic_bytes(w, T)

    def barrier():
        if dist:
            dist.barrier()

    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            graph.replay()
        stream.synchronize()
        barrier()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with Clocks(local) as clk:
            torch.cuda.synchronize()
            clk.mark("start")
            e0.record(stream)
            for _ in range(args.steps):
                graph.replay()
            e1.record(stream)
            e1.synchronize()
            torch.cuda.synchronize()
            clk.mark("end")
        barrier()
    ms = reduce_max(e0.elapsed_time(e1), dist, dev)
    ms_step = ms / args.steps
    value = job_throughput(step_bytes, args.steps, world, ms / 1e3)

    # ---- per-kernel durations (events on the launching stream) -------------
    # A replay of the same step, built from kvk_decode_partial + the split-K
    # merge so that a pair of timing-event nodes brackets each layer's decode
    # kernel inside the graph (no host launch gaps in the interval).  Falls
    # back to eager launches bracketed by events where graph event nodes are
    # not available.
    from paper_2609_37988_gb300.cache import splitk_reduce
    kt, aux, kernel_timing = kernel_durations(w, cache, stream, new_kv, qs, outs, splits, per_layer,
                                         src, layer_call if w.kind == "mla" else None, dev,
                                         splitk_reduce)
    hbm, peak_kind = peaks()
    totals = {k: sum(t for t, _ in v) for k, v in kt.items()}
    dom = max(totals, key=totals.get)
    durs = [t for t, _ in kt[dom]]
    bts = [b for _, b in kt[dom]]
    avg_ms = sum(durs) / len(durs)
    achieved = (sum(bts) / len(bts)) / (avg_ms / 1e3) / 1e9
    def summary(v):
        d = sum(t for t, _ in v) / len(v)
        b = sum(x for _, x in v) / len(v)
        return {"avg_us": round(d * 1e3, 2), "bytes": int(b), "gbs": round(b / (d / 1e3) / 1e9, 1),
                "frac": round(b / (d / 1e3) / 1e9 / hbm, 4)}
    kernels = {k: summary(v) for k, v in kt.items()}
    # the step's other kernels: a decode-step append (one new row per
    # sequence and kv head) and a split-K merge move a few hundred KB to a
    # few MB each, so their time is launch and memory latency, not bandwidth
    other_kernels = {k: summary(v) for k, v in aux.items()}
    # DRAM bytes per launch of the dominant kernel from the committed ncu
    # summary, used only while the decode sources still hash to the value
    # recorded with it (null otherwise: the counters would be stale)
    traffic = None
    tf = os.path.join(ROOT, "profiles", "gqa_decode_traffic.json")
    if os.path.exists(tf):
        with open(tf) as f:
            tj = json.load(f)
        ent = tj.get("kernels", {}).get(dom)
        if ent and tj.get("source_hash") == _source_hash() and ent.get("workload") == w.name:
            traffic = ent.get("bytes_per_launch")

    # ---- end to end through the public API, host buffers --------------------
    # The step's host copies run on a copy stream beside the layers, as a
    # serving loop would issue them: the first layer's inputs, then the rest
    # of the step's inputs, while the first layer runs; each group of
    # OUT_CHUNK layers' outputs leave as soon as that group is done.  Every
    # copy is inside the timed region; events order each layer after its
    # inputs and each output copy after its layers.
    OUT_CHUNK = 8
    copy_stream = torch.cuda.Stream(device=dev)
    n_out_chunks = (w.n_layers + OUT_CHUNK - 1) // OUT_CHUNK
    ev_in = [torch.cuda.Event() for _ in range(2)]
    ev_out = [torch.cuda.Event() for _ in range(n_out_chunks)]

    def copies_in(first, rest):
        # first(), rest(): the copies of layer 0's inputs and of the others'
        copy_stream.wait_stream(stream)
        with torch.cuda.stream(copy_stream):
            first()
            ev_in[0].record(copy_stream)
            rest()
            ev_in[1].record(copy_stream)
        stream.wait_event(ev_in[0])

    def copy_out(l, h_all, d_all):
        # after layer l: the outputs of its group, when it is the group's last
        if (l + 1) % OUT_CHUNK and l != w.n_layers - 1:
            return
        c = l // OUT_CHUNK
        ev_out[c].record(stream)
        copy_stream.wait_event(ev_out[c])
        with torch.cuda.stream(copy_stream):
            lo = c * OUT_CHUNK
            h_all[lo:l + 1].copy_(d_all[lo:l + 1], non_blocking=True)

    e2e = None
    if args.e2e_steps > 0:
        # one pinned host buffer and one device buffer per kind of tensor
        e_out_all = torch.empty((w.n_layers,) + tuple(outs[0].shape), dtype=outs[0].dtype, device=dev)
        e_outs = list(e_out_all.unbind(0))
        h_out_all = torch.empty(e_out_all.shape, dtype=e_out_all.dtype).pin_memory()
        d2h = h_out_all.numel() * h_out_all.element_size()
        if w.kind == "mla":
            # the step's inputs are every layer's q_nope and q_pe; the
            # up-projection weights are model parameters, resident
            h_qn = torch.stack([a for a, _ in mq]).cpu().pin_memory()
            h_qp = torch.stack([b for _, b in mq]).cpu().pin_memory()
            d_qn = torch.empty_like(h_qn, device=dev)
            d_qp = torch.empty_like(h_qp, device=dev)
            h2d = h_qn.numel() * h_qn.element_size() + h_qp.numel() * h_qp.element_size()

            def e2e_body():
                def first():
                    d_qn[:1].copy_(h_qn[:1], non_blocking=True)
                    d_qp[:1].copy_(h_qp[:1], non_blocking=True)

                def rest():
                    d_qn[1:].copy_(h_qn[1:], non_blocking=True)
                    d_qp[1:].copy_(h_qp[1:], non_blocking=True)
                copies_in(first, rest)
                for l in range(w.n_layers):
                    if l == 1:
                        stream.wait_event(ev_in[1])
                    cache.decode_mla(l, d_qn[l], d_qp[l], mw[l][0], mw[l][1], w.sigma, out=e_outs[l])
                    copy_out(l, h_out_all, e_out_all)
                stream.wait_stream(copy_stream)
    if args.e2e_steps > 0 and w.kind == "gqa":
        h_q_all = torch.stack([q.cpu() for q in qs]).pin_memory()
        d_q_all = torch.empty_like(h_q_all, device=dev)
        d_q = list(d_q_all.unbind(0))
        kv_layers = sorted(new_kv)
        h_kv_all = (torch.stack([t for a in kv_layers for t in new_kv[a]]).cpu().pin_memory()
                    if kv_layers else None)
        d_kv_all = torch.empty_like(h_kv_all, device=dev) if kv_layers else None
        d_kv = {a: (d_kv_all[2 * i], d_kv_all[2 * i + 1]) for i, a in enumerate(kv_layers)}
        h2d = h_q_all.numel() * h_q_all.element_size() + \
            (h_kv_all.numel() * h_kv_all.element_size() if kv_layers else 0)

        # layer 0's K/V, when it appends, are the first pair of the stack
        n_kv0 = 2 if kv_layers and kv_layers[0] == 0 else 0

        def e2e_body():
            def first():
                d_q_all[:1].copy_(h_q_all[:1], non_blocking=True)
                if n_kv0:
                    d_kv_all[:n_kv0].copy_(h_kv_all[:n_kv0], non_blocking=True)

            def rest():
                d_q_all[1:].copy_(h_q_all[1:], non_blocking=True)
                if kv_layers:
                    d_kv_all[n_kv0:].copy_(h_kv_all[n_kv0:], non_blocking=True)
            copies_in(first, rest)
            for l in range(w.n_layers):
                if l == 1:
                    stream.wait_event(ev_in[1])
                if l in d_kv:
                    cache.append(l, *d_kv[l])
                cache.decode(l, d_q[l], w.sigma, out=e_outs[l])
                copy_out(l, h_out_all, e_out_all)
            stream.wait_stream(copy_stream)
            if w.append_per_step:
                cache.rewind(1)
    if args.e2e_steps > 0:
        e2e_mode = "eager"
        with torch.cuda.stream(stream):
            def e2e_step():
                e2e_body()
                stream.synchronize()
            e2e_step()
            # the same API calls and pinned-host copies recorded once as a CUDA
            # graph: every replay copies the step's inputs in and its outputs out
            try:
                g_e2e = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g_e2e, stream=stream):
                    e2e_body()

                def e2e_step():
                    g_e2e.replay()
                    stream.synchronize()
                e2e_step()
                e2e_mode = ("cuda graph of the API calls and host copies (copies on a second "
                            "stream beside the layers)")
            except Exception:  # capture unsupported: stay eager
                torch.cuda.synchronize()
            barrier()
            t0 = time.perf_counter()
            for _ in range(args.e2e_steps):
                e2e_step()
            dt = time.perf_counter() - t0
        dt = reduce_max(dt, dist, dev)
        e2e = {"value": job_throughput(step_bytes, args.e2e_steps, world, dt), "unit": UNIT,
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "launch": e2e_mode,
               "ms_per_step": dt / args.e2e_steps * 1e3}

    err = cache.device_error()
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        g, sample, cores = cpu_baseline(w) if w.kind == "gqa" else cpu_baseline_mla(w)
        cpu = {"value": g, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": sample}
    clocks = clk.summary()
    if rank == 0:
        rec = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_step, "us_per_step": ms_step * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": ("/".join(sorted({_layer_kind(w, l, src) for l in range(w.n_layers)}))
                      if w.kind == "mla" else
                      "/".join(sorted({_layer_kind(w, a, src) for a in w.anchors}))),
            "data": "synthetic",
            "config": {"workload": w.name, "layers": w.n_layers, "batch": w.batch, "context": T,
                       "q_heads": w.n_q_heads, "kv_heads": w.n_kv_heads, "head_dim": w.head_dim,
                       "anchors": {k: sum(1 for a in w.anchors if _layer_kind(w, a, src) == k)
                                   for k in sorted({_layer_kind(w, a, src) for a in w.anchors})},
                       "inheritors": w.n_layers - len(w.anchors),
                       "bytes_per_step": step_bytes, "cuda_graph": True,
                       "l2": (f"no flush; smallest per-layer read {min(per_layer) / 1e6:.0f} MB vs 126 MB L2"
                              + (" (every layer's read exceeds L2)" if min(per_layer) > 126e6 else
                                 " (some layers fit in L2; consecutive inheritors may hit it)")),
                       "parallelism": f"replicas x{world}",
                       "decode_schedule": (args.schedule if args.run_ctas == 0 else
                                           f"{args.schedule}, {args.run_ctas} run CTAs")},
            "fraction_of_peak": value / hbm, "peak_gbs": hbm, "peak_kind": peak_kind,
            "fraction_of_nominal_8tbs": value / 8000.0,
            "roofline": {"bound": "hbm", "kernel": (f"gqa_decode ({dom})" if w.kind == "gqa" else
                                                   f"mla decode call ({dom})"), "achieved": achieved,
                         "peak": hbm, "unit": "GB/s", "frac": achieved / hbm, "traffic": traffic,
                         "peak_source": f"MEASURED_PEAKS.json hbm_gbs ({peak_kind})"},
            "kernels": kernels,
            "other_kernels": other_kernels,
            "kernel_timing": kernel_timing,
            "cpu_baseline": cpu,
            "e2e": e2e,
            "gpu_launches": launches * args.steps,
            "clocks": clocks,
            "device_error": err,
        }
        print(json.dumps(rec))


EVICT_WINDOW = 32


def evict_flops(lens, n_win, G, H_kv, D, budget):
    """Algorithmic FLOPs of one eviction call: every window query row scores
    its causal range once (2 D per score); sequences within the budget do
    nothing."""
    total = 0
    for L in lens:
        if L <= budget:
            continue
        P = L - n_win
        total += H_kv * G * sum(P + w + 1 for w in range(n_win)) * 2 * D
    return total


def alu_peak_tflops(sm_count, sm_mhz):
    """FP32 FMA peak: 128 FP32 lanes per SM, 2 FLOP per FMA, at ``sm_mhz``."""
    return sm_count * 128 * 2 * sm_mhz * 1e6 / 1e12


def _evict_setup(B, T, dev):
    import torch
    from paper_2609_37988_gb300 import workloads as W
    from paper_2609_37988_gb300.cache import Cache, Layer
    w = W.config(5, n_layers=1, batch=B, context=T)
    c = Cache(n_layers=1, n_q_heads=w.n_q_heads, n_kv_heads=w.n_kv_heads, head_dim=w.head_dim,
              max_batch=w.batch, max_ctx=T,
              layers=[Layer(bits=4, group=32, evict_capacity=w.keep)], device=dev)
    for b0 in range(0, T, 16384):
        k, v = W.kv_inputs(w, 0, b0, min(T, b0 + 16384), device=dev)
        c.append(0, k.contiguous(), v.contiguous())
        del k, v
    q = W.window_queries(w, 0, EVICT_WINDOW, device=dev)
    torch.cuda.synchronize()
    return w, c, q


def evict_bench(args):
    """The window-vote evictor (Sec. 3.4) at the long-context 14B shape: one
    int4 g32 anchor, B=4, 8 KV / 40 q heads, d_h 128, 131072 cached
    positions, a 32-query window, budget T/8.  Each call scores the window
    against the whole cache, merges the softmax statistics, votes and selects;
    timed with CUDA events on the launching stream (inputs: the 0.8 GB cache
    and the 2.7 GB score buffer, both larger than L2)."""
    import torch
    from __graft_entry__ import build
    build()
    torch.cuda.set_device(0)
    dev = torch.device("cuda", 0)
    w, c, q = _evict_setup(4, 131072, dev)
    budget = w.keep
    for _ in range(max(3, args.warmup)):
        c.evict_window(0, q, w.sigma, budget)
    torch.cuda.synchronize()
    stream = torch.cuda.current_stream()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps)]
    with Clocks(0) as clk:
        torch.cuda.synchronize()
        clk.mark("start")
        for s, e in ev:
            s.record(stream)
            c.evict_window(0, q, w.sigma, budget)
            e.record(stream)
        torch.cuda.synchronize()
        clk.mark("end")
    ms = [s.elapsed_time(e) for s, e in ev]
    assert c.device_error() == 0
    clocks = clk.summary()
    lens = [w.context] * w.batch
    G = w.n_q_heads // w.n_kv_heads
    flops = evict_flops(lens, EVICT_WINDOW, G, w.n_kv_heads, w.head_dim, budget)
    mean_ms = statistics.mean(ms)
    achieved = flops / (mean_ms * 1e-3) / 1e12
    # head_dim 128 with at most 256 window rows per KV head scores on the
    # tensor cores (bf16 hi/lo operands); other shapes on the CUDA cores
    R = EVICT_WINDOW * G
    if w.head_dim == 128 and R <= 256:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            peak = float(json.load(f)["bf16_tflops"])
        roof = {"bound": "tensor", "peak_source": "measured bf16 dense (burst)"}
    else:
        sms = torch.cuda.get_device_properties(0).multi_processor_count
        max_mhz = (clocks or {}).get("sm_max_mhz") or 2070.0
        peak = alu_peak_tflops(sms, max_mhz)
        roof = {"bound": "alu", "peak_source": f"{sms} SMs x 128 FP32 lanes x 2 x {max_mhz:.0f} MHz"}
    roof.update({"achieved": round(achieved, 2), "peak": round(peak, 1), "unit": "TFLOP/s",
                 "frac": round(achieved / peak, 4), "traffic": None,
                 "work": "score contraction counted once (171.8 GFLOP)"})
    line = {"metric": "window-vote eviction: ms per call, TFLOP/s of the score contraction",
            "value": round(mean_ms, 4), "unit": "ms", "higher_is_better": False,
            "steps": args.steps, "warmup": max(3, args.warmup), "n_gpus": 1,
            "dtype": "bf16x2 (hi/lo) in, f32 accumulate", "data": "synthetic",
            "config": {"workload": "qwen2.5-14b-b4-t131072-int4g32 one anchor, window 32, "
                                   f"budget {budget}", "l2": "inputs larger than L2"},
            "roofline": roof,
            "ms_min": round(min(ms), 4), "ms_max": round(max(ms), 4),
            "gpu_launches": 4 * args.steps, "clocks": clocks}
    print(json.dumps(line))


PREFILL_CHUNK = 2048


def prefill_flops(lens, n_q, Hq, D):
    """Algorithmic FLOPs of one pre-fill call: every query scores and weights
    its causal range once (2 D for the score, 2 D for the value product)."""
    total = 0
    for L in lens:
        for i in range(n_q):
            p = L - n_q + i
            if p >= 0:
                total += (p + 1) * Hq * 4 * D
    return total


def _prefill_setup(B, T, n_q, dev, bits=4):
    import torch
    from paper_2609_37988_gb300 import workloads as W
    from paper_2609_37988_gb300.cache import Cache, Layer
    w = W.config(3, n_layers=1, batch=B, context=T)
    layer = Layer(bits=bits, group=32) if bits != 16 else Layer(bits=16)
    c = Cache(n_layers=1, n_q_heads=w.n_q_heads, n_kv_heads=w.n_kv_heads, head_dim=w.head_dim,
              max_batch=B, max_ctx=T, layers=[layer], device=dev)
    for b0 in range(0, T, 4096):
        k, v = W.kv_inputs(w, 0, b0, min(T, b0 + 4096), device=dev)
        c.append(0, k.contiguous(), v.contiguous())
        del k, v
    q = W.randn((B, n_q, w.n_q_heads, w.head_dim), w.seed, 0, 11, dtype=torch.bfloat16, device=dev)
    torch.cuda.synchronize()
    return w, c, q


def prefill_bench(args):
    """Pre-fill over one compressed anchor at the 14B shape: int4 g32, B=4
    sequences of 8192 positions, the last 2048 of which are the chunk (the
    last chunk of a chunked pre-fill: 6144 cached positions before it);
    40 q / 8 KV heads, head_dim 128, bf16 queries.  CUDA events on the
    launching stream, inputs (0.8 GB of cache) larger than L2."""
    import torch
    from __graft_entry__ import build
    build()
    torch.cuda.set_device(0)
    dev = torch.device("cuda", 0)
    B, T = 4, 8192
    w, c, q = _prefill_setup(B, T, PREFILL_CHUNK, dev)
    out = torch.empty(q.shape, dtype=torch.float32, device=dev)
    for _ in range(max(3, args.warmup)):
        c.prefill(0, q, w.sigma, out=out)
    torch.cuda.synchronize()
    stream = torch.cuda.current_stream()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps)]
    with Clocks(0) as clk:
        torch.cuda.synchronize()
        clk.mark("start")
        for s0, e0 in ev:
            s0.record(stream)
            c.prefill(0, q, w.sigma, out=out)
            e0.record(stream)
        torch.cuda.synchronize()
        clk.mark("end")
    ms = [s0.elapsed_time(e0) for s0, e0 in ev]
    assert c.device_error() == 0
    flops = prefill_flops([T] * B, PREFILL_CHUNK, w.n_q_heads, w.head_dim)
    mean_ms = statistics.mean(ms)
    achieved = flops / (mean_ms * 1e-3) / 1e12
    with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
        peak = float(json.load(f)["bf16_tflops"])
    line = {"metric": "pre-fill over a compressed anchor: ms per call, TFLOP/s of the attention",
            "value": round(mean_ms, 4), "unit": "ms", "higher_is_better": False,
            "steps": args.steps, "warmup": max(3, args.warmup), "n_gpus": 1,
            "dtype": "bf16x2 (hi/lo) in, f32 accumulate", "data": "synthetic",
            "config": {"workload": f"qwen2.5-14b-b{B}-t{T} int4g32 anchor, chunk {PREFILL_CHUNK}",
                       "l2": "inputs larger than L2"},
            "roofline": {"bound": "tensor", "achieved": round(achieved, 2), "peak": round(peak, 1),
                         "unit": "TFLOP/s", "frac": round(achieved / peak, 4), "traffic": None,
                         "peak_source": "measured bf16 dense (burst)",
                         "work": f"scores and value products counted once ({flops / 1e9:.1f} GFLOP)"},
            "ms_min": round(min(ms), 4), "ms_max": round(max(ms), 4),
            "gpu_launches": 2 * args.steps, "clocks": clk.summary()}
    print(json.dumps(line))


MLA_PREFILL_CHUNK = 1024


def prefill_mla_bench(args):
    """MLA pre-fill over one latent layer of the MLA workload (16 heads,
    latent 512 + k^R 64) at B=4 sequences of 4096 positions, the last 1024
    of which are the chunk, for every kept width (bf16 latents, or quantised
    with --mla-bits / --mla-scheme).  CUDA events on the launching stream.
    value = ms per call at width 512; the roofline counts the attention's
    score and value products once against the measured bf16 dense peak."""
    import torch
    from __graft_entry__ import build
    build()
    from paper_2609_37988_gb300 import workloads as W
    from paper_2609_37988_gb300.cache import Cache, Layer
    torch.cuda.set_device(0)
    dev = torch.device("cuda", 0)
    B, T, n_q = 4, 4096, MLA_PREFILL_CHUNK
    w = W.config(4, batch=B, mla_bits=args.mla_bits, mla_scheme=args.mla_scheme)
    with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
        peak = float(json.load(f)["bf16_tflops"])
    res = {}
    with Clocks(0) as clk:
        for width in (512, 256, 128, 64):
            l = next(i for i, a in enumerate(w.layers) if a["width"] == width)
            a = dict(w.layers[l])
            c = Cache(kind="mla", n_layers=1, n_q_heads=w.n_q_heads, head_dim=w.head_dim,
                      latent_dim=w.latent_dim, rope_dim=w.rope_dim, max_batch=B, max_ctx=T,
                      layers=[Layer(**a)], device=dev)
            cl, kr = W.mla_inputs(w, l, 0, T, device=dev)
            c.append(0, cl, kr)
            del cl, kr
            wk, wv = W.mla_weights(w, l, device=dev)
            qn = W.randn((B, n_q, w.n_q_heads, w.head_dim), w.seed, l, 12, dtype=torch.bfloat16, device=dev)
            qp = W.randn((B, n_q, w.n_q_heads, w.rope_dim), w.seed, l, 13, dtype=torch.bfloat16, device=dev)
            out = torch.empty(qn.shape, dtype=torch.float32, device=dev)
            for _ in range(max(3, args.warmup)):
                c.prefill_mla(0, qn, qp, wk, wv, w.sigma, out=out)
            torch.cuda.synchronize()
            stream = torch.cuda.current_stream()
            ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                  for _ in range(args.steps)]
            if width == 512:
                clk.mark("start")
            for s0, e0 in ev:
                s0.record(stream)
                c.prefill_mla(0, qn, qp, wk, wv, w.sigma, out=out)
                e0.record(stream)
            torch.cuda.synchronize()
            if width == 512:
                clk.mark("end")
            assert c.device_error() == 0
            ms = statistics.mean(s0.elapsed_time(e0) for s0, e0 in ev)
            rows = sum(T - n_q + i + 1 for i in range(n_q)) * B * w.n_q_heads
            flops = rows * 2 * (2 * width + w.rope_dim)
            res[f"d{width}"] = {"ms": round(ms, 4), "tflops": round(flops / (ms * 1e-3) / 1e12, 2),
                                "frac": round(flops / (ms * 1e-3) / 1e12 / peak, 4)}
            del c
    m = res["d512"]
    q = "bf16" if args.mla_bits is None else f"{'sym' if args.mla_scheme == 'symmetric' else 'int'}{args.mla_bits}"
    line = {"metric": "MLA pre-fill over the latent cache: ms per call, TFLOP/s of the attention",
            "value": m["ms"], "unit": "ms", "higher_is_better": False, "steps": args.steps,
            "warmup": max(3, args.warmup), "n_gpus": 1, "dtype": f"{q} latents, f16/bf16 hi+lo products",
            "data": "synthetic",
            "config": {"workload": f"mla-h16-r512 {q}, B={B}, T={T}, chunk {n_q}",
                       "l2": "each sequence's latent cache fits in L2; the rows re-read it from there"},
            "roofline": {"bound": "tensor", "achieved": m["tflops"], "peak": round(peak, 1), "unit": "TFLOP/s",
                         "frac": m["frac"], "traffic": None, "peak_source": "measured bf16 dense (burst)",
                         "work": "score and value products of every row over its causal range, once"},
            "widths": res, "gpu_launches": 3 * args.steps, "clocks": clk.summary()}
    print(json.dumps(line))


APPEND_CHUNK = 2048


def append_bench(args):
    """Bulk append (quantise on write) at the 14B shape: B=32 sequences, a
    chunk of 2048 new positions each (a pre-fill chunk), 8 KV heads, head_dim
    128, bf16 keys and values (268 MB read per call, larger than L2), into
    one anchor of each format; the cache is reset between calls so every
    call writes positions 0..2047.  CUDA events around each append on the
    launching stream.  value = GB/s of the int4 g32 per-token append."""
    import torch
    from __graft_entry__ import build
    build()
    from paper_2609_37988_gb300 import workloads as W
    from paper_2609_37988_gb300.cache import Cache, Layer
    torch.cuda.set_device(0)
    dev = torch.device("cuda", 0)
    B, n, Hkv, D = 32, APPEND_CHUNK, 8, 128
    w = W.config(3)
    k, v = W.kv_inputs(w, 0, 0, n, device=dev)
    formats = {"int4 g32": dict(bits=4, group=32), "int8 g64": dict(bits=8, group=64),
               "bf16": dict(bits=16), "sym4": dict(bits=4, scheme="symmetric"),
               "sym8": dict(bits=8, scheme="symmetric"),
               "int4 g32 per-channel keys": dict(bits=4, group=32, key_axis="channel")}
    res = {}
    hbm, peak_kind = peaks()
    with Clocks(0) as clk:
        for name, cfg in formats.items():
            c = Cache(n_layers=1, n_q_heads=40, n_kv_heads=Hkv, head_dim=D, max_batch=B,
                      max_ctx=n, layers=[Layer(**cfg)], max_splits=8, device=dev)
            stored = B * n * Hkv * _rec_bytes(dataclasses.asdict(Layer(**cfg)), D)
            nbytes = k.numel() * k.element_size() + v.numel() * v.element_size() + stored
            stream = torch.cuda.current_stream()
            for _ in range(max(3, args.warmup)):
                c.reset()
                c.append(0, k, v)
            torch.cuda.synchronize()
            ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                  for _ in range(args.steps)]
            if name == "int4 g32":
                clk.mark("start")
            for s0, e0 in ev:
                c.reset()
                s0.record(stream)
                c.append(0, k, v)
                e0.record(stream)
            torch.cuda.synchronize()
            if name == "int4 g32":
                clk.mark("end")
            assert c.device_error() == 0
            ms = statistics.mean(s0.elapsed_time(e0) for s0, e0 in ev)
            res[name] = {"us": round(ms * 1e3, 2), "bytes": int(nbytes),
                         "gbs": round(nbytes / (ms * 1e-3) / 1e9, 1),
                         "frac": round(nbytes / (ms * 1e-3) / 1e9 / hbm, 4)}
            del c
    main_ = res["int4 g32"]
    line = {"metric": "bulk append with quantise on write: GB/s of algorithmic bytes",
            "value": main_["gbs"], "unit": "GB/s", "higher_is_better": True,
            "steps": args.steps, "warmup": max(3, args.warmup), "n_gpus": 1,
            "dtype": "bf16 in, int4 codes + f32 scale/zero out", "data": "synthetic",
            "config": {"workload": f"qwen2.5-14b kv, B={B}, {n} new positions per sequence, "
                                   f"{Hkv} kv heads, d_h {D}",
                       "l2": "inputs (268 MB) larger than L2"},
            "roofline": {"bound": "hbm", "kernel": "append (int4 g32, per token)",
                         "achieved": main_["gbs"], "peak": hbm, "unit": "GB/s",
                         "frac": main_["frac"], "traffic": None,
                         "peak_source": f"MEASURED_PEAKS.json hbm_gbs ({peak_kind})",
                         "work": "keys and values read once (bf16), records and metadata written once"},
            "formats": res, "gpu_launches": args.steps, "clocks": clk.summary()}
    print(json.dumps(line))


def profile_case(kind):
    """The kernel-level ncu case.  gqa: one int4 g32 and one bf16 anchor at
    the 14B step shape (B=32, 8 kv / 40 q heads, d_h 128, T=8192; 1.5 GB of
    cache, both anchors larger than L2); each decode runs 3 times in the order
    int4, bf16.  mla / mla64: one d=512 (302 MB) / d=64 (67 MB) latent layer
    at B=64, T=4096; mlaq / mlaq64: the same layer stored with the symmetric
    8-bit quantiser (152 / 35 MB).  append: bulk appends at the 14B shape.
    gather: one int4 g32 anchor at B=4, T=131072 with a kept list of T/8
    positions per sequence (805 MB cache, 101 MB read per decode), 3 decodes.
    sym: one symmetric anchor of each bit-width (8, 4, 2) at the 14B step
    shape (2.2 GB of cache), each decoded 3 times.  kpc: per-channel keys at
    the 7B step shape, one int4 g32 and one int8 g64 anchor (250 MB), 3
    decodes each."""
    import torch
    from __graft_entry__ import build
    build()
    from paper_2609_37988_gb300 import workloads as W
    from paper_2609_37988_gb300.cache import Cache, Layer
    torch.cuda.set_device(0)
    if kind == "gqa":
        w = W.config(3)
        layers = [Layer(bits=4, group=32), Layer(bits=16)]
        c = Cache(n_layers=2, n_q_heads=40, n_kv_heads=8, head_dim=128, max_batch=32,
                  max_ctx=8192, layers=layers)
        for l in range(2):
            k, v = W.kv_inputs(w, l, 0, 8192, device="cuda")
            c.append(l, k, v)
            del k, v
        q = W.queries(w, 0, device="cuda")
        for _ in range(3):
            for l in range(2):
                c.decode(l, q, w.sigma)
    elif kind == "append":
        # bulk append at the 14B shape: 32 sequences x 2048 new positions x
        # 8 kv heads into an int4 g32 anchor (268 MB of bf16 inputs), 3 calls
        w = W.config(3)
        c = Cache(n_layers=1, n_q_heads=40, n_kv_heads=8, head_dim=128, max_batch=32,
                  max_ctx=APPEND_CHUNK, layers=[Layer(bits=4, group=32)])
        k, v = W.kv_inputs(w, 0, 0, APPEND_CHUNK, device="cuda")
        for _ in range(3):
            c.reset()
            c.append(0, k, v)
    elif kind == "kpc":
        # per-channel keys at the 7B step shape: one int4 g32 and one int8
        # g64 anchor (B=16, 4 kv / 28 q heads, T=8192)
        w = W.config(2)
        layers = [Layer(bits=4, group=32, key_axis="channel"),
                  Layer(bits=8, group=64, key_axis="channel")]
        c = Cache(n_layers=2, n_q_heads=28, n_kv_heads=4, head_dim=128, max_batch=16,
                  max_ctx=8192, layers=layers)
        a0 = w.anchors[0]
        for l in range(2):
            k, v = W.kv_inputs(w, a0, 0, 8192, device="cuda")
            c.append(l, k, v)
            del k, v
        q = W.queries(w, 0, device="cuda")
        for _ in range(3):
            for l in range(2):
                c.decode(l, q, w.sigma)
    elif kind == "sym":
        # one anchor of each symmetric bit-width at the 14B step shape
        w = W.config(3)
        layers = [Layer(bits=b, scheme="symmetric") for b in (8, 4, 2)]
        c = Cache(n_layers=3, n_q_heads=40, n_kv_heads=8, head_dim=128, max_batch=32,
                  max_ctx=8192, layers=layers)
        for l in range(3):
            k, v = W.kv_inputs(w, l, 0, 8192, device="cuda")
            c.append(l, k, v)
            del k, v
        q = W.queries(w, 0, device="cuda")
        for _ in range(3):
            for l in range(3):
                c.decode(l, q, w.sigma)
    elif kind in ("evict", "evict-small"):
        # the evictor at the long-context 14B shape, or its one-sequence slice
        # (B=1: 168 MB of cache, a quarter of the items) for multi-pass captures
        B, T = (4, 131072) if kind == "evict" else (1, 131072)
        w, c, q = _evict_setup(B, T, torch.device("cuda", 0))
        for _ in range(3):
            c.evict_window(0, q, w.sigma, w.keep)
    elif kind in ("prefill", "prefill-small"):
        # pre-fill at the 14B shape (B=4, T=8192, chunk 2048), or one sequence
        # of 4096 positions with a 1024-query chunk for multi-pass captures
        B, T, n = (4, 8192, PREFILL_CHUNK) if kind == "prefill" else (1, 4096, 1024)
        w, c, q = _prefill_setup(B, T, n, torch.device("cuda", 0))
        for _ in range(3):
            c.prefill(0, q, w.sigma)
    elif kind == "gather":
        import numpy as np
        w = W.config(5, n_layers=1)
        T = w.context
        c = Cache(n_layers=1, n_q_heads=40, n_kv_heads=8, head_dim=128, max_batch=w.batch,
                  max_ctx=T, layers=[Layer(bits=4, group=32, evict_capacity=w.keep)])
        k, v = W.kv_inputs(w, 0, 0, T, device="cuda")
        c.append(0, k, v)
        del k, v
        idx, n = W.kept_positions(w, 0, np.full(w.batch, T), device="cuda")
        c.set_kept(0, idx, n)
        q = W.queries(w, 0, device="cuda")
        for _ in range(3):
            c.decode(0, q, w.sigma)
    else:
        # mla / mla64: one bf16 latent layer of width 512 / 64; mlaq / mlaq64:
        # the same stored with the symmetric 8-bit quantiser (B=64, T=4096)
        width = 64 if kind.endswith("64") else 512
        bits = 8 if kind.startswith("mlaq") else 16
        w = W.config(4, n_layers=1)
        w.layers[0]["width"] = width
        c = Cache(kind="mla", n_layers=1, n_q_heads=16, head_dim=128, latent_dim=512, rope_dim=64,
                  max_batch=w.batch, max_ctx=w.context,
                  layers=[Layer(bits=bits, width=width, scheme="symmetric")])
        cl, kr = W.mla_inputs(w, 0, 0, w.context, device="cuda")
        c.append(0, cl, kr)
        wk, wv = W.mla_weights(w, 0, device="cuda")
        qn, qp = W.mla_queries(w, 0, device="cuda")
        for _ in range(3):
            c.decode_mla(0, qn, qp, wk, wv, w.sigma)
    torch.cuda.synchronize()
    print(f"profile case {kind}: ok, device error {c.device_error()}")


def _source_hash():
    import hashlib
    h = hashlib.sha256()
    d = os.path.join(ROOT, "paper_2609_37988_gb300", "csrc")
    for n in sorted(os.listdir(d)):
        if n.startswith("decode_gqa") or n in ("layout.h", "common.cuh", "kernels.h"):
            with open(os.path.join(d, n), "rb") as f:
                h.update(f.read())
    return h.hexdigest()[:16]


if __name__ == "__main__":
    main()
