"""GPU parity of the run schedule of the GQA decode (kvk_set_decode_schedule):
CTAs that each take an equal run of the flattened (sequence, KV head, tile)
grid, a run meeting at most two units, each unit's pieces merged from its
partial slots.  Against the fp64 oracle over the formats that have runs
(grouped int8/int4 with per-token keys, the symmetric 8/4/2-bit scheme),
ragged and empty sequences, CTA counts that align with the units, cross
their boundaries or give one tile per CTA; the partial slots a unit does not
use are empty; a recorded launch replayed after the sequences grew still
covers every position; and formats without runs fall back to the splits."""
import math

import numpy as np
import pytest
import torch

from _parity import assert_close, f32, gqa_expected, oracle_state

pytestmark = pytest.mark.gpu

RUNS = 2  # KVK_SCHEDULE_RUNS
SPLITS = 1

FORMATS = [
    dict(bits=4, group=32, key_axis="token"),
    dict(bits=8, group=64, key_axis="token"),
    dict(bits=8, group=32, key_axis="token"),
    dict(bits=4, group=64, key_axis="token"),
    dict(bits=8, group=64, key_axis="token", scheme="symmetric"),
    dict(bits=4, group=64, key_axis="token", scheme="symmetric"),
    dict(bits=2, group=64, key_axis="token", scheme="symmetric"),
]


def _fid(f):
    return f"{f.get('scheme', 'grouped')[:3]}{f['bits']}-g{f['group']}"


def _cache(B, Hq, Hkv, D, T, fmt, max_splits=32):
    from paper_2609_37988_gb300.cache import Cache, Layer
    return Cache(n_layers=2, n_q_heads=Hq, n_kv_heads=Hkv, head_dim=D, max_batch=B, max_ctx=T,
                 layers=[Layer(**fmt), Layer(inherit=True)], max_splits=max_splits)


def _fill(c, B, Hkv, D, lens, seed):
    g = torch.Generator().manual_seed(seed)
    T = max(lens)
    k = (torch.randn((B, T, Hkv, D), generator=g) * 1.5 + 0.3).to(torch.bfloat16)
    v = torch.randn((B, T, Hkv, D), generator=g).to(torch.bfloat16)
    c.append(0, k.cuda(), v.cuda(), n_per_seq=torch.tensor(lens, dtype=torch.int32, device="cuda"))
    return f32(k), f32(v)


def _tiles(fmt, D, len_hi):
    """Kernel tiles per unit the host plans from its length bound."""
    kt = 128 if ((fmt["bits"] == 4 and fmt.get("scheme") != "symmetric")
                 or (fmt.get("scheme") == "symmetric" and fmt["bits"] <= 4)) else 64
    return -(-(-(-len_hi // 64)) // (kt // 64))


@pytest.mark.parametrize("fmt", FORMATS, ids=_fid)
def test_runs_match_the_oracle(fmt):
    B, Hkv, G, D = 4, 2, 5, 128
    lens = [700, 0, 1, 385]
    c = _cache(B, G * Hkv, Hkv, D, 768, fmt)
    K, V, = _fill(c, B, Hkv, D, lens, seed=fmt["bits"] * 7 + fmt["group"])
    st = oracle_state(K, V, np.array(lens), fmt)
    sigma = 1.0 / math.sqrt(D)
    q = torch.randn((B, G * Hkv, D), generator=torch.Generator().manual_seed(1)).to(torch.bfloat16)
    ref = gqa_expected(q, st, np.array(lens), sigma)
    units = B * Hkv
    c.set_decode_schedule(SPLITS)
    split = f32(c.decode(0, q.cuda(), sigma, n_splits=0))
    # aligned with the units, crossing unit boundaries, one planned tile per
    # CTA; planned set-up tiles per unit (runs holding only set-up tiles
    # decode nothing)
    for ctas, setup in ((units, 0), (units + 1, 0), ((7 * units) // 3, 4), (10 ** 6, 0),
                        (10 ** 6, 3), (units + 3, 4)):
        c.set_decode_schedule(RUNS, ctas, setup)
        tpu = _tiles(fmt, D, max(lens)) + setup
        n = min(max(ctas, units), units * tpu)
        slots = max(((u + 1) * tpu * n - 1) // (units * tpu) - ((u * tpu + 1) * n - 1) // (units * tpu) + 1
                    for u in range(units))
        assert c.plan_splits(0) == slots
        for layer in (0, 1):  # the inheritor reads the same anchor
            out = f32(c.decode(layer, q.cuda(), sigma, n_splits=0))
            assert_close(out, ref, what=f"{_fid(fmt)} runs ctas={ctas} setup={setup}")
            assert_close(out, split, max_abs=1e-4, rel_l2=2e-5, what="runs vs splits")
            assert (out[1] == 0).all()  # the empty sequence
    assert c.device_error() == 0


@pytest.mark.parametrize("D,G", [(64, 8), (128, 1)])
def test_runs_other_shapes(D, G):
    fmt = dict(bits=4, group=32, key_axis="token")
    B, Hkv = 3, 3
    lens = [1000, 129, 640]
    c = _cache(B, G * Hkv, Hkv, D, 1024, fmt)
    K, V = _fill(c, B, Hkv, D, lens, seed=D + G)
    st = oracle_state(K, V, np.array(lens), fmt)
    q = torch.randn((B, G * Hkv, D), generator=torch.Generator().manual_seed(2)).to(torch.float32)
    ref = gqa_expected(q, st, np.array(lens), 0.1)
    for ctas in (B * Hkv + 2, 20):
        c.set_decode_schedule(RUNS, ctas)
        assert_close(f32(c.decode(0, q.cuda(), 0.1)), ref, what=f"D{D} G{G} ctas={ctas}")
    assert c.device_error() == 0


def test_run_partials_slots_and_merge():
    """Partial-only calls with n_splits = 0 write kvk_decode_plan_splits
    slots; the slots a unit's run pieces do not fill are empty (m = -inf,
    l = 0); merging the slots gives exactly the decode's output."""
    from paper_2609_37988_gb300.cache import splitk_reduce
    fmt = dict(bits=4, group=32, key_axis="token")
    B, Hkv, G, D = 3, 2, 4, 128
    lens = [1000, 300, 517]
    c = _cache(B, G * Hkv, Hkv, D, 1024, fmt)
    _fill(c, B, Hkv, D, lens, seed=11)
    q = torch.randn((B, G * Hkv, D)).to(torch.bfloat16).cuda()
    units, tpu = B * Hkv, _tiles(fmt, D, max(lens)) + 2
    n = 11
    c.set_decode_schedule(RUNS, n, 2)
    S = c.plan_splits(0)
    # every slot row is written: a buffer full of NaN merges like the workspace
    p = c.decode_partial(0, q, 0.1, 0,
                         partials=torch.full((S, B * G * Hkv, D + 2), float("nan"), device="cuda"))
    assert p.shape == (S, B * G * Hkv, D + 2)
    assert not torch.isnan(p).any()
    total = units * tpu
    for u in range(units):
        c0 = ((u * tpu + 1) * n - 1) // total
        c1 = ((u + 1) * tpu * n - 1) // total
        b, j = divmod(u, Hkv)
        rows = slice(b * G * Hkv + j * G, b * G * Hkv + (j + 1) * G)
        for k in range(c1 - c0 + 1, S):
            assert torch.isinf(p[k, rows, D]).all() and (p[k, rows, D + 1] == 0).all()
            assert (p[k, rows, :D] == 0).all()
    merged = splitk_reduce(p).view(B, G * Hkv, D)
    assert torch.equal(merged, c.decode(0, q, 0.1))
    assert c.device_error() == 0


def test_recorded_run_launch_covers_longer_sequences():
    """A decode recorded in a CUDA graph at one length bound and replayed
    after appends: the CTA holding each unit's last planned tile runs to the
    sequence's end, so every position is still read."""
    fmt = dict(bits=8, group=64, key_axis="token")
    B, Hkv, G, D = 2, 2, 4, 128
    c = _cache(B, G * Hkv, Hkv, D, 1024, fmt)
    g = torch.Generator().manual_seed(3)
    k = (torch.randn((B, 900, Hkv, D), generator=g)).to(torch.bfloat16)
    v = torch.randn((B, 900, Hkv, D), generator=g).to(torch.bfloat16)
    c.append(0, k[:, :600].contiguous().cuda(), v[:, :600].contiguous().cuda())
    c.set_decode_schedule(RUNS, 7)
    q = torch.randn((B, G * Hkv, D), generator=g).to(torch.bfloat16).cuda()
    out = torch.empty((B, G * Hkv, D), device="cuda")
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        c.decode(0, q, 0.1, out=out, stream=s)  # warm (kernel attributes set outside capture)
        s.synchronize()
        gr = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gr, stream=s):
            c.decode(0, q, 0.1, out=out, stream=s)
    torch.cuda.synchronize()
    c.append(0, k[:, 600:].contiguous().cuda(), v[:, 600:].contiguous().cuda())
    torch.cuda.synchronize()
    gr.replay()
    torch.cuda.synchronize()
    st = oracle_state(f32(k), f32(v), np.array([900, 900]), fmt)
    assert_close(f32(out), gqa_expected(q.cpu(), st, np.array([900, 900]), 0.1), what="replayed")
    assert c.device_error() == 0


def test_formats_without_runs_use_the_splits():
    """bf16 anchors, per-channel keys and kept lists have no run kernel:
    under the run schedule they decode with the splits, as before."""
    B, Hkv, G, D = 2, 2, 4, 128
    for fmt in (dict(bits=16, group=64, key_axis="token"), dict(bits=4, group=32, key_axis="channel")):
        c = _cache(B, G * Hkv, Hkv, D, 512, fmt)
        K, V = _fill(c, B, Hkv, D, [512, 200], seed=5)
        st = oracle_state(K, V, np.array([512, 200]), fmt)
        q = torch.randn((B, G * Hkv, D)).to(torch.bfloat16)
        c.set_decode_schedule(SPLITS)
        plain = c.decode(0, q.cuda(), 0.1).clone()
        ns = c.plan_splits(0)
        c.set_decode_schedule(RUNS, 5)
        assert c.plan_splits(0) == ns
        out = c.decode(0, q.cuda(), 0.1)
        assert torch.equal(out, plain)
        assert_close(f32(out), gqa_expected(q, st, np.array([512, 200]), 0.1), what=str(fmt))
    # a kept list on a run format: the gather kernel
    fmt = dict(bits=4, group=32, key_axis="token", evict_capacity=128)
    c = _cache(B, G * Hkv, Hkv, D, 512, fmt)
    K, V = _fill(c, B, Hkv, D, [512, 300], seed=6)
    idx = torch.arange(0, 256, 2, dtype=torch.int32).repeat(B, 1)
    c.set_kept(0, idx.cuda(), torch.tensor([128, 128], dtype=torch.int32).cuda())
    c.set_decode_schedule(RUNS, 5)
    st = oracle_state(K, V, np.array([512, 300]), dict(bits=4, group=32, key_axis="token"))
    q = torch.randn((B, G * Hkv, D)).to(torch.bfloat16)
    kept = [np.arange(0, 256, 2, dtype=np.int32)] * B
    assert_close(f32(c.decode(0, q.cuda(), 0.1)), gqa_expected(q, st, np.array([512, 300]), 0.1, kept),
                 what="gather under runs")
    assert c.device_error() == 0


def test_schedule_argument_checks():
    from paper_2609_37988_gb300.cache import KVKError
    c = _cache(1, 4, 1, 64, 128, dict(bits=4, group=32, key_axis="token"))
    with pytest.raises(KVKError, match="INVALID_ARG"):
        c.set_decode_schedule(3)
    with pytest.raises(KVKError, match="INVALID_ARG"):
        c.set_decode_schedule(RUNS, -1)
