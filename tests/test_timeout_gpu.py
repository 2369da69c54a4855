"""The bounded-wait timeout path of the decode kernels, exercised without a
fault: kvk_set_wait_limit(0) makes every wait of a decode's tile loop give
up at its first poll.  The call must then set KVK_DEVERR_TIMEOUT (and
nothing else), let the copies it had in flight land and return; the context
stays usable, so with the default limit restored the next decode on the same
cache matches the fp64 oracle and leaves the error word clear.

Covered: the GQA decode's bulk-copy ring with early refill (per-token int8,
split grid and run schedule), its per-channel-key loop (bulk copies awaited at the top of each tile), and
the quantised MLA decode (every role of the warp-specialised kernel gives
up, the copy warp drains what it issued)."""
import math

import pytest
import torch

from _parity import assert_close, f32, gqa_expected, oracle_state
from oracle import attention as oatt
from oracle import cache as ocache

pytestmark = pytest.mark.gpu

TIMEOUT = 8  # KVK_DEVERR_TIMEOUT
B, HQ, HKV, D, T = 3, 8, 2, 128, 1000
LENS = [T, 513, 64]


@pytest.mark.parametrize("cfg", [dict(bits=8, group=64, key_axis="token"),
                                 dict(bits=4, group=32, key_axis="channel")],
                         ids=["int8-token", "int4-channel"])
def test_gqa_decode_gives_up_and_recovers(cfg):
    from paper_2609_37988_gb300.cache import Cache, Layer
    c = Cache(n_layers=1, n_q_heads=HQ, n_kv_heads=HKV, head_dim=D, max_batch=B, max_ctx=T,
              layers=[Layer(**cfg)], max_splits=16)
    g = torch.Generator().manual_seed(5)
    k = torch.randn((B, T, HKV, D), generator=g).to(torch.bfloat16)
    v = torch.randn((B, T, HKV, D), generator=g).to(torch.bfloat16)
    c.append(0, k.cuda(), v.cuda(), n_per_seq=torch.tensor(LENS, dtype=torch.int32, device="cuda"))
    st = oracle_state(f32(k), f32(v), LENS, cfg)
    q = torch.randn((B, HQ, D), generator=g).to(torch.bfloat16)
    scale = 1.0 / math.sqrt(D)
    assert c.device_error() == 0

    c.set_wait_limit(0)
    for ns in (1, 4):
        c.decode(0, q.cuda(), scale, n_splits=ns)
        assert c.device_error() == TIMEOUT, f"splits={ns}: the timeout was not reported"
    if cfg["key_axis"] == "token":
        # the run schedule: a CTA whose first segment gives up skips its second
        c.set_decode_schedule(c.SCHEDULE_RUNS, 5)
        c.decode(0, q.cuda(), scale)
        assert c.device_error() == TIMEOUT, "runs: the timeout was not reported"

    c.set_wait_limit(c.WAIT_LIMIT_DEFAULT)
    expected = gqa_expected(q, st, LENS, scale)
    for ns in (0, 1, 4):
        out = c.decode(0, q.cuda(), scale, n_splits=ns)
        assert_close(f32(out), expected, what=f"after timeout, splits={ns}")
    c.set_decode_schedule(c.SCHEDULE_AUTO)
    assert c.device_error() == 0


@pytest.mark.parametrize("fmt", [("symmetric", 4), ("grouped", 8)], ids=["sym4", "g8"])
def test_quantised_mla_decode_gives_up_and_recovers(fmt):
    from paper_2609_37988_gb300.cache import Cache, Layer
    Bm, H, width, Tm = 3, 16, 128, 700
    lens = [700, 300, 5]
    c = Cache(kind="mla", n_layers=1, n_q_heads=H, head_dim=128, latent_dim=512, rope_dim=64,
              max_batch=Bm, max_ctx=Tm, layers=[Layer(bits=fmt[1], scheme=fmt[0], width=width)],
              max_splits=16)
    g = torch.Generator().manual_seed(9)
    decay = torch.arange(512).add(1.0).rsqrt()
    cl = (torch.randn((Bm, Tm, 512), generator=g) * decay).to(torch.bfloat16)
    kr = torch.randn((Bm, Tm, 64), generator=g).to(torch.bfloat16)
    c.append(0, cl.cuda(), kr.cuda(), n_per_seq=torch.tensor(lens, dtype=torch.int32, device="cuda"))
    wk = (torch.randn((H, 128, 512), generator=g) / math.sqrt(512)).to(torch.bfloat16)
    wv = (torch.randn((H, 128, 512), generator=g) / math.sqrt(512)).to(torch.bfloat16)
    qn = torch.randn((Bm, H, 128), generator=g).to(torch.bfloat16)
    qp = torch.randn((Bm, H, 64), generator=g).to(torch.bfloat16)
    sigma = 1.0 / math.sqrt(192)
    args = (qn.cuda(), qp.cuda(), wk.cuda(), wv.cuda(), sigma)
    assert c.device_error() == 0

    c.set_wait_limit(0)
    for ns in (1, 3):
        c.decode_mla(0, *args, n_splits=ns)
        assert c.device_error() == TIMEOUT, f"splits={ns}: the timeout was not reported"

    c.set_wait_limit(c.WAIT_LIMIT_DEFAULT)
    st = ocache.mla_anchor_state(f32(cl), f32(kr), lens, width, fmt[1], fmt[0])
    ref = oatt.mla_decode_unabsorbed(f32(qn), f32(qp), st["c_hat"], st["kr_hat"], f32(wk), f32(wv),
                                     width, lens, sigma)
    for ns in (0, 3):
        out = c.decode_mla(0, *args, n_splits=ns)
        assert_close(f32(out), ref, what=f"mla after timeout, splits={ns}")
    assert c.device_error() == 0

