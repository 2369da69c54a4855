"""kvk_decode_attention_noalloc: the decode entry point for callers that
cannot provide scratch device memory.  Its split-K partials live in a fixed
buffer inside the library; these checks call it through the C ABI on two
calls in a row (the second call reuses a buffer still holding the first
call's partials) and compare each result with the fp64 oracle on the same
inputs and with kvk_decode_attention (split grid and run schedule), and
check that a request too large for the buffer is refused before anything
runs.

Kept in a file of its own, collected last."""
import ctypes
import math

import numpy as np
import pytest
import torch

from _parity import assert_close, f32, gqa_expected, oracle_state

pytestmark = pytest.mark.gpu

B, HQ, HKV, D, T = 3, 10, 2, 128, 1500
LENS = [T, T // 2, 77]
CFGS = [dict(bits=4, group=32, key_axis="token"), dict(bits=16, group=64, key_axis="token")]


def _noalloc(cache, layer, q, scale, out, n_splits):
    from paper_2609_37988_gb300 import _lib
    lib = _lib.load()
    code = _lib.DTYPE_F32 if q.dtype == torch.float32 else _lib.DTYPE_BF16
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    return lib.kvk_decode_attention_noalloc(cache.handle, layer, ctypes.c_void_p(q.data_ptr()), code,
                                            ctypes.c_float(scale), ctypes.c_void_p(out.data_ptr()),
                                            n_splits, stream)


def _cache_with_data(seed=0):
    from paper_2609_37988_gb300.cache import Cache, Layer
    c = Cache(n_layers=2, n_q_heads=HQ, n_kv_heads=HKV, head_dim=D, max_batch=B, max_ctx=T,
              layers=[Layer(bits=4, group=32), Layer(bits=16)], max_splits=64)
    g = torch.Generator().manual_seed(seed)
    states = []
    for l in range(2):
        k = torch.randn((B, T, HKV, D), generator=g).to(torch.bfloat16)
        v = torch.randn((B, T, HKV, D), generator=g).to(torch.bfloat16)
        c.append(l, k.cuda(), v.cuda(), n_per_seq=torch.tensor(LENS, dtype=torch.int32, device="cuda"))
        states.append(oracle_state(f32(k), f32(v), LENS, CFGS[l]))
    return c, states


def test_matches_oracle_and_decode_on_two_calls_in_a_row():
    c, states = _cache_with_data()
    scale = 1.0 / math.sqrt(D)
    g = torch.Generator().manual_seed(1)
    calls = [(0, torch.randn((B, HQ, D), generator=g).to(torch.bfloat16), 0),
             (1, torch.randn((B, HQ, D), generator=g).to(torch.float32), 5)]
    for layer, q, ns in calls:
        expected = gqa_expected(q, states[layer], LENS, scale)
        q = q.cuda()
        out = torch.full((B, HQ, D), float("nan"), device="cuda")
        assert _noalloc(c, layer, q, scale, out, ns) == 0
        torch.cuda.synchronize()
        assert_close(out.cpu().numpy(), expected, what=f"noalloc layer {layer} vs oracle")
        ref = c.decode(layer, q, scale, n_splits=ns)
        torch.cuda.synchronize()
        assert_close(out.cpu().numpy(), ref.cpu().numpy(), what=f"noalloc layer {layer} vs decode")
    assert c.device_error() == 0


def test_run_schedule():
    """With the run schedule the automatic call (n_splits = 0) writes the
    plan's partial slots into the fixed buffer and merges them: equal to the
    oracle and to kvk_decode_attention on the same schedule."""
    c, states = _cache_with_data(seed=3)
    c.set_decode_schedule(c.SCHEDULE_RUNS, 11)
    scale = 1.0 / math.sqrt(D)
    q = torch.randn((B, HQ, D), generator=torch.Generator().manual_seed(4)).to(torch.bfloat16)
    expected = gqa_expected(q, states[0], LENS, scale)
    q = q.cuda()
    out = torch.full((B, HQ, D), float("nan"), device="cuda")
    assert _noalloc(c, 0, q, scale, out, 0) == 0
    torch.cuda.synchronize()
    assert_close(out.cpu().numpy(), expected, what="noalloc runs vs oracle")
    ref = c.decode(0, q, scale)
    torch.cuda.synchronize()
    assert torch.equal(out, ref)
    assert c.device_error() == 0


def test_refuses_requests_larger_than_its_buffer():
    from paper_2609_37988_gb300 import _lib
    from paper_2609_37988_gb300.cache import Cache, Layer
    # 64 splits x 64 sequences x 64 heads x 130 floats = 34 M floats > 4 M
    c = Cache(n_layers=1, n_q_heads=64, n_kv_heads=8, head_dim=128, max_batch=64, max_ctx=8192,
              layers=[Layer(bits=4, group=32)], max_splits=64)
    x = torch.zeros((64, 8192, 8, 128), dtype=torch.bfloat16, device="cuda")
    c.append(0, x, x)
    del x
    q = torch.zeros((64, 64, 128), dtype=torch.bfloat16, device="cuda")
    out = torch.full((64, 64, 128), 7.0, device="cuda")
    st = _noalloc(c, 0, q, 0.1, out, 64)
    assert st == 4  # KVK_ERR_CAPACITY
    assert "fixed buffer" in _lib.load().kvk_last_error().decode()
    torch.cuda.synchronize()
    assert (out == 7.0).all()  # nothing ran
    # one split needs no partials at all
    assert _noalloc(c, 0, q, 0.1, out, 1) == 0
    torch.cuda.synchronize()
    assert torch.isfinite(out).all()
