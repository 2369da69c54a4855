"""C-ABI boundary checks that need no GPU: the library builds and loads,
exports every function include/kvk.h declares, and its host-side plan
validation and cost accounting agree with the oracle and the paper."""
import ctypes
import os
import re

import pytest

from paper_2609_37988_gb300 import build as kbuild

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    kbuild.build()
    from paper_2609_37988_gb300 import _lib
    return _lib


def _declared():
    txt = open(os.path.join(ROOT, "include", "kvk.h")).read()
    txt = re.sub(r"/\*.*?\*/", "", txt, flags=re.S)
    return sorted(set(re.findall(r"\b(kvk_[a-z_]+)\s*\(", txt)))


def test_every_declared_symbol_is_exported(lib):
    names = _declared()
    assert len(names) >= 20
    so = ctypes.CDLL(lib.LIB_PATH)
    for n in names:
        assert hasattr(so, n), n
    assert set(names) == set(lib.exported_symbols())
    assert lib.load().kvk_version().decode().endswith("sm_103a")


def _desc(lib, **kw):
    d = dict(kind=0, n_layers=4, n_q_heads=8, n_kv_heads=2, head_dim=128, latent_dim=0, rope_dim=0,
             max_batch=2, max_ctx=1000)
    d.update(kw)
    return lib.ModelDesc(**d)


def _plan(lib, *rows):
    arr = (lib.LayerCfg * len(rows))()
    for i, r in enumerate(rows):
        arr[i] = lib.LayerCfg(*r)
    return arr


def _plan_status(lib, desc, plan):
    sizes = (ctypes.c_size_t * desc.n_layers)()
    return lib.load().kvk_cache_plan(ctypes.byref(desc), plan, sizes), list(sizes)


# (inherit, bits, group, key_axis, value_axis, width, evict_capacity)
BF16 = (0, 16, 0, 0, 0, 0, 0)
INH = (1, 0, 0, 0, 0, 0, 0)


def test_plan_validation(lib):
    d = _desc(lib)
    ok, sizes = _plan_status(lib, d, _plan(lib, BF16, INH, (0, 4, 32, 0, 0, 0, 0), (0, 8, 64, 1, 0, 0, 0)))
    assert ok == 0 and sizes[1] == 0 and all(sizes[i] > 0 for i in (0, 2, 3))
    assert _plan_status(lib, d, _plan(lib, INH, BF16, BF16, BF16))[0] == 2      # layer 0 inherits
    assert _plan_status(lib, d, _plan(lib, BF16, (0, 2, 32, 0, 0, 0, 0), BF16, BF16))[0] == 5  # 2-bit
    assert _plan_status(lib, d, _plan(lib, BF16, (0, 3, 32, 0, 0, 0, 0), BF16, BF16))[0] == 2  # 3-bit
    assert _plan_status(lib, d, _plan(lib, BF16, (0, 4, 48, 0, 0, 0, 0), BF16, BF16))[0] == 2  # 48 !| 128
    assert _plan_status(lib, d, _plan(lib, BF16, (0, 4, 32, 0, 1, 0, 0), BF16, BF16))[0] == 5  # per-channel V
    assert _plan_status(lib, _desc(lib, head_dim=96), _plan(lib, BF16, BF16, BF16, BF16))[0] == 5
    assert _plan_status(lib, _desc(lib, n_q_heads=7), _plan(lib, BF16, BF16, BF16, BF16))[0] == 1
    m = _desc(lib, kind=1, n_layers=2, n_q_heads=16, head_dim=128, latent_dim=512, rope_dim=64)
    assert _plan_status(lib, m, _plan(lib, (0, 16, 0, 0, 0, 512, 0), (0, 16, 0, 0, 0, 64, 0)))[0] == 0
    assert _plan_status(lib, m, _plan(lib, (0, 16, 0, 0, 0, 512, 0), (0, 16, 0, 0, 0, 100, 0)))[0] == 2
    err = lib.load().kvk_last_error().decode()
    assert "width" in err


def test_arena_sizes_follow_record_bytes(lib):
    # per (position, kv head): bf16 512 B; int8 g64 288 B; int4 g32 192 B
    B, H, T = 3, 2, 640
    d = _desc(lib, n_layers=3, max_batch=B, max_ctx=T)
    ok, sizes = _plan_status(lib, d, _plan(lib, BF16, (0, 8, 64, 0, 0, 0, 0), (0, 4, 32, 0, 0, 0, 0)))
    assert ok == 0
    for s, rec in zip(sizes, (512, 288, 192)):
        assert B * H * T * rec <= s <= B * H * T * rec + 4096


def _plan_cost(lib, desc, plan):
    b, s, r = ctypes.c_double(), ctypes.c_double(), ctypes.c_double()
    st = lib.load().kvk_plan_cost(ctypes.byref(desc), plan, ctypes.byref(b), ctypes.byref(s), ctypes.byref(r))
    assert st == 0
    return b.value, s.value, r.value


def test_plan_cost_matches_oracle_and_paper(lib):
    from oracle import cost
    from paper_2609_37988_gb300 import workloads as W
    # the 14B-shaped mixed plan: 12 bf16 + 20 int4 + 16 inheritors
    w = W.config(3)
    d = _desc(lib, n_layers=48, n_q_heads=40, n_kv_heads=8, max_batch=1, max_ctx=64)
    rows = [INH if a["inherit"] else (0, a["bits"], a["group"], 0, 0, 0, 0) for a in w.layers]
    bits, stored, rho = _plan_cost(lib, d, _plan(lib, *rows))
    acts = ["inherit" if a["inherit"] else (None, a["bits"]) for a in w.layers]
    assert rho == pytest.approx(cost.compression(acts, 48, 8, 128, mla=False), rel=1e-12)
    assert rho == pytest.approx(768 / 272, rel=1e-12)     # 2.82x, the realised factor
    assert stored == 12 * 8 * 512 + 20 * 8 * 192
    # Tab. ranges end points on Qwen2.5-14B geometry
    allbf = _plan_cost(lib, d, _plan(lib, *([BF16] * 48)))[2]
    assert allbf == pytest.approx(1.0)
    one = _plan_cost(lib, d, _plan(lib, *([(0, 4, 32, 0, 0, 0, 0)] + [INH] * 47)))[2]
    assert one == pytest.approx(48 * 4.0)
    m = _desc(lib, kind=1, n_layers=48, n_q_heads=16, head_dim=128, latent_dim=1024, rope_dim=64,
              max_batch=1, max_ctx=64)
    # rank axis: full width 1.88x (MLA conversion), r/8 = 128 -> 10.7x (Tab. ranges)
    full = _plan_cost(lib, m, _plan(lib, *([(0, 16, 0, 0, 0, 1024, 0)] * 48)))[2]
    assert round(full, 2) == 1.88
    m5 = _desc(lib, kind=1, n_layers=48, n_q_heads=16, head_dim=128, latent_dim=512, rope_dim=64,
               max_batch=1, max_ctx=64)
    narrow = _plan_cost(lib, m5, _plan(lib, *([(0, 16, 0, 0, 0, 64, 0)] * 48)))
    assert narrow[0] == 48 * (64 + 64) * 16


# symmetric per-vector scheme: (inherit, bits, group, key_axis, value_axis,
# width, evict_capacity, scheme)
def _sym(bits, key_axis=0, value_axis=0, evict=0):
    return (0, bits, 0, key_axis, value_axis, 0, evict, 1)


def test_symmetric_plan_validation(lib):
    d = _desc(lib)
    ok, sizes = _plan_status(lib, d, _plan(lib, _sym(2), _sym(4), INH, _sym(8, evict=100)))
    assert ok == 0 and sizes[2] == 0
    # a per-channel axis contradicts one scale per token-head row
    assert _plan_status(lib, d, _plan(lib, _sym(4, key_axis=1), BF16, BF16, BF16))[0] == 2
    assert _plan_status(lib, d, _plan(lib, _sym(4, value_axis=1), BF16, BF16, BF16))[0] == 2
    # unknown scheme; 3 bits
    assert _plan_status(lib, d, _plan(lib, (0, 4, 32, 0, 0, 0, 0, 2), BF16, BF16, BF16))[0] == 2
    assert _plan_status(lib, d, _plan(lib, _sym(3), BF16, BF16, BF16))[0] == 2
    # head_dim 64 is outside what the library supports; MLA latents take
    # the symmetric 8/4/2-bit and grouped 8/4-bit vectors, not grouped 2-bit
    assert _plan_status(lib, _desc(lib, head_dim=64), _plan(lib, _sym(4), BF16, BF16, BF16))[0] == 5
    m = _desc(lib, kind=1, n_layers=1, n_q_heads=16, head_dim=128, latent_dim=512, rope_dim=64)
    for bits, scheme in ((8, 1), (4, 1), (2, 1), (8, 0), (4, 0)):
        ok, sizes = _plan_status(lib, m, _plan(lib, (0, bits, 0, 0, 0, 256, 0, scheme)))
        assert ok == 0 and sizes[0] > 0
    assert _plan_status(lib, m, _plan(lib, (0, 2, 0, 0, 0, 256, 0, 0)))[0] == 5
    # grouped 2-bit stays unsupported, and says where 2-bit codes are
    assert _plan_status(lib, d, _plan(lib, BF16, (0, 2, 32, 0, 0, 0, 0, 0), BF16, BF16))[0] == 5
    assert "symmetric" in lib.load().kvk_last_error().decode()


def test_symmetric_arena_and_cost(lib):
    from oracle import cost
    # per (position, kv head): codes of K and V (2 * 128 b / 8 bytes), plus
    # one 4-byte scale word in the scale plane
    B, H, T = 3, 2, 640
    d = _desc(lib, n_layers=3, max_batch=B, max_ctx=T)
    ok, sizes = _plan_status(lib, d, _plan(lib, _sym(8), _sym(4), _sym(2)))
    assert ok == 0
    for s, rec in zip(sizes, (256, 128, 64)):
        assert B * H * T * (rec + 4) <= s <= B * H * T * (rec + 4) + 4096
    # stored bits per element = b + 16/128 (Tab. realized_bits, "ours")
    for bits in (8, 4, 2):
        d1 = _desc(lib, n_layers=1, n_kv_heads=8, n_q_heads=40, max_batch=1, max_ctx=64)
        b, stored, rho = _plan_cost(lib, d1, _plan(lib, _sym(bits)))
        assert b == 2 * 8 * 128 * bits                    # eq. (cost): metadata-free
        per_elem = stored * 8 / (2 * 8 * 128)
        assert per_elem == pytest.approx(cost.bits_per_element_symmetric(bits))
        assert rho == pytest.approx(16 / bits)


def test_wait_limit_rejects_a_null_cache(lib):
    assert lib.load().kvk_set_wait_limit(None, 5) == 1  # KVK_ERR_INVALID_ARG


def test_decode_schedule_rejects_a_null_cache(lib):
    assert lib.load().kvk_set_decode_schedule(None, 0, 0, -1) == 1  # KVK_ERR_INVALID_ARG
