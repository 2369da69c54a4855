"""Pins for oracle/cost.py against numbers the paper prints (no GPU)."""
import json
import math
import os

import pytest

from oracle import cost


def _golden(golden_dir, name):
    with open(os.path.join(golden_dir, name)) as f:
        return json.load(f)


def _close_printed(value, printed):
    # the paper prints 2-3 significant digits
    s = f"{printed}"
    decimals = len(s.split(".")[1]) if "." in s else 0
    return abs(value - printed) <= 0.5 * 10 ** (-decimals) + 1e-9


def test_tab_ranges(golden_dir):
    g = _golden(golden_dir, "tab_ranges.json")
    for row in g["rows"]:
        for name, m in g["models"].items():
            acts = cost.action_space(m["r"], depth=row["depth"], rank=row["rank"], precision=row["precision"])
            assert len(acts) == row["actions"]
            assert round(cost.plan_count_log10(m["L"], len(acts))) == row["plans_log10"][name]
            lo, hi = cost.rho_range(m["L"], m["n_kv"], m["d_h"], m["r"], row["mla"],
                                    row["depth"], row["rank"], row["precision"])
            plo, phi = row["range"][name]
            assert _close_printed(lo, plo), (row["axes"], name, lo, plo)
            assert _close_printed(hi, phi), (row["axes"], name, hi, phi)


def test_action_space_has_17_actions():
    assert len(cost.action_space(1024)) == 17            # eq. (action space)


def test_tab_realized_bits(golden_dir):
    g = _golden(golden_dir, "tab_realized_bits.json")
    for row in g["ours"]:
        bits = cost.bits_per_element_symmetric(row["b"])
        assert _close_printed(bits, row["bits"]) and _close_printed(16 / bits, row["rho"])
    for row in g["kivi"]:
        bits = cost.bits_per_element_grouped(row["b"], row["g"], meta_bits=32,
                                            window=g["kivi_window"], context=g["kivi_context"])
        assert _close_printed(bits, row["bits"]), (row, bits)
        assert _close_printed(16 / bits, row["rho"]), (row, 16 / bits)
    tv = g["text_values"]
    assert _close_printed(16 / cost.bits_per_element_grouped(2, 128), tv["kivi_2bit_g128_no_window_rho"])
    b16k = cost.bits_per_element_grouped(4, 128, window=128, context=16384)
    assert _close_printed(b16k, tv["kivi_4bit_g128_16k_bits"]) and _close_printed(16 / b16k, tv["kivi_4bit_g128_16k_rho"])


def test_intro_cache_size_and_on_device_factors(golden_dir):
    g = _golden(golden_dir, "cache_sizes.json")
    m = g["intro"]["model"]
    per_tok = m["L"] * 2 * m["n_kv"] * m["d_h"] * m["bytes_per_scalar"]
    assert per_tok == g["intro"]["kib_per_token"] * 1024
    tot = per_tok * g["intro"]["sequences"] * g["intro"]["tokens_per_sequence"]
    assert tot == g["intro"]["gib_total"] * 2 ** 30
    od = g["on_device"]
    L, nkv, dh = 48, 8, 128
    bits4 = cost.bits_per_element_grouped(4, od["mlx_group"], od["mlx_meta_bits"])
    assert _close_printed(16 / bits4, od["rho_4bit"])
    rank = cost.compression([(128, 16)] * L, L, nkv, dh, mla=True)
    assert _close_printed(rank, od["rho_rank128"])
    depth = cost.compression([(None, 16) if l % 4 == 0 else "inherit" for l in range(L)], L, nkv, dh, mla=False)
    assert _close_printed(depth, od["rho_depth"])
    # all three: rank-128 latent + positional key at the MLX 4.5 bits, 12 anchors
    all3 = cost.c0_bits(L, nkv, dh) / (12 * (128 + 64) * bits4)
    assert round(all3) == od["rho_all"]
    ms = g["mla_start"]
    r14 = cost.compression([(1024, 16)] * 48, 48, 8, 128, mla=True)
    r3 = cost.compression([(256, 16)] * 36, 36, 2, 128, mla=True)
    assert _close_printed(r3, ms["rho_min"]) and _close_printed(r14, ms["rho_max"])
    assert cost.rho_range(48, 8, 128, 1024, True, True, True, True)[1] == g["max_compression"]["rho"]


def test_layer_one_must_own_a_cache():
    with pytest.raises(ValueError):
        cost.compression(["inherit"] + [(None, 16)] * 3, 4, 8, 128, mla=False)
