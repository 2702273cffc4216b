"""The C ABI library loads and exports every declared entry point; host-side validation rules
(no GPU needed: nothing here launches a kernel)."""
from __future__ import annotations

import ctypes
import re
from pathlib import Path

import pytest

ROOT = Path(__file__).resolve().parents[1]


def declared_symbols():
    text = (ROOT / "include" / "voltron.h").read_text()
    return sorted(set(re.findall(r"^VT_API\s+[^;(]*?\b(vt_[a-z0-9_]+)\s*\(", text, flags=re.M)))


def test_header_declares_the_core_calls():
    names = declared_symbols()
    for must in ("vt_model_create", "vt_partition_create", "vt_prefill", "vt_decode_step",
                 "vt_combine", "vt_kv_create", "vt_decode_token", "vt_prefill_tokens"):
        assert must in names
    assert len(names) >= 30


def test_library_exports_every_declared_symbol(vtlib):
    L = ctypes.CDLL(str(vtlib.LIB_PATH))
    missing = [n for n in declared_symbols() if not hasattr(L, n)]
    assert not missing, missing


def test_version(vtlib):
    assert re.fullmatch(r"\d+\.\d+\.\d+", vtlib.vt_version())


def S(vt, **kw):
    base = dict(n_layers=2, d_model=512, n_heads=8, n_kv_heads=8, d_head=64, d_ffn=1408, vocab=0,
                max_seq=256)
    base.update(kw)
    return vt.make_shapes(**base)


@pytest.mark.parametrize("kw,ok", [
    (dict(), True),
    (dict(d_model=500), False),
    (dict(d_head=96), False),
    (dict(n_heads=8, n_kv_heads=3), False),
    (dict(n_heads=32, n_kv_heads=2), False),   # 16 query heads per KV head: unsupported
    (dict(n_heads=32, n_kv_heads=4), True),
    (dict(n_heads=24, n_kv_heads=4), False),   # group of 6: not instantiated
    (dict(n_layers=0), False),
    (dict(d_ffn=0), False),
    (dict(max_seq=0), False),
])
def test_shapes_validate(vtlib, kw, ok):
    st = vtlib.vt_shapes_validate(S(vtlib, **kw))
    assert (st == vtlib.VT_OK) == ok
    if not ok:
        assert st == vtlib.VT_ERR_SHAPE and vtlib.vt_last_error()


@pytest.mark.parametrize("heads,cols,code", [
    ([(0, 4), (4, 8)], [(0, 704), (704, 1408)], 0),
    ([(0, 8)], [(0, 1408)], 0),
    ([(0, 4), (4, 4), (4, 8)], [(0, 0), (0, 1), (1, 1408)], 0),          # empty shards
    ([(0, 5), (4, 8)], [(0, 704), (704, 1408)], 3),                       # overlap
    ([(0, 3), (4, 8)], [(0, 704), (704, 1408)], 4),                       # gap
    ([(0, 4), (4, 7)], [(0, 704), (704, 1408)], 4),                       # union short
    ([(0, 4), (4, 8)], [(0, 704), (704, 1407)], 4),
    ([(0, 4), (4, 9)], [(0, 704), (704, 1408)], 6),                       # beyond H
    ([(0, 4), (5, 4)], [(0, 704), (704, 1408)], 6),                       # begin > end
    ([(0, 4), (4, 8)], [(0, 800), (704, 1408)], 3),
])
def test_partition_validate(vtlib, heads, cols, code):
    assert vtlib.vt_partition_validate(S(vtlib), heads, cols) == code


def test_partition_validate_gqa_alignment(vtlib):
    s = S(vtlib, n_heads=32, n_kv_heads=8, d_head=128, d_model=4096, d_ffn=14336)
    even = [(0, 8), (8, 16), (16, 24), (24, 32)]
    cols = [(0, 3584), (3584, 7168), (7168, 10752), (10752, 14336)]
    assert vtlib.vt_partition_validate(s, even, cols) == vtlib.VT_OK
    assert vtlib.vt_partition_validate(s, [(0, 6), (6, 32)], cols[:2]) == vtlib.VT_ERR_PARTITION_GQA


def test_partition_validate_device_count(vtlib):
    s = S(vtlib)
    assert vtlib.vt_partition_validate(s, [], []) == vtlib.VT_ERR_INVALID_ARG
    heads = [(i // 2 * 1, i // 2 * 1) for i in range(17)]
    assert vtlib.vt_partition_validate(s, heads, heads) == vtlib.VT_ERR_INVALID_ARG


def test_workload_partitions_are_valid(vtlib):
    import synthetic
    for wl in synthetic.WORKLOADS.values():
        s = vtlib.make_shapes(wl.n_layers, wl.d_model, wl.n_heads, wl.n_kv_heads, wl.d_head,
                              wl.d_ffn, wl.vocab, wl.max_seq, wl.rms_eps, wl.rope_theta)
        assert vtlib.vt_shapes_validate(s) == 0, (wl.name, vtlib.vt_last_error())
        assert vtlib.vt_partition_validate(s, wl.head_ranges, wl.ffn_ranges) == 0, wl.name


def test_partition_table_rules(vtlib):
    """Per-layer partition tables (host-only validation): gaps need VT_PARTITION_PRUNE, KV-group
    alignment and ordering still hold, unknown flags are refused."""
    from tests.test_gpu_layers import PER_LAYER, PRUNED, WL
    vt = vtlib
    wl = WL
    s = vt.make_shapes(wl.n_layers, wl.d_model, wl.n_heads, wl.n_kv_heads, wl.d_head, wl.d_ffn, wl.vocab,
                       wl.max_seq, wl.rms_eps, wl.rope_theta)
    heads, cols = PRUNED
    assert vt.vt_partition_validate_layers(s, heads, cols, 0) == vt.VT_ERR_PARTITION_GAP
    assert vt.vt_partition_validate_layers(s, heads, cols, vt.VT_PARTITION_PRUNE) == vt.VT_OK
    assert vt.vt_partition_validate_layers(s, *PER_LAYER, 0) == vt.VT_OK
    bad = [[(0, 3), (3, 6), (6, 8)]] + PER_LAYER[0][1:]  # a head range off the KV groups of 2
    assert vt.vt_partition_validate_layers(s, bad, PER_LAYER[1], 0) == vt.VT_ERR_PARTITION_GQA
    over = [[(0, 4), (2, 6), (6, 8)]] + PER_LAYER[0][1:]
    assert vt.vt_partition_validate_layers(s, over, PER_LAYER[1], vt.VT_PARTITION_PRUNE) == vt.VT_ERR_PARTITION_OVERLAP
    assert vt.vt_partition_validate_layers(s, *PER_LAYER, 2) == vt.VT_ERR_INVALID_ARG
