"""Heterogeneity-aware tensor-parallel shares (Voltron Section 4.2.1: under TP, shards go to
devices greedily by performance so that their execution times balance; within the memory budgets).
Host only: vt_plan_tp_shares launches nothing.

Pins: the 13B workload's stated 50/30/20 split of heads and FFN columns; even splits for equal
devices; KV-group alignment under GQA; the minimum makespan over every split, by brute force, on
small blocks; the block's bytes from the layer definition; memory budgets."""
from __future__ import annotations

import dataclasses
import itertools
import math

import numpy as np
import pytest

import synthetic


def shapes(vt, wl, max_seq=None):
    return vt.make_shapes(wl.n_layers, wl.d_model, wl.n_heads, wl.n_kv_heads, wl.d_head, wl.d_ffn,
                          0, wl.kv_len + 8 if max_seq is None else max_seq, wl.rms_eps, wl.rope_theta)


def block_bytes(wl, block, max_seq):
    """fp16 bytes of a whole ATTN or FFN block of one layer, from the layer's definition."""
    D, H, Hk, dh, F = wl.d_model, wl.n_heads, wl.n_kv_heads, wl.d_head, wl.d_ffn
    if block == 0:
        wqkv = (H + 2 * Hk) * dh * D
        wo = D * H * dh
        cache = 2 * Hk * max_seq * dh
        return 2 * (wqkv + wo + cache)
    return 2 * 3 * D * F


def sizes(ranges):
    return [b - a for a, b in ranges]


def contiguous(ranges, total):
    at = 0
    for a, b in ranges:
        assert a == at and b >= a
        at = b
    assert at == total


def test_13b_fifty_thirty_twenty(vtlib):
    """Device rates 5:3:2 give the 13B workload's own partition: heads 20/12/8, FFN columns
    6912/4147/2765 (the integer split of 13824 in that ratio with the smallest makespan)."""
    wl = synthetic.WORKLOADS[3]
    s = shapes(vtlib, wl)
    heads, _ = vtlib.vt_plan_tp_shares(s, vtlib.VT_BLOCK_ATTN, [5.0, 3.0, 2.0])
    cols, _ = vtlib.vt_plan_tp_shares(s, vtlib.VT_BLOCK_FFN, [5.0, 3.0, 2.0])
    assert heads == list(wl.head_ranges) == [(0, 20), (20, 32), (32, 40)]
    assert cols == list(wl.ffn_ranges) == [(0, 6912), (6912, 11059), (11059, 13824)]
    assert vtlib.vt_partition_validate(s, heads, cols) == vtlib.VT_OK


def test_equal_devices_split_evenly(vtlib):
    wl = synthetic.WORKLOADS[2]
    s = shapes(vtlib, wl)
    heads, _ = vtlib.vt_plan_tp_shares(s, vtlib.VT_BLOCK_ATTN, [1.0] * 4)
    cols, _ = vtlib.vt_plan_tp_shares(s, vtlib.VT_BLOCK_FFN, [1.0] * 4)
    assert heads == list(wl.head_ranges) and cols == list(wl.ffn_ranges)


def test_gqa_shares_are_whole_kv_groups(vtlib):
    wl = synthetic.WORKLOADS[5]   # 32 query heads, 8 KV heads
    s = shapes(vtlib, wl)
    heads, _ = vtlib.vt_plan_tp_shares(s, vtlib.VT_BLOCK_ATTN, [3.0, 1.0])
    assert heads == [(0, 24), (24, 32)]
    heads, _ = vtlib.vt_plan_tp_shares(s, vtlib.VT_BLOCK_ATTN, [1.0, 1.0, 1.0, 1.0])
    assert heads == list(wl.head_ranges)
    for rates in ([7.0, 1.0, 2.5], [1.0, 100.0], [2.0, 2.0, 1.0, 0.5, 3.0]):
        heads, _ = vtlib.vt_plan_tp_shares(s, vtlib.VT_BLOCK_ATTN, rates)
        assert all(a % 4 == 0 and b % 4 == 0 for a, b in heads)
        cols, _ = vtlib.vt_plan_tp_shares(s, vtlib.VT_BLOCK_FFN, rates, col_unit=64)
        assert vtlib.vt_partition_validate(s, heads, cols) == vtlib.VT_OK


def test_one_device_takes_the_whole_block(vtlib):
    """The makespan of a single device is the block's bytes (from the layer definition) over its rate."""
    for cid in (1, 2, 5):
        wl = synthetic.WORKLOADS[cid]
        max_seq = wl.kv_len + 8
        s = shapes(vtlib, wl, max_seq)
        for block in (0, 1):
            r, ms = vtlib.vt_plan_tp_shares(s, block, [2.5e12])
            assert r == [(0, wl.n_heads if block == 0 else wl.d_ffn)]
            assert ms == pytest.approx(block_bytes(wl, block, max_seq) / 2.5e12, rel=1e-12)


def brute_force(units, rates, cap=None):
    """Smallest makespan over every split of `units` equal units (unit time 1 / rate)."""
    best = math.inf
    n = len(rates)
    for cuts in itertools.product(range(units + 1), repeat=n - 1):
        c = list(cuts) + [units - sum(cuts)]
        if c[-1] < 0:
            continue
        if cap is not None and any(c[d] > cap[d] for d in range(n)):
            continue
        best = min(best, max(c[d] / rates[d] for d in range(n)))
    return best


@pytest.mark.parametrize("seed", range(12))
def test_greedy_reaches_the_brute_force_minimum(vtlib, seed):
    rng = np.random.default_rng(500 + seed)
    n = int(rng.integers(2, 4))
    rates = [float(x) for x in rng.uniform(0.2, 5.0, n)]
    F = int(rng.integers(1, 14))
    s = vtlib.make_shapes(1, 256, 4, 4, 64, F, 0, 64)
    cols, ms = vtlib.vt_plan_tp_shares(s, vtlib.VT_BLOCK_FFN, rates)
    contiguous(cols, F)
    unit = 2 * 3 * 256
    best = brute_force(F, rates)
    assert ms == pytest.approx(best * unit, rel=1e-12)
    assert max(c * unit / r for c, r in zip(sizes(cols), rates)) == pytest.approx(ms, rel=1e-12)


@pytest.mark.parametrize("seed", range(6))
def test_memory_budgets_are_respected_and_still_minimal(vtlib, seed):
    rng = np.random.default_rng(700 + seed)
    rates = [float(x) for x in rng.uniform(0.5, 4.0, 3)]
    F = 12
    unit = 2 * 3 * 256
    cap = [int(x) for x in rng.integers(2, 9, 3)]
    if sum(cap) < F:
        cap[0] = F
    s = vtlib.make_shapes(1, 256, 4, 4, 64, F, 0, 64)
    cols, ms = vtlib.vt_plan_tp_shares(s, vtlib.VT_BLOCK_FFN, rates, mem_bytes=[c * unit for c in cap])
    contiguous(cols, F)
    assert all(n <= c for n, c in zip(sizes(cols), cap))
    assert ms == pytest.approx(brute_force(F, rates, cap) * unit, rel=1e-12)


def test_the_fastest_device_fills_first_up_to_its_budget(vtlib):
    s = vtlib.make_shapes(1, 256, 4, 4, 64, 100, 0, 64)
    unit = 2 * 3 * 256
    cols, _ = vtlib.vt_plan_tp_shares(s, vtlib.VT_BLOCK_FFN, [100.0, 1.0], mem_bytes=[30 * unit, 1e30])
    assert sizes(cols) == [30, 70]
    with pytest.raises(vtlib.VtError) as e:
        vtlib.vt_plan_tp_shares(s, vtlib.VT_BLOCK_FFN, [1.0, 1.0], mem_bytes=[30 * unit, 60 * unit])
    assert e.value.status == vtlib.VT_ERR_PLAN_MEMORY


def test_column_units_and_a_short_last_unit(vtlib):
    s = vtlib.make_shapes(1, 256, 4, 4, 64, 1000, 0, 64)
    cols, _ = vtlib.vt_plan_tp_shares(s, vtlib.VT_BLOCK_FFN, [1.0, 1.0, 1.0], col_unit=64)
    contiguous(cols, 1000)
    assert all(a % 64 == 0 for a, _ in cols)
    assert sizes(cols) == [384, 320, 296]   # 16 units of 64 (the last one 40 columns): 6 / 5 / 5


@pytest.mark.parametrize("rates,kw", [
    ([0.0, 1.0], {}), ([-1.0], {}), ([float("nan")], {}), ([float("inf")], {}), ([], {}),
    ([1.0] * 17, {}), ([1.0], dict(col_unit=0)), ([1.0, 1.0], dict(mem_bytes=[1.0, float("nan")])),
])
def test_invalid_arguments(vtlib, rates, kw):
    s = vtlib.make_shapes(1, 256, 4, 4, 64, 100, 0, 64)
    with pytest.raises(vtlib.VtError) as e:
        vtlib.vt_plan_tp_shares(s, vtlib.VT_BLOCK_FFN, rates, **kw)
    assert e.value.status == vtlib.VT_ERR_INVALID_ARG


# ------------------------------------------------------------------ layer-wise MP / TP plan

def block_time_bytes(wl, block, kv_len, tokens):
    """Bytes a whole block streams for `tokens` new rows: fp16 weights, plus for ATTN the K and V
    rows read at kv_len and written for the new rows."""
    D, H, Hk, dh, F = wl.d_model, wl.n_heads, wl.n_kv_heads, wl.d_head, wl.d_ffn
    if block == 0:
        return 2 * ((H + 2 * Hk) * dh * D + D * H * dh) + 2 * 2 * Hk * dh * (kv_len + tokens)
    return 2 * 3 * D * F


def block_flops(wl, block, kv_len, tokens):
    """Multiply-adds x 2 of a block over `tokens` rows: projections, and for ATTN the scores and the
    weighted values over the causally visible positions (row i sees kv_len + i + 1)."""
    D, H, Hk, dh, F = wl.d_model, wl.n_heads, wl.n_kv_heads, wl.d_head, wl.d_ffn
    if block == 0:
        proj = 2 * tokens * ((H + 2 * Hk) * dh * D + D * H * dh)
        visible = sum(kv_len + i + 1 for i in range(tokens))
        return proj + 2 * 2 * H * dh * visible
    return 2 * tokens * 3 * D * F


def plan_shapes(vt, wl, max_seq):
    return vt.make_shapes(wl.n_layers, wl.d_model, wl.n_heads, wl.n_kv_heads, wl.d_head, wl.d_ffn, 0, max_seq,
                          wl.rms_eps, wl.rope_theta)


def test_one_device_runs_every_block_without_transfers(vtlib):
    wl = synthetic.WORKLOADS[2]
    s = plan_shapes(vtlib, wl, 2048)
    plans, total = vtlib.vt_plan_layers(s, [3e12], link_bytes_per_s=1e9, link_latency_s=1e-3, kv_len=1024)
    assert len(plans) == 2 * wl.n_layers
    for i, p in enumerate(plans):
        assert not p["tp"] and p["device"] == 0 and p["comm_s"] == 0.0
        assert p["compute_s"] == pytest.approx(block_time_bytes(wl, i % 2, 1024, 1) / 3e12, rel=1e-12)
    want = wl.n_layers * (block_time_bytes(wl, 0, 1024, 1) + block_time_bytes(wl, 1, 1024, 1)) / 3e12
    assert total == pytest.approx(want, rel=1e-12)


def test_free_link_splits_every_block_evenly(vtlib):
    """Two equal devices and a link that costs nothing: TP halves every block's time."""
    wl = synthetic.WORKLOADS[2]
    s = plan_shapes(vtlib, wl, 2048)
    one, t1 = vtlib.vt_plan_layers(s, [1e12], kv_len=1024)
    two, t2 = vtlib.vt_plan_layers(s, [1e12, 1e12], link_bytes_per_s=1e30, link_latency_s=0.0, kv_len=1024)
    for i, p in enumerate(two):
        assert p["tp"] and p["device"] == 0
        assert p["ranges"] == ([(0, 16), (16, 32)] if i % 2 == 0 else [(0, 5504), (5504, 11008)])
    assert t2 == pytest.approx(t1 / 2, rel=1e-9)


def test_slow_link_keeps_the_stack_on_the_fastest_device(vtlib):
    """A link too slow for TP: every block on the fastest device (device 1); the input moves there
    once, before the first block."""
    wl = synthetic.WORKLOADS[2]
    s = plan_shapes(vtlib, wl, 2048)
    bps, lat = 1e6, 2e-3
    plans, total = vtlib.vt_plan_layers(s, [1e12, 2e12], link_bytes_per_s=bps, link_latency_s=lat, kv_len=1024)
    assert all(not p["tp"] and p["device"] == 1 for p in plans)
    assert plans[0]["comm_s"] == pytest.approx(lat + wl.d_model * 2 / bps, rel=1e-12)
    assert all(p["comm_s"] == 0.0 for p in plans[1:])
    assert plans[0]["ranges"][1] == (0, wl.n_heads) and plans[1]["ranges"][1] == (0, wl.d_ffn)


def test_memory_moves_the_rest_of_the_stack_once(vtlib):
    """The fastest device holds 3 blocks: blocks 0-2 run there, the rest on device 0, with one
    transfer when the activations change device (slow link, so TP never pays)."""
    wl = dataclasses.replace(synthetic.WORKLOADS[2], n_layers=4)
    max_seq = 2048
    s = plan_shapes(vtlib, wl, max_seq)
    D, H, Hk, dh, F = wl.d_model, wl.n_heads, wl.n_kv_heads, wl.d_head, wl.d_ffn
    attn_mem = 2 * ((H + 2 * Hk) * dh * D + D * H * dh) + 2 * 2 * Hk * dh * max_seq
    ffn_mem = 2 * 3 * D * F
    budget1 = 2 * attn_mem + ffn_mem + 1.0   # ATTN 0, FFN 0, ATTN 1
    bps, lat = 1e6, 1e-3
    plans, _ = vtlib.vt_plan_layers(s, [1e12, 4e12], mem_bytes=[1e30, budget1], link_bytes_per_s=bps,
                                    link_latency_s=lat, kv_len=1024)
    assert [p["device"] for p in plans] == [1, 1, 1, 0, 0, 0, 0, 0]
    assert not any(p["tp"] for p in plans)
    hop = lat + D * 2 / bps
    assert [p["comm_s"] for p in plans] == pytest.approx([hop, 0, 0, hop, 0, 0, 0, 0])


def test_prefill_time_is_the_flop_bound_when_the_flop_rate_is_low(vtlib):
    wl = dataclasses.replace(synthetic.WORKLOADS[4], n_layers=1)
    s = plan_shapes(vtlib, wl, 1024)
    plans, _ = vtlib.vt_plan_layers(s, [1e12], flop_rate=[1e9], tokens=512, kv_len=0)
    for b in (0, 1):
        assert plans[b]["compute_s"] == pytest.approx(block_flops(wl, b, 0, 512) / 1e9, rel=1e-12)
    plans, _ = vtlib.vt_plan_layers(s, [1e6], flop_rate=[1e30], tokens=512, kv_len=0)
    for b in (0, 1):
        assert plans[b]["compute_s"] == pytest.approx(block_time_bytes(wl, b, 0, 512) / 1e6, rel=1e-12)


def test_heterogeneous_devices_on_a_fast_link_get_their_rate_shares(vtlib):
    wl = synthetic.WORKLOADS[3]
    s = plan_shapes(vtlib, wl, 2056)
    plans, _ = vtlib.vt_plan_layers(s, [5e11, 3e11, 2e11], link_bytes_per_s=1e30, kv_len=2048)
    assert all(p["tp"] for p in plans)
    assert plans[1]["ranges"] == list(wl.ffn_ranges)


def test_no_device_can_hold_a_block(vtlib):
    wl = dataclasses.replace(synthetic.WORKLOADS[2], n_layers=2)
    s = plan_shapes(vtlib, wl, 2048)
    with pytest.raises(vtlib.VtError) as e:
        vtlib.vt_plan_layers(s, [1e12, 1e12], mem_bytes=[1e6, 1e6], kv_len=0)
    assert e.value.status == vtlib.VT_ERR_PLAN_MEMORY


@pytest.mark.parametrize("kw", [
    dict(tokens=0), dict(kv_len=-1), dict(kv_len=2048, tokens=1), dict(link_bytes_per_s=0.0),
    dict(link_latency_s=-1.0), dict(link_bytes_per_s=float("nan")), dict(flop_rate=[0.0, 1.0]),
])
def test_plan_layers_invalid_arguments(vtlib, kw):
    wl = dataclasses.replace(synthetic.WORKLOADS[2], n_layers=1)
    s = plan_shapes(vtlib, wl, 2048)
    args = dict(rate=[1e12, 1e12], kv_len=0)
    args.update(kw)
    with pytest.raises(vtlib.VtError) as e:
        vtlib.vt_plan_layers(s, **args)
    assert e.value.status == vtlib.VT_ERR_INVALID_ARG


@pytest.mark.parametrize("seed", range(20))
def test_plans_are_always_valid_partitions(vtlib, seed):
    """Random shapes, device counts, rates and budgets: the share balancer's and the layer plan's
    ranges always pass vt_partition_validate (whole KV groups, full coverage, device order)."""
    rng = np.random.default_rng(900 + seed)
    H = int(rng.choice([4, 8, 16, 32, 40]))
    Hk = int(rng.choice([g for g in (1, 2, 4, 8, 16, 32, 40) if H % g == 0 and H // g in (1, 2, 4, 8)]))
    F = int(rng.integers(1, 3000))
    s = vtlib.make_shapes(2, 256, H, Hk, 64, F, 0, 128)
    n = int(rng.integers(1, 9))
    rates = [float(x) for x in rng.uniform(0.1, 10.0, n)]
    heads, _ = vtlib.vt_plan_tp_shares(s, vtlib.VT_BLOCK_ATTN, rates)
    cols, _ = vtlib.vt_plan_tp_shares(s, vtlib.VT_BLOCK_FFN, rates, col_unit=int(rng.choice([1, 8, 64])))
    assert vtlib.vt_partition_validate(s, heads, cols) == vtlib.VT_OK
    plans, total = vtlib.vt_plan_layers(s, rates, link_bytes_per_s=float(10 ** rng.uniform(5, 12)),
                                        link_latency_s=float(rng.uniform(0, 1e-2)), tokens=int(rng.integers(1, 64)),
                                        kv_len=int(rng.integers(0, 64)))
    assert total > 0
    for i in range(0, len(plans), 2):
        assert vtlib.vt_partition_validate(s, plans[i]["ranges"], plans[i + 1]["ranges"]) == vtlib.VT_OK
        for p in plans[i:i + 2]:
            if not p["tp"]:
                sizes_ = [b - a for a, b in p["ranges"]]
                assert sum(1 for x in sizes_ if x) == 1 and sizes_[p["device"]] > 0


# ------------------------------------------------------------------ importance-aware precision
# Voltron Section 4.2.2: blocks are lowered one precision step at a time (fp16 -> INT8 -> INT4) in
# ascending order of importance, and the number of steps is the smallest that meets the memory
# budgets and the time budget, found by binary search (memory and time do not grow with steps).
# Pins: the byte counts restated here from the layer definition and the block format (codes plus
# one fp16 scale per 32 weights along the contraction axis); the result equals a linear scan over
# every configuration; the lowered blocks are the least important ones; no budget lowers nothing.

def _q_bytes(rows, k, bits):
    if bits == 16:
        return rows * k * 2
    return rows * math.ceil(k / 32) * (32 * bits // 8 + 2)


def _config(nb, order, k):
    bits = [16] * nb
    for i, b in enumerate(order):
        if i < k:
            bits[b] = 8
        if i < k - nb:
            bits[b] = 4
    return bits


def _cost(wl, plans, bits, rate, kv_len, max_seq):
    """Each device's memory and the stack's time for one configuration, from the definitions."""
    D, dh, g = wl.d_model, wl.d_head, wl.n_heads // wl.n_kv_heads
    n = len(rate)
    used = [0.0] * n
    t = 0.0
    for b, p in enumerate(plans):
        slow = 0.0
        for d, (lo, hi) in enumerate(p["ranges"]):
            c = hi - lo
            if c == 0:
                continue
            if b % 2 == 0:
                hk = c // g
                w = _q_bytes((c + 2 * hk) * dh, D, bits[b]) + _q_bytes(D, c * dh, bits[b])
                mem = w + 2 * 2 * hk * max_seq * dh
                stream = w + 2 * 2 * hk * dh * (kv_len + 1)
            else:
                w = _q_bytes(2 * c, D, bits[b]) + _q_bytes(D, c, bits[b])
                mem = stream = w
            used[d] += mem
            slow = max(slow, stream / rate[d])
        t += slow + p["comm_s"]
    return used, t


def _even_plans(wl, n):
    """Every block split evenly (whole KV groups for ATTN) over n devices."""
    g = wl.n_heads // wl.n_kv_heads

    def split(total, unit):
        units = total // unit
        cuts = [unit * (units * d // n) for d in range(n + 1)]
        cuts[-1] = total
        return [(cuts[d], cuts[d + 1]) for d in range(n)]

    plans = []
    for _ in range(wl.n_layers):
        plans.append(dict(tp=1, device=0, ranges=split(wl.n_heads, g), comm_s=1e-5))
        plans.append(dict(tp=1, device=0, ranges=split(wl.d_ffn, 1), comm_s=1e-5))
    return plans


def _precision_wl():
    return synthetic.small("prec", n_layers=4, d_model=512, n_heads=8, n_kv_heads=4, d_head=64, d_ffn=1000,
                           head_ranges=((0, 4), (4, 8)), ffn_ranges=((0, 500), (500, 1000)), kv_len=64)


def test_precision_without_budgets_stays_fp16(vtlib):
    wl = _precision_wl()
    sh = shapes(vtlib, wl, max_seq=128)
    plans = _even_plans(wl, 2)
    bits, steps, t = vtlib.vt_plan_precision(sh, plans, list(range(8)), [1e9, 1e9], kv_len=64)
    assert bits == [16] * 8 and steps == 0
    assert t == pytest.approx(_cost(wl, plans, bits, [1e9, 1e9], 64, 128)[1], rel=1e-12)


@pytest.mark.parametrize("seed", range(12))
def test_precision_binary_search_equals_a_linear_scan(vtlib, seed):
    rng = np.random.default_rng(seed)
    wl = _precision_wl()
    max_seq, kv_len = 128, int(rng.integers(0, 127))
    sh = shapes(vtlib, wl, max_seq=max_seq)
    n = int(rng.integers(1, 4))
    plans = _even_plans(wl, n)
    nb = 2 * wl.n_layers
    importance = list(rng.normal(size=nb))
    rate = list(rng.uniform(1e9, 4e9, size=n))
    order = sorted(range(nb), key=lambda b: (importance[b], b))
    costs = [_cost(wl, plans, _config(nb, order, k), rate, kv_len, max_seq) for k in range(2 * nb + 1)]
    # memory and time do not grow with k
    for (m0, t0), (m1, t1) in zip(costs, costs[1:]):
        assert all(b <= a + 1e-9 for a, b in zip(m0, m1)) and t1 <= t0 + 1e-15
    # budgets between the fp16 and all-INT4 costs
    k_mem, k_t = rng.integers(0, 2 * nb + 1, size=2)
    mem = [costs[k_mem][0][d] for d in range(n)]
    qos = costs[k_t][1] * (1 + 1e-12)
    want = next(k for k in range(2 * nb + 1)
                if all(costs[k][0][d] <= mem[d] for d in range(n)) and costs[k][1] <= qos)
    bits, steps, t = vtlib.vt_plan_precision(sh, plans, importance, rate, mem_bytes=mem, qos_s=qos, kv_len=kv_len)
    assert steps == want
    assert bits == _config(nb, order, want)
    assert t == pytest.approx(costs[want][1], rel=1e-12)
    # the lowered blocks are the least important ones
    lowered = [b for b in range(nb) if bits[b] < 16]
    kept = [b for b in range(nb) if bits[b] == 16]
    if lowered and kept:
        assert max(importance[b] for b in lowered) <= min(importance[b] for b in kept)


def test_precision_budgets_that_no_configuration_meets(vtlib):
    wl = _precision_wl()
    sh = shapes(vtlib, wl, max_seq=128)
    plans = _even_plans(wl, 2)
    imp = [0.0] * 8
    with pytest.raises(vtlib.VtError) as e:
        vtlib.vt_plan_precision(sh, plans, imp, [1e9, 1e9], mem_bytes=[1.0, 1.0])
    assert e.value.status == vtlib.VT_ERR_PLAN_MEMORY
    with pytest.raises(vtlib.VtError) as e:
        vtlib.vt_plan_precision(sh, plans, imp, [1e9, 1e9], qos_s=1e-9)
    assert e.value.status == vtlib.VT_ERR_PLAN_QOS
    bad = [dict(p) for p in plans]
    bad[0] = dict(bad[0], ranges=[(0, 3), (3, 8)])  # 3 heads are not whole KV groups of 2
    with pytest.raises(vtlib.VtError) as e:
        vtlib.vt_plan_precision(sh, bad, imp, [1e9, 1e9])
    assert e.value.status == vtlib.VT_ERR_PARTITION_GQA


def test_precision_int8_shard_bytes_match_the_library_format(vtlib):
    """The planner's INT8 / INT4 bytes are the block format vt_quantize_rows writes: one code per
    weight (a nibble at INT4) and one fp16 scale per 32 weights of a row."""
    rows, k = 6, 70
    w = np.random.default_rng(1).normal(0, 0.02, size=(rows, k)).astype(np.float16)
    for bits in (8, 4):
        q, sc = vtlib.vt_quantize_rows(w, bits)
        assert sc.shape == (rows, math.ceil(k / 32))
        assert _q_bytes(rows, k, bits) == rows * math.ceil(k / 32) * 32 * bits // 8 + sc.nbytes
