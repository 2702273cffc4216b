"""The benchmark's roofline arithmetic (algorithmic bytes and FLOPs per step), recomputed on CPU a
second way: weights summed shard by shard from the partition's head and column ranges, KV bytes
per position and KV head, FLOPs of the causal attention summed row by row.  These figures are the
numerators of every `roofline.achieved` the bench prints."""
from __future__ import annotations

import dataclasses
import sys
from pathlib import Path

import pytest

import synthetic

ROOT = Path(__file__).resolve().parents[1]
sys.path.insert(0, str(ROOT))
import bench  # noqa: E402


def shard_weight_bytes(wl):
    """fp16 bytes of one layer's weights, shard by shard, and its two RMSNorm gains (one buffer
    each on the device, read by every shard)."""
    D, H, Hk, dh = wl.d_model, wl.n_heads, wl.n_kv_heads, wl.d_head
    total = 2 * 2 * D
    for (h0, h1), (c0, c1) in zip(wl.head_ranges, wl.ffn_ranges):
        hq, c = h1 - h0, c1 - c0
        hk = hq * Hk // H
        if hq:
            total += 2 * ((hq + 2 * hk) * dh * D + D * hq * dh)  # Wqkv rows, Wo columns
        if c:
            total += 2 * (2 * c * D + D * c)  # gate and up rows, down columns
    return total


@pytest.mark.parametrize("cid", [2, 3, 4, 5])
def test_decode_bytes_equal_the_shards_weights_and_the_cache(cid):
    wl = synthetic.WORKLOADS[cid]
    kv_mean = wl.kv_len + 63.5
    per_layer_kv = 2 * 2 * wl.n_kv_heads * wl.d_head * (kv_mean + 1)  # K and V rows read, one written
    expect = wl.n_layers * (shard_weight_bytes(wl) + per_layer_kv)
    assert bench.decode_bytes_per_token(wl, kv_mean) == pytest.approx(expect, rel=1e-12)


def test_7b_decode_bytes_match_the_quoted_figures():
    """12.952 GB of weights per token and 13.523 GB at the 128-token schedule's mean length."""
    wl = synthetic.WORKLOADS[2]
    weights = bench.decode_bytes_per_token(wl, -1)  # kv_mean + 1 = 0: weights alone
    assert weights == pytest.approx(12.952e9, rel=1e-4)
    assert bench.decode_bytes_per_token(wl, 1024 + 127 / 2) == pytest.approx(13.523e9, rel=1e-4)


def test_quantized_bytes_are_codes_and_block_scales():
    """At 8 bits the codes take half the fp16 bytes, at 4 bits a quarter, plus one 2-byte scale
    per 32 weights; the gains stay fp16."""
    wl = dataclasses.replace(synthetic.WORKLOADS[2], n_layers=1)
    q8 = bench.quant_bytes_per_token(wl, 8, -1)
    fp16 = bench.decode_bytes_per_token(wl, -1)
    gains = 2 * 2 * wl.d_model
    # every weight matrix here has a multiple of 32 columns: codes = weights / 2, scales = weights / 32
    weights = fp16 - gains
    assert q8 == pytest.approx(weights / 2 + weights / 32 + gains, rel=1e-12)
    q4 = bench.quant_bytes_per_token(wl, 4, -1)
    assert q4 == pytest.approx(weights / 4 + weights / 32 + gains, rel=1e-12)


def test_prefill_flops_row_by_row():
    wl = synthetic.WORKLOADS[4]
    n = 512
    D, H, Hk, dh, F = wl.d_model, wl.n_heads, wl.n_kv_heads, wl.d_head, wl.d_ffn
    gemm = 0
    for (h0, h1), (c0, c1) in zip(wl.head_ranges, wl.ffn_ranges):
        hq, c = h1 - h0, c1 - c0
        hk = hq * Hk // H
        gemm += 2 * n * ((hq + 2 * hk) * dh * D + D * hq * dh + 3 * c * D)
    assert bench.prefill_gemm_flops(wl, n) == wl.n_layers * gemm
    assert bench.prefill_gemm_flops(wl, n) == pytest.approx(6.631e12, rel=1e-3)
    attn = sum(4 * dh * H * (i + 1) for i in range(n)) * wl.n_layers
    assert bench.prefill_attn_flops(wl, n) == attn
    assert attn == pytest.approx(68.85e9, rel=1e-3)
