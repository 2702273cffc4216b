"""Pins the CPU oracle to things other than itself (CPU only, no GPU).

Each test names what fixes the expected value: the IEEE binary16 definition, a closed form, an
invariant the mathematics guarantees, or PyTorch library routines (tests/torch_reference.py).
A plausible slip in the oracle (a dropped eps or gain, a wrong rotation sign or pairing, a wrong
softmax scale, a transposed projection, a wrong GQA head mapping, a misplaced causal limit or
cache position, a residual added twice) fails at least one of them.
"""
from __future__ import annotations

import math
from pathlib import Path

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle
import synthetic
from tests import torch_reference

GOLDEN = Path(__file__).parent / "golden"


def rel(a, b):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300))


def ulps(a16: np.ndarray, b16: np.ndarray) -> int:
    """Largest distance in binary16 units between two finite fp16 arrays of equal sign pattern."""
    ai = a16.view(np.int16).astype(np.int32)
    bi = b16.view(np.int16).astype(np.int32)
    ai = np.where(ai < 0, -32768 - ai, ai)
    bi = np.where(bi < 0, -32768 - bi, bi)
    return int(np.max(np.abs(ai - bi))) if ai.size else 0


# ------------------------------------------------------------------ binary16 ---------------

def _golden_binary16():
    for line in (GOLDEN / "binary16.txt").read_text().splitlines():
        line = line.split("#", 1)[0].strip()
        if not line:
            continue
        val, bits = line.split()
        x = float.fromhex(val) if "0x" in val and "p" in val else float(val)
        yield x, int(bits, 16)


@pytest.mark.parametrize("x,bits", list(_golden_binary16()))
def test_binary16_encode_golden(x, bits):
    assert oracle.f64_to_f16(x) == bits


def test_binary16_decode_all_patterns_match_numpy():
    pats = np.arange(65536, dtype=np.uint32).astype(np.uint16)
    ref = pats.view(np.float16).astype(np.float64)
    got = np.array([oracle.f16_to_f64(int(p)) for p in pats])
    finite = np.isfinite(ref)
    assert np.array_equal(got[finite], ref[finite])
    assert np.array_equal(np.isnan(got), np.isnan(ref))
    assert np.array_equal(got[np.isinf(ref)], ref[np.isinf(ref)])


def test_binary16_encode_matches_numpy_random():
    rng = np.random.default_rng(7)
    xs = np.concatenate([
        rng.standard_normal(4000) * 10.0 ** rng.integers(-9, 5, 4000),
        rng.uniform(-70000, 70000, 1000),
        # exact midpoints between neighbouring fp16 values (ties go to even)
        (np.arange(-3000, 3000).astype(np.float16).astype(np.float64) + 0.5) * 2.0 ** -8,
    ])
    with np.errstate(over="ignore"):
        ref = xs.astype(np.float16).view(np.uint16)
    got = np.array([oracle.f64_to_f16(float(x)) for x in xs], dtype=np.uint16)
    assert np.array_equal(got, ref)


# ------------------------------------------------------------------ RMSNorm ----------------

@pytest.mark.parametrize("c", [3.0, -0.5, 1e-3])
def test_rmsnorm_constant_vector_closed_form(c):
    # mean(x^2) = c^2  =>  y_i = c g_i / sqrt(c^2 + eps) = sign(c) g_i / sqrt(1 + eps / c^2)
    n, eps = 64, 1e-5
    g = synthetic.normal_f16((n,), 11, 1.0, 0.3)
    y = oracle.rmsnorm(np.full(n, c), g, eps)
    expect = math.copysign(1.0, c) * g.astype(np.float64) / math.sqrt(1.0 + eps / c**2)
    assert np.allclose(y, expect, rtol=1e-14, atol=0)


def test_rmsnorm_matches_torch_rms_norm():
    x = np.random.default_rng(3).standard_normal(300) * 4
    g = synthetic.normal_f16((300,), 12, 1.0, 0.02)
    ref = F.rms_norm(torch.tensor(x), (300,), weight=torch.tensor(g.astype(np.float64)), eps=1e-5)
    assert rel(oracle.rmsnorm(x, g, 1e-5), ref.numpy()) < 1e-14


# ------------------------------------------------------------------ RoPE -------------------

def _golden_rope():
    for line in (GOLDEN / "rope_closed_form.txt").read_text().splitlines():
        line = line.split("#", 1)[0].strip()
        if not line:
            continue
        head, vin, vout = [p.split() for p in line.split("|")]
        yield int(head[0]), float(head[1]), int(head[2]), [float(v) for v in vin], [float(v) for v in vout]


@pytest.mark.parametrize("dh,theta,pos,vin,vout", list(_golden_rope()))
def test_rope_closed_forms(dh, theta, pos, vin, vout):
    assert len(vin) == dh
    assert np.allclose(oracle.rope(vin, pos, theta), vout, rtol=0, atol=1e-14)


def test_rope_is_an_isometry_per_pair():
    dh = 128
    v = np.random.default_rng(5).standard_normal(dh)
    for pos in (0, 1, 17, 4095, 100000):
        r = oracle.rope(v, pos, 1e4)
        pn_in = v[:64] ** 2 + v[64:] ** 2
        pn_out = r[:64] ** 2 + r[64:] ** 2
        assert np.allclose(pn_out, pn_in, rtol=1e-12)
    assert np.array_equal(oracle.rope(v, 0, 5e5), v)


def test_rope_scores_depend_only_on_relative_position():
    rng = np.random.default_rng(6)
    q, k = rng.standard_normal(64), rng.standard_normal(64)
    for p, pp in ((5, 2), (300, 7), (4000, 4000)):
        base = oracle.rope(q, p, 1e4) @ oracle.rope(k, pp, 1e4)
        for shift in (1, 33, 1000):
            moved = oracle.rope(q, p + shift, 1e4) @ oracle.rope(k, pp + shift, 1e4)
            assert abs(moved - base) < 1e-10 * max(1.0, abs(base))


# ------------------------------------------------------------------ SwiGLU -----------------

def test_silu_values():
    assert oracle.silu(0.0) == 0.0
    assert abs(oracle.silu(40.0) - 40.0) < 1e-12
    assert abs(oracle.silu(-40.0)) < 1e-15
    zs = np.linspace(-12, 12, 97)
    got = np.array([oracle.silu(z) for z in zs])
    assert rel(got, F.silu(torch.tensor(zs)).numpy()) < 1e-15


# ------------------------------------------------------------------ single-head attention --

def _kv(n, dh, seed, std=1.3):
    return synthetic.normal_f16((n, dh), seed, 0, std), synthetic.normal_f16((n, dh), seed + 1, 0, std)


def test_attention_weights_sum_to_one():
    k, v = _kv(777, 128, 20)
    q = np.random.default_rng(1).standard_normal(128) * 1.3
    w, _ = oracle.attend(q, k, v)
    assert abs(w.sum() - 1.0) < 1e-12 and (w >= 0).all()


def test_attention_single_position_returns_v():
    k, v = _kv(1, 64, 22)
    _, o = oracle.attend(np.ones(64), k, v)
    assert np.array_equal(o, v[0].astype(np.float64))


def test_attention_equal_keys_average_values():
    k, v = _kv(50, 32, 24)
    k[:] = k[0]
    _, o = oracle.attend(np.random.default_rng(2).standard_normal(32), k, v)
    assert np.allclose(o, v.astype(np.float64).mean(0), rtol=1e-12, atol=1e-14)


def test_attention_two_positions_closed_form_scale():
    # w_0 = 1 / (1 + exp((s_1 - s_0)/sqrt(dh))) with s_t = q.k_t
    dh = 16
    k = np.zeros((2, dh), np.float16)
    v = np.zeros((2, dh), np.float16)
    k[0, 0], k[1, 1] = 1.0, 1.0
    v[0, 2], v[1, 3] = 1.0, 1.0
    q = np.zeros(dh)
    q[0], q[1] = 3.0, -1.0
    w, o = oracle.attend(q, k, v)
    w0 = 1.0 / (1.0 + math.exp((-1.0 - 3.0) / math.sqrt(dh)))
    assert abs(w[0] - w0) < 1e-15 and abs(o[2] - w0) < 1e-15 and abs(o[3] - (1 - w0)) < 1e-15


def test_attention_invariant_to_common_key_shift():
    # q.(k_t + c) = q.k_t + q.c for every t: softmax is unchanged by a shift common to all keys.
    dh = 32
    k, v = _kv(40, dh, 26)
    k = (np.round(k.astype(np.float64) * 16) / 16).astype(np.float16)  # multiples of 1/16, |k| < 8
    q = np.random.default_rng(4).standard_normal(dh)
    _, o1 = oracle.attend(q, k, v)
    k2 = (k.astype(np.float64) + 0.25).astype(np.float16)  # exact: fp16 spacing <= 1/128 below 8
    assert np.array_equal(k2.astype(np.float64) - 0.25, k.astype(np.float64))
    _, o2 = oracle.attend(q, k2, v)
    assert rel(o2, o1) < 1e-12


def test_attention_matches_torch_sdpa_single_head():
    k, v = _kv(129, 64, 28)
    q = np.random.default_rng(8).standard_normal(64)
    _, o = oracle.attend(q, k, v)
    ref = F.scaled_dot_product_attention(torch.tensor(q)[None, None, None],
                                         torch.tensor(k.astype(np.float64))[None, None],
                                         torch.tensor(v.astype(np.float64))[None, None])
    assert rel(o, ref.numpy().reshape(-1)) < 1e-13


# ------------------------------------------------------------------ whole layer vs torch ---

def _mini(**kw):
    return synthetic.small(**kw)


@pytest.mark.parametrize("kw", [dict(), dict(n_kv_heads=4), dict(n_heads=6, n_kv_heads=2,
                                head_ranges=((0, 3), (3, 6)), d_model=40, d_ffn=56,
                                ffn_ranges=((0, 56),))])
def test_layer_matches_torch_reference_prefill_then_decode(kw):
    wl = _mini(**kw)
    w = wl.layer_weights(0)
    cap = 16
    kc, vc = oracle.new_cache(wl, cap)
    x = wl.hidden(7)
    full_h = ((0, wl.n_heads),)
    full_f = ((0, wl.d_ffn),)
    h, xn, ap, fp = oracle.tp_layer(wl, w, x, 0, kc, vc, full_h, full_f)
    ref = torch_reference.layer(wl, w, x, 0, None, None)
    assert rel(ap[0], ref["attn_out"]) < 1e-12
    assert np.array_equal(kc[:, :7], ref["k_new"]) and np.array_equal(vc[:, :7], ref["v_new"])
    assert ulps(h, ref["h"]) <= 1
    assert rel(fp[0], oracle.ffn_partial(wl, w, (0, wl.d_ffn), ref["h"])) < 1e-12
    assert rel(oracle.ffn_partial(wl, w, (0, wl.d_ffn), ref["h"]), ref["ffn_out"]) < 1e-12
    assert ulps(xn, ref["x_next"]) <= 1
    # two decode steps that attend to the cache written above
    for step in range(2):
        xd = wl.hidden(1, stream=10 + step)
        pos0 = 7 + step
        kp, vp = kc.copy(), vc.copy()
        h, xn, ap, fp = oracle.tp_layer(wl, w, xd, pos0, kc, vc, full_h, full_f)
        ref = torch_reference.layer(wl, w, xd, pos0, kp, vp)
        assert rel(ap[0], ref["attn_out"]) < 1e-12
        assert np.array_equal(kc[:, pos0:pos0 + 1], ref["k_new"])
        assert ulps(h, ref["h"]) <= 1 and ulps(xn, ref["x_next"]) <= 1


# ------------------------------------------------------------------ TP invariants ----------

PARTITIONS = [
    (((0, 2), (2, 4)), ((0, 25), (25, 40))),
    (((0, 4),), ((0, 40),)),
    (((0, 2), (2, 2), (2, 4)), ((0, 0), (0, 13), (13, 40))),   # empty shards
    (((0, 2), (2, 4)), ((0, 1), (1, 39), (39, 40))),
]


@pytest.mark.parametrize("heads,cols", PARTITIONS)
def test_sum_of_shard_partials_equals_unpartitioned_layer(heads, cols):
    wl = _mini()
    w = wl.layer_weights(1)
    x = wl.hidden(6, stream=3)
    kc1, vc1 = oracle.new_cache(wl, 12)
    kc2, vc2 = oracle.new_cache(wl, 12)
    h1, xn1, ap1, fp1 = oracle.tp_layer(wl, w, x, 0, kc1, vc1, ((0, 4),), ((0, 40),))
    h2, xn2, ap2, fp2 = oracle.tp_layer(wl, w, x, 0, kc2, vc2, heads, cols)
    assert np.array_equal(kc1, kc2) and np.array_equal(vc1, vc2)
    assert rel(sum(ap2), ap1[0]) < 1e-13
    assert ulps(h1, h2) <= 1
    assert rel(sum(fp2), fp1[0]) < 1e-13
    assert ulps(xn1, xn2) <= 1
    for (a, b), p in zip(heads, ap2):
        if a == b:
            assert not p.any()
    for (a, b), p in zip(cols, fp2):
        if a == b:
            assert not p.any()


def test_decode_after_prefill_equals_longer_prefill():
    """Row M of a prefill of M+1 tokens == decoding token M after a prefill of M tokens: pins the
    causal limit, the append position and the RoPE position."""
    wl = _mini()
    w = wl.layer_weights(0)
    x = wl.hidden(9, stream=4)
    kc_a, vc_a = oracle.new_cache(wl, 12)
    h_a, xn_a, ap_a, _ = oracle.tp_layer(wl, w, x, 0, kc_a, vc_a)
    kc_b, vc_b = oracle.new_cache(wl, 12)
    oracle.tp_layer(wl, w, x[:8], 0, kc_b, vc_b)
    h_b, xn_b, ap_b, _ = oracle.tp_layer(wl, w, x[8:], 8, kc_b, vc_b)
    assert np.array_equal(kc_a, kc_b) and np.array_equal(vc_a, vc_b)
    assert rel(sum(ap_b), sum(ap_a)[8:]) < 1e-13
    assert np.array_equal(xn_b, xn_a[8:])


def test_gqa_equals_mha_with_duplicated_kv_heads():
    """Query head h uses KV head h // (H/Hk): the layer equals an MHA layer whose K/V weights are
    the GQA ones repeated per contiguous group."""
    gqa = _mini(n_heads=4, n_kv_heads=2)
    mha = _mini(n_heads=4, n_kv_heads=4)
    w = gqa.layer_weights(0)
    dh = gqa.d_head
    wd = dict(w)
    for name in ("wk", "wv"):
        blocks = w[name].reshape(2, dh, -1)
        wd[name] = np.ascontiguousarray(np.repeat(blocks, 2, axis=0).reshape(4 * dh, -1))
    x = gqa.hidden(5, stream=2)
    kc, vc = oracle.new_cache(gqa, 8)
    _, xn_g, ap_g, _ = oracle.tp_layer(gqa, w, x, 0, kc, vc)
    kc2, vc2 = oracle.new_cache(mha, 8)
    _, xn_m, ap_m, _ = oracle.tp_layer(mha, wd, x, 0, kc2, vc2, head_ranges=((0, 2), (2, 4)))
    assert rel(sum(ap_g), sum(ap_m)) < 1e-13
    assert ulps(xn_g, xn_m) <= 1


def test_combine_adds_residual_once_in_shard_order():
    parts = [np.full(4, 0.5), np.full(4, 0.25), np.full(4, -1.0)]
    res = np.array([1, 2, 3, 4], np.float16)
    out = oracle.combine(parts, res)
    assert np.array_equal(out, np.array([0.75, 1.75, 2.75, 3.75], np.float16))
    assert np.array_equal(oracle.combine(parts, None), np.full(4, -0.25, np.float16))


def test_argument_checks():
    wl = _mini()
    w = wl.layer_weights(0)
    kc, vc = oracle.new_cache(wl, 4)
    with pytest.raises(ValueError):
        oracle.kv_append(wl, w, (0, 2), wl.hidden(5), 0, kc, vc)   # beyond capacity
    with pytest.raises(ValueError):
        oracle.attn_partial(wl, w, (0, 5), wl.hidden(1), [0], kc, vc)  # head range beyond H
    with pytest.raises(ValueError):
        oracle.ffn_partial(wl, w, (3, 2), wl.hidden(1))
