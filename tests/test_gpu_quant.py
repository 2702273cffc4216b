"""Mixed-precision shards on the GPU (vt_partition_set_precision): the library's INT8 / INT4 codes
and scales equal the oracle's quantizer bit for bit (including ragged last blocks), and decode
through quantized shards matches the oracle's quantized-shard layer (or_attn_partial_q,
or_ffn_partial_q, or_kv_append_q) within the parity tolerance, per shard and for whole tokens with
shards at different precisions.
"""
from __future__ import annotations

import dataclasses

import numpy as np
import pytest

import oracle
import synthetic
from tests.parity import assert_close, kv_range, shapes_of

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

ATTN, FFN = 0, 1


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def host(t):
    torch.cuda.synchronize()
    return t.detach().cpu().numpy()


def stack(vt, wl, capacity, precision=None, layer_ids=None, windows=None):
    from paper_2607_07046_gb300.stack import Stack
    layer_ids = list(range(wl.n_layers)) if layer_ids is None else list(layer_ids)
    shapes = shapes_of(vt, wl, max_seq=max(wl.max_seq, capacity))
    shapes.n_layers = len(layer_ids)
    return Stack(shapes, lambda i: wl.layer_weights(layer_ids[i]), wl.head_ranges, wl.ffn_ranges, capacity,
                 precision=precision, windows=windows)


UNEVEN = synthetic.small("quant-uneven", n_layers=2, d_model=512, n_heads=8, n_kv_heads=4, d_head=64, d_ffn=1408,
                         head_ranges=((0, 2), (2, 6), (6, 8)), ffn_ranges=((0, 701), (701, 1000), (1000, 1408)),
                         kv_len=40, decode_steps=2, prompt_len=0, model_id=130)


@pytest.mark.parametrize("bits", [8, 4])
def test_codes_and_scales_equal_the_oracle_quantizer(vtlib, bits):
    """Every quantized tensor of every shard (QKV rows in the shard's RoPE-pair order, O columns,
    interleaved gate/up rows, the down columns; FFN widths 701 / 299 / 408 leave ragged blocks)."""
    vt = vtlib
    wl = UNEVEN
    w = wl.layer_weights(1)
    D, dh = wl.d_model, wl.d_head
    with stack(vt, wl, 0, layer_ids=[1]) as st:
        fp16 = {}
        for d in range(3):
            fp16[(d, 1)] = vt.vt_shard_weights_read(st.part, (0, d, ATTN), 1)
            fp16[(d, 2)] = vt.vt_shard_weights_read(st.part, (0, d, ATTN), 2)
            fp16[(d, 4)] = vt.vt_shard_weights_read(st.part, (0, d, FFN), 4)
        for d in range(3):
            vt.vt_partition_set_precision(st.part, (0, d, ATTN), bits)
            vt.vt_partition_set_precision(st.part, (0, d, FFN), bits)
            assert vt.vt_shard_precision(st.part, (0, d, ATTN)) == bits
        for d, ((h0, h1), (c0, c1)) in enumerate(zip(wl.head_ranges, wl.ffn_ranges)):
            hk = (h1 - h0) // (wl.n_heads // wl.n_kv_heads)
            c = c1 - c0
            cases = [(ATTN, 1, fp16[(d, 1)], (h1 - h0 + 2 * hk) * dh, D),
                     (ATTN, 2, fp16[(d, 2)], D, (h1 - h0) * dh),
                     (FFN, 4, fp16[(d, 4)], 2 * c, D),
                     (FFN, 5, np.ascontiguousarray(w["w_down"][:, c0:c1]), D, c)]
            for blk, which, src, rows, k in cases:
                q_ref, s_ref = oracle.quantize_rows(np.ascontiguousarray(src), bits)
                q, sc = vt.vt_shard_qweights_read(st.part, (0, d, blk), which, rows, k)
                assert np.array_equal(q, q_ref), (d, which)
                assert np.array_equal(sc.view(np.uint16), s_ref.view(np.uint16)), (d, which)
                with pytest.raises(vt.VtError) as e:
                    vt.vt_shard_weights_read(st.part, (0, d, blk), which)
                assert e.value.status == vt.VT_ERR_STATE


def _shard_checks(vt, st, wl, w, layer, x, L, kc, vc, attn_bits, ffn_bits, tag, window=0):
    """Every shard's decode partial (vt_decode_step) against the oracle's quantized shard."""
    D = wl.d_model
    qws = [oracle.shard_qweights(wl, w, hr, cr, ab, fb)
           for hr, cr, ab, fb in zip(wl.head_ranges, wl.ffn_ranges, attn_bits, ffn_bits)]
    parts = [torch.empty(D, dtype=torch.float32, device="cuda") for _ in wl.head_ranges]
    for d in range(len(wl.head_ranges)):
        vt.vt_decode_step(st.part, (layer, d, ATTN), dev(x.reshape(D)), st.kv, parts[d])
    h_ref, _, ap, _ = oracle.tp_layer_mixed(wl, w, x, L, kc, vc, attn_bits, [16] * len(ffn_bits), window)
    for d in range(len(wl.head_ranges)):
        assert_close(host(parts[d]), ap[d], f"{tag} ATTN partial dev {d} ({attn_bits[d]} bits)")
    for d, hr in enumerate(wl.head_ranges):
        k0, k1 = kv_range(wl, hr)
        if k1 > k0:
            kg, vg = vt.vt_kv_read(st.kv, layer, d, L + 1, k1 - k0, wl.d_head)
            assert_close(kg[:, L], kc[k0:k1, L], f"{tag} k append dev {d}")
            assert_close(vg[:, L], vc[k0:k1, L], f"{tag} v append dev {d}")
    fparts = [torch.empty(D, dtype=torch.float32, device="cuda") for _ in wl.ffn_ranges]
    hin = dev(h_ref.reshape(D))
    for d in range(len(wl.ffn_ranges)):
        vt.vt_decode_step(st.part, (layer, d, FFN), hin, None, fparts[d])
    for d, (cr, fb) in enumerate(zip(wl.ffn_ranges, ffn_bits)):
        ref = oracle.ffn_partial(wl, w, cr, h_ref) if fb == 16 else oracle.ffn_partial_q(wl, w, cr, h_ref, qws[d])
        assert_close(host(fparts[d]), ref, f"{tag} FFN partial dev {d} ({fb} bits)")


@pytest.mark.parametrize("attn_bits,ffn_bits", [([8, 8, 8], [8, 8, 8]), ([4, 4, 4], [4, 4, 4]),
                                                ([8, 16, 4], [4, 8, 16])])
def test_decode_step_quantized_shards(vtlib, attn_bits, ffn_bits):
    vt = vtlib
    wl = UNEVEN
    layer, L, cap = 1, 40, 48
    w = wl.layer_weights(layer)
    kc, vc = wl.kv_fill(layer, L, cap)
    prec = lambda l, d, b: (attn_bits if b == ATTN else ffn_bits)[d]
    with stack(vt, wl, cap, precision=prec, layer_ids=[layer]) as st:
        fused = vt.vt_decode_token_fused_available(st.part)
        assert not fused[0] and "quantized" in fused[1]
        for d, hr in enumerate(wl.head_ranges):
            k0, k1 = kv_range(wl, hr)
            vt.vt_kv_write_raw(st.kv, 0, d, kc[k0:k1, :L], vc[k0:k1, :L])
        vt.vt_kv_set_length(st.kv, 0, L)
        _shard_checks(vt, st, wl, w, 0, wl.hidden(1, stream=300), L, kc, vc, attn_bits, ffn_bits, "uneven")
        assert vt.vt_kv_status(st.kv) == 0 and vt.vt_partition_status(st.part) == 0


def test_static_step_quantized_attention_shard(vtlib):
    vt = vtlib
    wl = UNEVEN
    layer, L, cap = 0, 40, 48
    w = wl.layer_weights(layer)
    kc, vc = wl.kv_fill(layer, L, cap)
    with stack(vt, wl, cap, precision=lambda l, d, b: 4 if b == ATTN else 16, layer_ids=[layer]) as st:
        for d, hr in enumerate(wl.head_ranges):
            k0, k1 = kv_range(wl, hr)
            vt.vt_kv_write_raw(st.kv, 0, d, kc[k0:k1, :L], vc[k0:k1, :L])
        vt.vt_kv_set_length(st.kv, 0, L)
        x = wl.hidden(1, stream=301)
        part = torch.empty(wl.d_model, dtype=torch.float32, device="cuda")
        vt.vt_decode_step_static(st.part, (0, 1, ATTN), dev(x.reshape(-1)), st.kv, part)
        _, _, ap, _ = oracle.tp_layer_mixed(wl, w, x, L, kc, vc, [4, 4, 4], [16, 16, 16])
        assert_close(host(part), ap[1], "static step, INT4 shard")


@pytest.mark.parametrize("cid,bits", [(2, 8), (2, 4), (5, 4), (3, 8)])
def test_full_size_layer_quantized(vtlib, cid, bits):
    """One full-width layer (7B 4-way, 8B GQA, 13B uneven 3-way with FFN widths 6912 / 4147 /
    2765) at the workload's KV length, every shard at `bits`."""
    vt = vtlib
    wl = synthetic.WORKLOADS[cid]
    layer, L = wl.n_layers - 1, wl.kv_len
    cap = L + 8
    w = wl.layer_weights(layer)
    kc, vc = wl.kv_fill(layer, L, cap)
    n = len(wl.head_ranges)
    with stack(vt, wl, cap, precision=lambda l, d, b: bits, layer_ids=[layer]) as st:
        for d, hr in enumerate(wl.head_ranges):
            k0, k1 = kv_range(wl, hr)
            vt.vt_kv_write_raw(st.kv, 0, d, kc[k0:k1, :L], vc[k0:k1, :L])
        vt.vt_kv_set_length(st.kv, 0, L)
        _shard_checks(vt, st, wl, w, 0, wl.hidden(1, stream=310 + cid), L, kc, vc, [bits] * n, [bits] * n,
                      f"{wl.name} {bits}-bit")
        assert vt.vt_kv_status(st.kv) == 0


def test_whole_tokens_mixed_precision_per_layer(vtlib):
    """Two layers whose shards run at different precisions per layer and device (the per-layer
    allocation of Section 4.2.2), three tokens through vt_decode_token (per-shard kernels), against
    the oracle chained through the same mixed layers."""
    vt = vtlib
    wl = UNEVEN
    bits = {(0, ATTN): [8, 4, 16], (0, FFN): [16, 8, 4], (1, ATTN): [4, 8, 8], (1, FFN): [8, 16, 4]}
    L0, steps, cap = 40, 3, 48
    ws = [wl.layer_weights(l) for l in range(2)]
    caches = [wl.kv_fill(l, L0, cap) for l in range(2)]
    with stack(vt, wl, cap, precision=lambda l, d, b: bits[(l, b)][d]) as st:
        for l in range(2):
            for d, hr in enumerate(wl.head_ranges):
                k0, k1 = kv_range(wl, hr)
                vt.vt_kv_write_raw(st.kv, l, d, caches[l][0][k0:k1, :L0], caches[l][1][k0:k1, :L0])
        vt.vt_kv_set_length(st.kv, -1, L0)
        y = torch.empty(wl.d_model, dtype=torch.float16, device="cuda")
        for t in range(steps):
            x = wl.hidden(1, stream=320 + t)
            vt.vt_decode_token(st.part, st.kv, dev(x.reshape(-1)), y)
            r = x.reshape(1, -1)
            for l in range(2):
                _, r, _, _ = oracle.tp_layer_mixed(wl, ws[l], r, L0 + t, *caches[l], bits[(l, ATTN)], bits[(l, FFN)])
            assert_close(host(y), r.reshape(-1), f"mixed-precision token {t}")
        assert vt.vt_kv_status(st.kv) == 0


def test_planned_precisions_run_and_match_the_oracle(vtlib):
    """The precision plan of Section 4.2.2 applied end to end: seeded importance scores per block
    and a memory budget between the all-fp16 and all-INT4 footprints give vt_plan_precision's bits
    per block; the stack built with them decodes two tokens that equal the oracle's layers at the
    same precisions, and the blocks left at fp16 are the most important ones."""
    vt = vtlib
    wl = UNEVEN
    L0, steps, cap = 40, 2, 48
    sh = shapes_of(vt, wl, max_seq=max(wl.max_seq, cap))
    plans = [dict(ranges=list(wl.head_ranges), comm_s=0.0) if b % 2 == 0 else dict(ranges=list(wl.ffn_ranges), comm_s=0.0)
             for b in range(2 * wl.n_layers)]
    importance = list(np.random.default_rng(5).normal(size=2 * wl.n_layers))
    rate = [1e9] * len(wl.head_ranges)
    full, _, _ = vt.vt_plan_precision(sh, plans, importance, rate)
    assert full == [16] * 4
    # device 1 holds the most: a budget of 60% of its fp16 footprint forces several steps
    fp16_mem = []
    for d in range(len(rate)):
        h = wl.head_ranges[d][1] - wl.head_ranges[d][0]
        c = wl.ffn_ranges[d][1] - wl.ffn_ranges[d][0]
        hk = h // (wl.n_heads // wl.n_kv_heads)
        attn = 2 * ((h + 2 * hk) * wl.d_head * wl.d_model + wl.d_model * h * wl.d_head) + 4 * hk * sh.max_seq * wl.d_head
        fp16_mem.append(wl.n_layers * (attn + 2 * 3 * wl.d_model * c))
    budget = [m * 0.6 for m in fp16_mem]
    bits, k, _ = vt.vt_plan_precision(sh, plans, importance, rate, mem_bytes=budget)
    assert 0 < k < 4 * wl.n_layers and any(b != 16 for b in bits)
    kept = [b for b in range(4) if bits[b] == 16]
    lowered = [b for b in range(4) if bits[b] != 16]
    if kept:
        assert min(importance[b] for b in kept) >= max(importance[b] for b in lowered)
    ws = [wl.layer_weights(l) for l in range(2)]
    caches = [wl.kv_fill(l, L0, cap) for l in range(2)]
    n = len(rate)
    with stack(vt, wl, cap, precision=lambda l, d, b: bits[2 * l + b]) as st:
        for l in range(2):
            for d, hr in enumerate(wl.head_ranges):
                k0, k1 = kv_range(wl, hr)
                vt.vt_kv_write_raw(st.kv, l, d, caches[l][0][k0:k1, :L0], caches[l][1][k0:k1, :L0])
        vt.vt_kv_set_length(st.kv, -1, L0)
        y = torch.empty(wl.d_model, dtype=torch.float16, device="cuda")
        for t in range(steps):
            x = wl.hidden(1, stream=330 + t)
            vt.vt_decode_token(st.part, st.kv, dev(x.reshape(-1)), y)
            r = x.reshape(1, -1)
            for l in range(2):
                _, r, _, _ = oracle.tp_layer_mixed(wl, ws[l], r, L0 + t, *caches[l], [bits[2 * l]] * n,
                                                   [bits[2 * l + 1]] * n)
            assert_close(host(y), r.reshape(-1), f"planned-precision token {t}")
        assert vt.vt_kv_status(st.kv) == 0


def test_precision_api_rules(vtlib):
    vt = vtlib
    wl = dataclasses.replace(UNEVEN, n_layers=1)
    with stack(vt, wl, 0) as st:
        with pytest.raises(vt.VtError) as e:
            vt.vt_partition_set_precision(st.part, (0, 0, ATTN), 6)
        assert e.value.status == vt.VT_ERR_INVALID_ARG
        vt.vt_partition_set_precision(st.part, (0, 0, FFN), 4)
        x = torch.zeros((4, wl.d_model), dtype=torch.float16, device="cuda")
        out = torch.empty((4, wl.d_model), dtype=torch.float32, device="cuda")
        with pytest.raises(vt.VtError) as e:
            vt.vt_prefill(st.part, (0, 0, FFN), x, 4, None, out)
        assert e.value.status == vt.VT_ERR_STATE
        # back to fp16: the slices equal a fresh partition's, bit for bit
        vt.vt_partition_set_precision(st.part, (0, 0, FFN), 16)
        assert vt.vt_shard_precision(st.part, (0, 0, FFN)) == 16
        fresh = vt.vt_partition_create(st.model, wl.head_ranges, wl.ffn_ranges)
        try:
            for which in (4, 5):
                assert np.array_equal(vt.vt_shard_weights_read(st.part, (0, 0, FFN), which),
                                      vt.vt_shard_weights_read(fresh, (0, 0, FFN), which))
        finally:
            vt.vt_partition_destroy(fresh)
        kv = vt.vt_kv_create(st.part, 16)
        try:
            with pytest.raises(vt.VtError) as e:
                vt.vt_partition_set_precision(st.part, (0, 1, ATTN), 8)
            assert e.value.status == vt.VT_ERR_STATE
        finally:
            vt.vt_kv_destroy(kv)
        vt.vt_partition_set_precision(st.part, (0, 1, ATTN), 8)
