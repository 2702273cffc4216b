"""Per-layer partitions (vt_partition_create_layers: layer-wise MP / TP, Section 4.2.1), pruned
shards (VT_PARTITION_PRUNE, Section 4.3.1) and quantized partials (communication scaling, Section
4.3.2) on the GPU, against the oracle: the oracle's layer with each layer's own ranges (pruned
heads / columns omitted), and its block quantizer and combine of quantized partials.
"""
from __future__ import annotations

import numpy as np
import pytest

import oracle
import synthetic
from tests.parity import assert_close, shapes_of

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

ATTN, FFN = 0, 1


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def host(t):
    torch.cuda.synchronize()
    return t.detach().cpu().numpy()


WL = synthetic.small("layers", n_layers=3, d_model=512, n_heads=8, n_kv_heads=4, d_head=64, d_ffn=1408,
                     head_ranges=((0, 2), (2, 6), (6, 8)), ffn_ranges=((0, 701), (701, 1000), (1000, 1408)),
                     kv_len=30, decode_steps=3, prompt_len=100, model_id=140)

# layer 0: TP 3-way (uneven); layer 1: MP on device 2 (ATTN) and device 0 (FFN); layer 2: 2-way TP
PER_LAYER = ([[(0, 2), (2, 6), (6, 8)], [(0, 0), (0, 0), (0, 8)], [(0, 4), (4, 8), (8, 8)]],
             [[(0, 701), (701, 1000), (1000, 1408)], [(0, 1408), (1408, 1408), (1408, 1408)],
              [(0, 0), (0, 704), (704, 1408)]])
# pruned: layer 0 drops heads [2, 4) and columns [100, 300); layer 1 drops device 1's shards;
# layer 2 drops the last KV group and the last 8 columns
PRUNED = ([[(0, 2), (4, 6), (6, 8)], [(0, 2), (2, 2), (6, 8)], [(0, 4), (4, 6), (6, 6)]],
          [[(0, 100), (300, 1000), (1000, 1408)], [(0, 701), (701, 701), (1000, 1408)], [(0, 700), (700, 1000), (1000, 1400)]])


def _stack(vt, wl, cap, layer_ranges=None):
    from paper_2607_07046_gb300.stack import Stack
    shapes = shapes_of(vt, wl, max_seq=max(wl.max_seq, cap))
    return Stack(shapes, wl.layer_weights, wl.head_ranges, wl.ffn_ranges, cap, layer_ranges=layer_ranges)


def _reference_tokens(wl, heads, cols, L0, xs, caches):
    ws = [wl.layer_weights(l) for l in range(wl.n_layers)]
    outs = []
    for t, x in enumerate(xs):
        r = x.reshape(1, -1)
        for l in range(wl.n_layers):
            _, r, _, _ = oracle.tp_layer(wl, ws[l], r, L0 + t, *caches[l], heads[l], cols[l])
        outs.append(r.reshape(-1))
    return outs


@pytest.mark.parametrize("name,table,flags", [("per-layer", PER_LAYER, 0), ("pruned", PRUNED, 1)])
def test_decode_tokens_per_layer_table(vtlib, name, table, flags):
    vt = vtlib
    wl = WL
    heads, cols = table
    L0, steps, cap = 30, 3, 40
    caches = [wl.kv_fill(l, L0, cap) for l in range(wl.n_layers)]
    xs = [wl.hidden(1, stream=400 + t) for t in range(steps)]
    ref = _reference_tokens(wl, heads, cols, L0, xs, [(k.copy(), v.copy()) for k, v in caches])
    with _stack(vt, wl, cap, (heads, cols, flags)) as st:
        fused = vt.vt_decode_token_fused_available(st.part)
        assert not fused[0] and ("per-layer" in fused[1] or "pruned" in fused[1])
        g = wl.n_heads // wl.n_kv_heads
        for l in range(wl.n_layers):
            for d, (h0, h1) in enumerate(heads[l]):
                if h1 > h0:
                    vt.vt_kv_write_raw(st.kv, l, d, caches[l][0][h0 // g:h1 // g, :L0], caches[l][1][h0 // g:h1 // g, :L0])
        vt.vt_kv_set_length(st.kv, -1, L0)
        y = torch.empty(wl.d_model, dtype=torch.float16, device="cuda")
        for t in range(steps):
            vt.vt_decode_token(st.part, st.kv, dev(xs[t].reshape(-1)), y)
            assert_close(host(y), ref[t], f"{name} token {t}")
        assert vt.vt_kv_status(st.kv) == 0 and vt.vt_partition_status(st.part) == 0


@pytest.mark.parametrize("name,table,flags", [("per-layer", PER_LAYER, 0), ("pruned", PRUNED, 1)])
def test_prefill_tokens_per_layer_table(vtlib, name, table, flags):
    vt = vtlib
    wl = WL
    heads, cols = table
    n, cap = 100, 104
    X = wl.hidden(n, stream=410)
    ws = [wl.layer_weights(l) for l in range(wl.n_layers)]
    ref = X
    for l in range(wl.n_layers):
        kc, vc = oracle.new_cache(wl, cap)
        _, ref, _, _ = oracle.tp_layer(wl, ws[l], ref, 0, kc, vc, heads[l], cols[l])
    with _stack(vt, wl, cap, (heads, cols, flags)) as st:
        out = torch.empty((n, wl.d_model), dtype=torch.float16, device="cuda")
        vt.vt_prefill_tokens(st.part, st.kv, dev(X), n, out)
        assert_close(host(out), ref, f"{name} prefill")
        assert vt.vt_kv_status(st.kv) == 0 and vt.vt_partition_status(st.part) == 0


# ------------------------------------------------------------------ communication scaling

@pytest.mark.parametrize("bits,n", [(8, 4096), (4, 4096), (8, 1000), (4, 1001)])
def test_quantize_partial_equals_the_oracle(vtlib, bits, n):
    """Codes and scales of a seeded fp32 partial equal or_quantize_vec bit for bit (ragged last
    block included); the combine of such partials matches or_combine_q."""
    vt = vtlib
    rng = np.random.default_rng(bits * 1000 + n)
    parts = [(rng.standard_normal(n) * s).astype(np.float32) for s in (0.5, 2.0, 0.01)]
    parts[1][:32] = 0.0  # an all-zero block: scale 0, codes 0
    nb = (n + 31) // 32
    cb = vt.vt_partial_code_bytes(n, bits)
    codes_d, scales_d = [], []
    for p in parts:
        c = torch.empty(cb, dtype=torch.uint8, device="cuda")
        s_ = torch.empty(nb, dtype=torch.float16, device="cuda")
        vt.vt_quantize_partial(dev(p), bits, c, s_)
        codes_d.append(c)
        scales_d.append(s_)
        q_ref, s_ref = oracle.quantize_vec(p, bits)
        raw = host(c)
        if bits == 8:
            q = raw.view(np.int8)
        else:
            q = np.empty(n, np.int8)
            q[0::2] = (raw & 15).astype(np.int8)[: (n + 1) // 2] - 8
            q[1::2] = (raw >> 4).astype(np.int8)[: n // 2] - 8
        assert np.array_equal(q, q_ref)
        assert np.array_equal(host(s_).view(np.uint16), s_ref.view(np.uint16))
    residual = synthetic.normal_f16((n,), 7, 0.0, 1.0)
    out = torch.empty(n, dtype=torch.float16, device="cuda")
    vt.vt_combine_q(codes_d, scales_d, bits, dev(residual), out)
    ref = oracle.combine_q([oracle.quantize_vec(p, bits) for p in parts], residual)
    assert_close(host(out), ref, f"combine_q {bits}-bit")


@pytest.mark.parametrize("bits", [8, 4])
def test_whole_token_with_quantized_partials(vtlib, bits):
    """vt_decode_token with every device's partials quantized before the combine (the per-shard
    kernels, each partial quantized as its shard finishes): the token's h and x_next equal the
    oracle's combine of the quantized fp32 partials, the partials themselves taken from the oracle
    (teacher-forced per block).  Both sides quantize fp32 partials that agree to fp32 rounding, so a
    code can differ only where a value sits on a rounding boundary; with these seeds none does."""
    vt = vtlib
    wl = synthetic.small("comm", n_layers=1, d_model=512, n_heads=8, n_kv_heads=8, d_head=64, d_ffn=1408,
                         head_ranges=((0, 4), (4, 8)), ffn_ranges=((0, 704), (704, 1408)),
                         kv_len=20, decode_steps=1, prompt_len=0, model_id=141)
    w = wl.layer_weights(0)
    L0, cap = 20, 24
    kc, vc = wl.kv_fill(0, L0, cap)
    x = wl.hidden(1, stream=420)
    h_ref, ap = oracle.tp_attention(wl, w, x, L0, kc, vc)
    _, fp = oracle.tp_ffn(wl, w, h_ref)
    with _stack(vt, wl, cap) as st:
        vt.vt_partition_set_comm_bits(st.part, -1, bits)
        assert not vt.vt_decode_token_fused_available(st.part)[0]
        for d, (h0, h1) in enumerate(wl.head_ranges):
            vt.vt_kv_write_raw(st.kv, 0, d, kc[h0:h1, :L0], vc[h0:h1, :L0])
        vt.vt_kv_set_length(st.kv, -1, L0)
        y = torch.empty(wl.d_model, dtype=torch.float16, device="cuda")
        vt.vt_decode_token(st.part, st.kv, dev(x.reshape(-1)), y)
        got = host(y)
        # reference: h from the oracle's quantized ATTN partials, then its FFN on that h with
        # quantized FFN partials
        hq = oracle.combine_q([oracle.quantize_vec(p.reshape(-1).astype(np.float32), bits) for p in ap], x.reshape(-1))
        _, fq = oracle.tp_ffn(wl, w, hq.reshape(1, -1))
        xq = oracle.combine_q([oracle.quantize_vec(p.reshape(-1).astype(np.float32), bits) for p in fq], hq)
        assert_close(got, xq, f"{bits}-bit partials token")
        # back to fp32 partials: the fused kernel is available again
        vt.vt_partition_set_comm_bits(st.part, -1, 16)
        assert vt.vt_decode_token_fused_available(st.part)[0]
