"""Decode path on the GPU (through the C ABI) against the CPU oracle, element by element.

Every comparison uses the tolerance in tests/parity.py (rel-RMS <= 1e-3, max-abs <= 2e-2 per
tensor); weight slicing and KV-cache indexing are compared bit for bit.
"""
from __future__ import annotations

import numpy as np
import pytest

import oracle
import synthetic
from tests.parity import assert_close, kv_range, shapes_of

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

ATTN, FFN = 0, 1


def dev(a, dtype=None):
    t = torch.from_numpy(np.ascontiguousarray(a)).cuda()
    return t if dtype is None else t.to(dtype)


def host(t):
    torch.cuda.synchronize()
    return t.detach().cpu().numpy()


def build(vt, wl, layer_ids=None, capacity=None, ranges=None):
    """A Stack holding layers `layer_ids` of the workload's model (default: all)."""
    from paper_2607_07046_gb300.stack import Stack
    layer_ids = list(range(wl.n_layers)) if layer_ids is None else list(layer_ids)
    capacity = wl.max_seq if capacity is None else capacity
    shapes = shapes_of(vt, wl, max_seq=max(wl.max_seq, capacity))
    shapes.n_layers = len(layer_ids)
    heads, cols = ranges if ranges is not None else (wl.head_ranges, wl.ffn_ranges)
    return Stack(shapes, lambda i: wl.layer_weights(layer_ids[i]), heads, cols, capacity)


def write_cache(vt, st, layer, wl, kc, vc, n_pos, heads):
    for d, hr in enumerate(heads):
        k0, k1 = kv_range(wl, hr)
        if k1 > k0:
            vt.vt_kv_write_raw(st.kv, layer, d, kc[k0:k1, :n_pos], vc[k0:k1, :n_pos])


def decode_layer_check(vt, st, wl, w, layer, x, L, kc, vc, heads, cols, tag=""):
    """One decode token through layer `layer` of `st` (all shards + both combines) vs the oracle,
    teacher-forced (the FFN block gets the oracle's h).  kc/vc: full-layer oracle caches with L
    positions; they are extended in place by the oracle."""
    D = wl.d_model
    xg = dev(x.reshape(D))
    parts = [torch.empty(D, dtype=torch.float32, device="cuda") for _ in heads]
    for d in range(len(heads)):
        vt.vt_decode_step(st.part, (layer, d, ATTN), xg, st.kv, parts[d])
    hg = torch.empty(D, dtype=torch.float16, device="cuda")
    vt.vt_combine(parts, xg, hg, 1, D)
    h_ref, ap = oracle.tp_attention(wl, w, x.reshape(1, D), L, kc, vc, heads)
    for d in range(len(heads)):
        assert_close(host(parts[d]), ap[d], f"{tag} attn partial dev {d}")
    assert_close(host(hg), h_ref, f"{tag} h")
    # the appended K/V row and untouched earlier rows
    for d, hr in enumerate(heads):
        k0, k1 = kv_range(wl, hr)
        if k1 == k0:
            continue
        kg, vg = vt.vt_kv_read(st.kv, layer, d, L + 1, k1 - k0, wl.d_head)
        assert np.array_equal(kg[:, :L], kc[k0:k1, :L]) and np.array_equal(vg[:, :L], vc[k0:k1, :L])
        assert_close(kg[:, L], kc[k0:k1, L], f"{tag} k append dev {d}")
        assert_close(vg[:, L], vc[k0:k1, L], f"{tag} v append dev {d}")
    hgi = dev(h_ref.reshape(D))
    fparts = [torch.empty(D, dtype=torch.float32, device="cuda") for _ in cols]
    for d in range(len(cols)):
        vt.vt_decode_step(st.part, (layer, d, FFN), hgi, None, fparts[d])
    xn = torch.empty(D, dtype=torch.float16, device="cuda")
    vt.vt_combine(fparts, hgi, xn, 1, D)
    xn_ref, fp = oracle.tp_ffn(wl, w, h_ref, cols)
    for d in range(len(cols)):
        assert_close(host(fparts[d]), fp[d], f"{tag} ffn partial dev {d}")
    assert_close(host(xn), xn_ref, f"{tag} x_next")


# ------------------------------------------------------------------ tiny config (config 1)

def test_tiny_layer_decode_after_128_token_prefill(vtlib):
    """Hidden 512, 8 heads x 64, FFN 1408, 2-way; KV cache = oracle prefill of 128 seeded tokens."""
    wl = synthetic.WORKLOADS[1]
    w = wl.layer_weights(0)
    kc, vc = oracle.new_cache(wl, wl.max_seq)
    oracle.tp_layer(wl, w, wl.hidden(wl.kv_len, stream=1), 0, kc, vc)
    with build(vtlib, wl) as st:
        write_cache(vtlib, st, 0, wl, kc, vc, wl.kv_len, wl.head_ranges)
        vtlib.vt_kv_set_length(st.kv, 0, wl.kv_len)
        decode_layer_check(vtlib, st, wl, w, 0, wl.hidden(1, stream=2), wl.kv_len, kc, vc,
                           wl.head_ranges, wl.ffn_ranges, "tiny")
        assert vtlib.vt_kv_status(st.kv) == 0 and vtlib.vt_partition_status(st.part) == 0


@pytest.mark.parametrize("L", [0, 1, 2, 31, 32, 33, 95, 127, 129, 200])
def test_decode_kv_lengths_and_ragged_tiles(vtlib, L):
    wl = synthetic.WORKLOADS[1]
    w = wl.layer_weights(0)
    cap = 256
    kc, vc = wl.kv_fill(0, L, cap) if L > 0 else oracle.new_cache(wl, cap)
    with build(vtlib, wl, capacity=cap) as st:
        write_cache(vtlib, st, 0, wl, kc, vc, L, wl.head_ranges)
        vtlib.vt_kv_set_length(st.kv, 0, L)
        decode_layer_check(vtlib, st, wl, w, 0, wl.hidden(1, stream=3 + L), L, kc, vc,
                           wl.head_ranges, wl.ffn_ranges, f"L={L}")


UNEVEN = [
    # (heads, kv heads, head ranges, ffn ranges)
    (8, 8, ((0, 1), (1, 4), (4, 8)), ((0, 701), (701, 1000), (1000, 1408))),
    (8, 8, ((0, 8), (8, 8)), ((0, 0), (0, 1408))),            # an empty shard of each kind
    (8, 4, ((0, 2), (2, 8)), ((0, 9), (9, 1408))),            # GQA group 2
    (8, 2, ((0, 4), (4, 8)), ((0, 704), (704, 1408))),        # GQA group 4
    (8, 1, ((0, 8),), ((0, 1408),)),                          # GQA group 8 (MQA), 1-way
]


@pytest.mark.parametrize("H,Hk,heads,cols", UNEVEN)
def test_decode_uneven_and_gqa_partitions(vtlib, H, Hk, heads, cols):
    wl = synthetic.small("uneven", n_layers=1, d_model=512, n_heads=H, n_kv_heads=Hk, d_head=64,
                         d_ffn=1408, head_ranges=heads, ffn_ranges=cols, kv_len=77, decode_steps=1,
                         prompt_len=0, model_id=91)
    w = wl.layer_weights(0)
    cap = 96
    kc, vc = wl.kv_fill(0, 77, cap)
    with build(vtlib, wl, capacity=cap) as st:
        write_cache(vtlib, st, 0, wl, kc, vc, 77, heads)
        vtlib.vt_kv_set_length(st.kv, 0, 77)
        decode_layer_check(vtlib, st, wl, w, 0, wl.hidden(1, stream=5), 77, kc, vc, heads, cols,
                           f"H={H} Hk={Hk}")


def test_decode_head_dim_128_gqa_4(vtlib):
    wl = synthetic.small("dh128", n_layers=1, d_model=1024, n_heads=8, n_kv_heads=2, d_head=128,
                         d_ffn=2752, head_ranges=((0, 4), (4, 8)), ffn_ranges=((0, 1376), (1376, 2752)),
                         kv_len=300, decode_steps=1, prompt_len=0, model_id=92, rope_theta=5e5)
    w = wl.layer_weights(0)
    kc, vc = wl.kv_fill(0, 300, 320)
    with build(vtlib, wl, capacity=320) as st:
        write_cache(vtlib, st, 0, wl, kc, vc, 300, wl.head_ranges)
        vtlib.vt_kv_set_length(st.kv, 0, 300)
        decode_layer_check(vtlib, st, wl, w, 0, wl.hidden(1, stream=6), 300, kc, vc,
                           wl.head_ranges, wl.ffn_ranges, "dh128")


# ------------------------------------------------------------------ bit-exact bookkeeping

def test_shard_weights_are_exact_slices(vtlib):
    wl = synthetic.small("slices", n_layers=2, d_model=256, n_heads=4, n_kv_heads=2, d_head=64,
                         d_ffn=300, head_ranges=((0, 2), (2, 4)), ffn_ranges=((0, 101), (101, 300)),
                         model_id=93)
    dh, half = wl.d_head, wl.d_head // 2
    with build(vtlib, wl, capacity=8) as st:
        for l in range(2):
            w = wl.layer_weights(l)
            for d, (hr, cr) in enumerate(zip(wl.head_ranges, wl.ffn_ranges)):
                k0, k1 = kv_range(wl, hr)
                blocks = [w["wq"][h * dh:(h + 1) * dh] for h in range(*hr)]
                blocks += [w["wk"][j * dh:(j + 1) * dh] for j in range(k0, k1)]
                blocks += [w["wv"][j * dh:(j + 1) * dh] for j in range(k0, k1)]
                order = np.stack([np.arange(half), np.arange(half) + half], 1).reshape(-1)
                qkv = np.concatenate([b[order] for b in blocks])
                assert np.array_equal(vtlib.vt_shard_weights_read(st.part, (l, d, 0), 1), qkv)
                assert np.array_equal(vtlib.vt_shard_weights_read(st.part, (l, d, 0), 2),
                                      w["wo"][:, hr[0] * dh:hr[1] * dh])
                assert np.array_equal(vtlib.vt_shard_weights_read(st.part, (l, d, 0), 0)[0],
                                      w["attn_norm"])
                c0, c1 = cr
                gu = np.stack([w["w_gate"][c0:c1], w["w_up"][c0:c1]], 1).reshape(2 * (c1 - c0), -1)
                assert np.array_equal(vtlib.vt_shard_weights_read(st.part, (l, d, 1), 4), gu)
                down_t = vtlib.vt_shard_weights_read(st.part, (l, d, 1), 5)
                assert np.array_equal(down_t, w["w_down"][:, c0:c1].T)
                assert np.array_equal(vtlib.vt_shard_weights_read(st.part, (l, d, 1), 3)[0],
                                      w["ffn_norm"])


def _tagged(hk, n_pos, dh, layer, dev_):
    j, p, c = np.meshgrid(np.arange(hk), np.arange(n_pos), np.arange(dh), indexing="ij")
    bits = ((layer * 7 + dev_ * 3 + j) * 131 + p * 17 + c) % 0x7800  # finite, nonnegative halves
    return bits.astype(np.uint16).view(np.float16)


def test_kv_tagged_round_trip_and_append_position(vtlib):
    wl = synthetic.small("tags", n_layers=2, d_model=256, n_heads=4, n_kv_heads=2, d_head=64,
                         d_ffn=128, head_ranges=((0, 2), (2, 4)), ffn_ranges=((0, 64), (64, 128)),
                         model_id=94)
    cap, L = 40, 23
    with build(vtlib, wl, capacity=cap) as st:
        tags = {}
        for l in range(2):
            for d in range(2):
                k = _tagged(1, cap, 64, l, d)
                v = _tagged(1, cap, 64, l + 5, d)
                vtlib.vt_kv_write_raw(st.kv, l, d, k, v)
                tags[l, d] = (k, v)
        for l in range(2):
            for d in range(2):
                k, v = vtlib.vt_kv_read(st.kv, l, d, cap, 1, 64)
                assert k.view(np.uint16).tobytes() == tags[l, d][0].view(np.uint16).tobytes()
                assert v.view(np.uint16).tobytes() == tags[l, d][1].view(np.uint16).tobytes()
        vtlib.vt_kv_set_length(st.kv, 1, L)
        assert vtlib.vt_kv_length(st.kv, 1) == L and vtlib.vt_kv_length(st.kv, 0) == 0
        x = dev(wl.hidden(1, stream=1).reshape(-1))
        out = torch.empty(256, dtype=torch.float32, device="cuda")
        vtlib.vt_decode_step(st.part, (1, 1, ATTN), x, st.kv, out)
        k, v = vtlib.vt_kv_read(st.kv, 1, 1, cap, 1, 64)
        kt, vt_ = tags[1, 1]
        changed = [p for p in range(cap) if not np.array_equal(k[:, p], kt[:, p])]
        assert changed == [L]
        assert np.array_equal(v[:, :L], vt_[:, :L]) and np.array_equal(v[:, L + 1:], vt_[:, L + 1:])
        for other in ((0, 0), (0, 1), (1, 0)):   # no other cache was touched
            k2, v2 = vtlib.vt_kv_read(st.kv, *other, cap, 1, 64)
            assert np.array_equal(k2, tags[other][0]) and np.array_equal(v2, tags[other][1])
        assert vtlib.vt_kv_length(st.kv, 1) == L  # decode does not advance
        vtlib.vt_kv_advance(st.kv, -1, 3)
        assert [vtlib.vt_kv_length(st.kv, l) for l in range(2)] == [3, L + 3]


def test_decode_is_reproducible(vtlib):
    """ATTN partials repeat bit for bit; FFN partials are added into the output by bulk
    reductions whose order across CTAs varies, so they repeat to fp32 rounding."""
    wl = synthetic.WORKLOADS[1]
    kc, vc = wl.kv_fill(0, 128, 136)
    with build(vtlib, wl, capacity=136) as st:
        write_cache(vtlib, st, 0, wl, kc, vc, 128, wl.head_ranges)
        x = dev(wl.hidden(1, stream=9).reshape(-1))
        outs = []
        for _ in range(2):
            vtlib.vt_kv_set_length(st.kv, 0, 128)
            o = [torch.empty(512, dtype=torch.float32, device="cuda") for _ in range(4)]
            for d in range(2):
                vtlib.vt_decode_step(st.part, (0, d, ATTN), x, st.kv, o[d])
                vtlib.vt_decode_step(st.part, (0, d, FFN), x, None, o[2 + d])
            outs.append([host(t) for t in o])
        for d in range(2):
            assert outs[0][d].tobytes() == outs[1][d].tobytes()
            ffn_a, ffn_b = outs[0][2 + d].astype(np.float64), outs[1][2 + d].astype(np.float64)
            assert np.max(np.abs(ffn_a - ffn_b)) <= 1e-6 * max(1.0, np.max(np.abs(ffn_a)))


# ------------------------------------------------------------------ whole stack + graphs

def test_decode_token_stack_and_graph_replay(vtlib):
    """vt_decode_token over a 3-layer model, eager for step 0 and as a replayed CUDA graph for
    steps 1-3 (positions advance on the device), against the oracle run layer by layer."""
    wl = synthetic.small("stack", n_layers=3, d_model=256, n_heads=4, n_kv_heads=2, d_head=64,
                         d_ffn=320, head_ranges=((0, 2), (2, 2), (2, 4)),
                         ffn_ranges=((0, 100), (100, 217), (217, 320)), model_id=95)
    L0, steps, cap = 37, 4, 48
    ws = [wl.layer_weights(l) for l in range(3)]
    caches = []
    with build(vtlib, wl, capacity=cap) as st:
        for l in range(3):
            kc, vc = wl.kv_fill(l, L0, cap)
            caches.append((kc, vc))
            write_cache(vtlib, st, l, wl, kc, vc, L0, wl.head_ranges)
        vtlib.vt_kv_set_length(st.kv, -1, L0)
        xin = torch.empty(256, dtype=torch.float16, device="cuda")
        xout = torch.empty(256, dtype=torch.float16, device="cuda")
        graph = None
        for t in range(steps):
            x = wl.hidden(1, stream=20 + t)
            xin.copy_(dev(x.reshape(-1)))
            if t == 0:
                vtlib.vt_decode_token(st.part, st.kv, xin, xout)
            else:
                if graph is None:
                    graph = torch.cuda.CUDAGraph()
                    s = torch.cuda.Stream()
                    s.wait_stream(torch.cuda.current_stream())
                    with torch.cuda.stream(s):
                        with torch.cuda.graph(graph, stream=s):
                            vtlib.vt_decode_token(st.part, st.kv, xin, xout, stream=s)
                    torch.cuda.current_stream().wait_stream(s)
                graph.replay()
            ref = x.reshape(1, -1)
            for l in range(3):
                _, ref, _, _ = oracle.tp_layer(wl, ws[l], ref, L0 + t, *caches[l])
            assert_close(host(xout), ref.reshape(-1), f"step {t}")
        torch.cuda.synchronize()
        assert [vtlib.vt_kv_length(st.kv, l) for l in range(3)] == [L0 + steps] * 3
        assert vtlib.vt_kv_status(st.kv) == 0


def test_kv_overflow_is_reported_not_faulted(vtlib):
    wl = synthetic.WORKLOADS[1]
    cap = 10
    with build(vtlib, wl, capacity=cap) as st:
        vtlib.vt_kv_set_length(st.kv, 0, cap - 1)
        xin = dev(wl.hidden(1, stream=1).reshape(-1))
        xout = torch.empty_like(xin)
        g = torch.cuda.CUDAGraph()
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(s):
            with torch.cuda.graph(g, stream=s):
                vtlib.vt_decode_token(st.part, st.kv, xin, xout, stream=s)
        torch.cuda.current_stream().wait_stream(s)
        g.replay()                       # fills position cap-1
        assert vtlib.vt_kv_status(st.kv) == 0
        g.replay()                       # would write position cap: skipped and flagged
        torch.cuda.synchronize()
        assert vtlib.vt_kv_status(st.kv, clear=True) & vtlib.VT_DEV_KV_OVERFLOW
        assert np.isfinite(host(xout).astype(np.float32)).all()
        # eagerly, the host mirror (updated by vt_kv_length) refuses before launching
        assert vtlib.vt_kv_length(st.kv, 0) == cap + 1
        vtlib.vt_kv_set_length(st.kv, 0, cap)
        with pytest.raises(vtlib.VtError) as e:
            vtlib.vt_decode_step(st.part, (0, 0, ATTN), xin, st.kv,
                                 torch.empty(512, dtype=torch.float32, device="cuda"))
        assert e.value.status == vtlib.VT_ERR_KV_CAPACITY
