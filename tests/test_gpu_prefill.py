"""Prefill path on the GPU (through the C ABI) against the CPU oracle.

Every comparison uses the tolerance in tests/parity.py (rel-RMS <= 1e-3, max-abs <= 2e-2 per
tensor).  The oracle appends K/V for every row; where the full oracle would take minutes (7B- and
13B-shaped layers) the attention and FFN outputs are compared on sampled rows that span several
128-row GEMM tiles and the ragged tail.  The FFN block is teacher-forced: its input is the oracle's
h on the compared rows.
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


def build(vt, wl, capacity, ranges=None):
    from paper_2607_07046_gb300.stack import Stack
    shapes = shapes_of(vt, wl, max_seq=max(wl.max_seq, capacity))
    heads, cols = ranges if ranges is not None else (wl.head_ranges, wl.ffn_ranges)
    return Stack(shapes, wl.layer_weights, heads, cols, capacity)


def prefill_layer_check(vt, st, wl, w, layer, X, pos0, kc, vc, rows=None, tag=""):
    """Prefill rows X (at positions pos0 ..) through layer `layer`: every ATTN shard, the combine,
    every FFN shard (teacher-forced on the compared rows) and the combine, against the oracle.
    kc/vc are the oracle's full-layer caches holding pos0 positions; extended in place."""
    D, n = wl.d_model, X.shape[0]
    heads, cols = st.head_ranges, st.ffn_ranges
    rows = np.arange(n) if rows is None else np.asarray(rows)
    xg = dev(X)
    before = {}
    for d, hr in enumerate(heads):
        k0, k1 = kv_range(wl, hr)
        if k1 > k0 and pos0 > 0:
            before[d] = vt.vt_kv_read(st.kv, layer, d, pos0, k1 - k0, wl.d_head)
    parts = [torch.empty((n, D), dtype=torch.float32, device="cuda") for _ in heads]
    for d in range(len(heads)):
        vt.vt_prefill(st.part, (layer, d, ATTN), xg, n, st.kv, parts[d])
    hg = torch.empty((n, D), dtype=torch.float16, device="cuda")
    vt.vt_combine(parts, xg, hg, n, D)
    for hr in heads:
        k0, k1 = oracle.kv_heads_of(wl, hr)
        if k1 > k0:
            oracle.kv_append(wl, w, (k0, k1), X, pos0, kc, vc)
    ap = [oracle.attn_partial(wl, w, hr, X[rows], pos0 + rows, kc, vc) for hr in heads]
    h_ref = oracle.combine(ap, X[rows])
    for d in range(len(heads)):
        assert_close(host(parts[d])[rows], ap[d], f"{tag} attn partial dev {d}")
    assert_close(host(hg)[rows], h_ref, f"{tag} h")
    # the appended K/V rows, and the earlier rows untouched
    for d, hr in enumerate(heads):
        k0, k1 = kv_range(wl, hr)
        if k1 == k0:
            continue
        kg, vg = vt.vt_kv_read(st.kv, layer, d, pos0 + n, k1 - k0, wl.d_head)
        if d in before:
            assert np.array_equal(kg[:, :pos0], before[d][0]) and np.array_equal(vg[:, :pos0], before[d][1])
        assert_close(kg[:, pos0:], kc[k0:k1, pos0:pos0 + n], f"{tag} k rows dev {d}")
        assert_close(vg[:, pos0:], vc[k0:k1, pos0:pos0 + n], f"{tag} v rows dev {d}")
    # FFN block: GPU input = GPU h with the oracle's h on the compared rows
    hin = hg.clone()
    hin[torch.from_numpy(rows).cuda()] = dev(h_ref)
    fparts = [torch.empty((n, D), dtype=torch.float32, device="cuda") for _ in cols]
    for d in range(len(cols)):
        vt.vt_prefill(st.part, (layer, d, FFN), hin, n, None, fparts[d])
    xn = torch.empty((n, D), dtype=torch.float16, device="cuda")
    vt.vt_combine(fparts, hin, xn, n, D)
    fp = [oracle.ffn_partial(wl, w, cr, h_ref) for cr in cols]
    xn_ref = oracle.combine(fp, h_ref)
    for d in range(len(cols)):
        assert_close(host(fparts[d])[rows], fp[d], f"{tag} ffn partial dev {d}")
    assert_close(host(xn)[rows], xn_ref, f"{tag} x_next")
    vt.vt_kv_advance(st.kv, layer, n)
    return h_ref, xn_ref


# ------------------------------------------------------------------ tiny config (config 1)

def test_tiny_prefill_128_then_continue_then_decode(vtlib):
    """Config 1: a 128-row prompt, a second 37-row chunk at position 128, then one decode token."""
    vt = vtlib
    wl = synthetic.WORKLOADS[1]
    w = wl.layer_weights(0)
    cap = 192
    kc, vc = oracle.new_cache(wl, cap)
    with build(vt, wl, cap) as st:
        prefill_layer_check(vt, st, wl, w, 0, wl.hidden(128, stream=1), 0, kc, vc, tag="p128")
        prefill_layer_check(vt, st, wl, w, 0, wl.hidden(37, stream=11), 128, kc, vc, tag="p37@128")
        # a decode step on the cache the GPU prefill wrote
        x = wl.hidden(1, stream=2)
        D = wl.d_model
        parts = [torch.empty(D, dtype=torch.float32, device="cuda") for _ in wl.head_ranges]
        xg = dev(x.reshape(D))
        for d in range(len(wl.head_ranges)):
            vt.vt_decode_step(st.part, (0, d, ATTN), xg, st.kv, parts[d])
        h_ref, ap = oracle.tp_attention(wl, w, x, 165, kc, vc)
        for d in range(len(wl.head_ranges)):
            assert_close(host(parts[d]), ap[d][0], f"decode partial dev {d}")
        assert vt.vt_kv_status(st.kv) == 0 and vt.vt_partition_status(st.part) == 0


@pytest.mark.parametrize("n", [1, 2, 63, 64, 65, 127, 129, 200, 300])
def test_prefill_ragged_row_counts(vtlib, n):
    vt = vtlib
    wl = synthetic.WORKLOADS[1]
    w = wl.layer_weights(0)
    cap = 320
    kc, vc = oracle.new_cache(wl, cap)
    with build(vt, wl, cap) as st:
        prefill_layer_check(vt, st, wl, w, 0, wl.hidden(n, stream=20 + n), 0, kc, vc, tag=f"n={n}")


def test_prefill_at_offset_over_existing_cache(vtlib):
    """Rows appended after 77 cached positions (written through the test hook) attend to them."""
    vt = vtlib
    wl = synthetic.WORKLOADS[1]
    w = wl.layer_weights(0)
    cap, L = 256, 77
    kc, vc = wl.kv_fill(0, L, cap)
    with build(vt, wl, cap) as st:
        for d, hr in enumerate(wl.head_ranges):
            k0, k1 = kv_range(wl, hr)
            vt.vt_kv_write_raw(st.kv, 0, d, kc[k0:k1, :L], vc[k0:k1, :L])
        vt.vt_kv_set_length(st.kv, 0, L)
        prefill_layer_check(vt, st, wl, w, 0, wl.hidden(150, stream=3), L, kc, vc, tag="offset")


UNEVEN = [
    # (heads, kv heads, head ranges, ffn ranges): shards whose FFN columns start off a multiple
    # of 8, an empty shard of each kind, GQA groups 2, 4 and 8
    (8, 8, ((0, 1), (1, 4), (4, 8)), ((0, 701), (701, 1000), (1000, 1408))),
    (8, 8, ((0, 8), (8, 8)), ((0, 0), (0, 1408))),
    (8, 4, ((0, 2), (2, 8)), ((0, 9), (9, 1408))),
    (8, 2, ((0, 4), (4, 8)), ((0, 704), (704, 1408))),
    (8, 1, ((0, 8),), ((0, 1408),)),
    # nine shards (one head each and an empty one): more than one launch per block for the
    # attention (six shards a launch) and the GEMMs (eight)
    (8, 8, tuple((h, h + 1) for h in range(8)) + ((8, 8),), tuple((i * 1408 // 9, (i + 1) * 1408 // 9) for i in range(9))),
]


@pytest.mark.parametrize("H,Hk,heads,cols", UNEVEN)
def test_prefill_uneven_and_gqa_partitions(vtlib, H, Hk, heads, cols):
    vt = vtlib
    wl = synthetic.small("uneven", n_layers=1, d_model=512, n_heads=H, n_kv_heads=Hk, d_head=64,
                         d_ffn=1408, head_ranges=heads, ffn_ranges=cols, kv_len=0, decode_steps=1,
                         prompt_len=140, model_id=91)
    w = wl.layer_weights(0)
    cap = 160
    kc, vc = oracle.new_cache(wl, cap)
    with build(vt, wl, cap) as st:
        prefill_layer_check(vt, st, wl, w, 0, wl.hidden(140, stream=4), 0, kc, vc, tag=f"H={H} Hk={Hk}")


# ------------------------------------------------------------------ model-sized layers, sampled rows

SAMPLED = [0, 1, 64, 127, 128, 129, 255]


def test_prefill_8b_gqa_layer_sampled(vtlib):
    """One layer of the 8B GQA model (32/8 heads of 128, FFN 14336, theta 5e5), 4-way, 260 rows."""
    vt = vtlib
    wl = dataclasses.replace(synthetic.WORKLOADS[5], n_layers=1)
    w = wl.layer_weights(0)
    n, cap = 260, 272
    kc, vc = oracle.new_cache(wl, cap)
    with build(vt, wl, cap) as st:
        prefill_layer_check(vt, st, wl, w, 0, wl.hidden(n, stream=5), 0, kc, vc, rows=SAMPLED + [259], tag="8b")


def test_prefill_13b_uneven_layer_sampled(vtlib):
    """One layer of the 13B model with the uneven 3-way split (heads 20/12/8, FFN 6912/4147/2765)."""
    vt = vtlib
    wl = dataclasses.replace(synthetic.WORKLOADS[3], n_layers=1)
    w = wl.layer_weights(0)
    n, cap = 140, 160
    kc, vc = oracle.new_cache(wl, cap)
    with build(vt, wl, cap) as st:
        prefill_layer_check(vt, st, wl, w, 0, wl.hidden(n, stream=6), 0, kc, vc, rows=[0, 50, 127, 128, 139], tag="13b")


def test_prefill_7b_512_rows_sampled(vtlib):
    """One layer of the 7B prefill workload (512-row prompt, even 4-way split)."""
    vt = vtlib
    wl = dataclasses.replace(synthetic.WORKLOADS[4], n_layers=1)
    w = wl.layer_weights(0)
    n = 512
    kc, vc = oracle.new_cache(wl, n)
    with build(vt, wl, n) as st:
        prefill_layer_check(vt, st, wl, w, 0, wl.hidden(n, stream=7), 0, kc, vc,
                            rows=[0, 1, 127, 128, 300, 383, 384, 511], tag="7b")


# ------------------------------------------------------------------ whole stack

def test_prefill_tokens_two_layer_stack(vtlib):
    """vt_prefill_tokens through two tiny layers equals the oracle's layer-by-layer prefill."""
    vt = vtlib
    wl = dataclasses.replace(synthetic.WORKLOADS[1], n_layers=2)
    n, cap = 150, 160
    X = wl.hidden(n, stream=8)
    ref = X
    caches = []
    for l in range(2):
        kc, vc = oracle.new_cache(wl, cap)
        _, ref, _, _ = oracle.tp_layer(wl, wl.layer_weights(l), ref, 0, kc, vc)
        caches.append((kc, vc))
    with build(vt, wl, cap) as st:
        out = torch.empty((n, wl.d_model), dtype=torch.float16, device="cuda")
        vt.vt_prefill_tokens(st.part, st.kv, dev(X), n, out)
        assert_close(host(out), ref, "two-layer prefill")
        for l in range(2):
            assert vt.vt_kv_length(st.kv, l) == n
            for d, hr in enumerate(wl.head_ranges):
                k0, k1 = kv_range(wl, hr)
                kg, vg = vt.vt_kv_read(st.kv, l, d, n, k1 - k0, wl.d_head)
                assert_close(kg, caches[l][0][k0:k1, :n], f"layer {l} k dev {d}")
                assert_close(vg, caches[l][1][k0:k1, :n], f"layer {l} v dev {d}")


@pytest.mark.parametrize("H,Hk,heads,cols", UNEVEN)
def test_prefill_tokens_uneven_and_gqa_partitions(vtlib, H, Hk, heads, cols):
    """vt_prefill_tokens runs every shard of a block in one launch per GEMM: uneven, empty and GQA
    partitions through two layers against the oracle chained layer by layer."""
    vt = vtlib
    wl = synthetic.small("uneven-stack", n_layers=2, d_model=512, n_heads=H, n_kv_heads=Hk, d_head=64,
                         d_ffn=1408, head_ranges=heads, ffn_ranges=cols, kv_len=0, decode_steps=1,
                         prompt_len=140, model_id=92)
    n, cap = 140, 160
    X = wl.hidden(n, stream=10)
    ref = X
    caches = []
    for l in range(2):
        kc, vc = oracle.new_cache(wl, cap)
        _, ref, _, _ = oracle.tp_layer(wl, wl.layer_weights(l), ref, 0, kc, vc)
        caches.append((kc, vc))
    with build(vt, wl, cap) as st:
        out = torch.empty((n, wl.d_model), dtype=torch.float16, device="cuda")
        vt.vt_prefill_tokens(st.part, st.kv, dev(X), n, out)
        assert_close(host(out), ref, f"prefill stack H={H} Hk={Hk} {heads}")
        for l in range(2):
            for d, hr in enumerate(wl.head_ranges):
                k0, k1 = kv_range(wl, hr)
                if k1 == k0:
                    continue
                kg, vg = vt.vt_kv_read(st.kv, l, d, n, k1 - k0, wl.d_head)
                assert_close(kg, caches[l][0][k0:k1, :n], f"layer {l} k dev {d}")
                assert_close(vg, caches[l][1][k0:k1, :n], f"layer {l} v dev {d}")
        assert vt.vt_kv_status(st.kv) == 0 and vt.vt_partition_status(st.part) == 0


def test_decode_after_prefill_equals_longer_prefill(vtlib):
    """GPU only: decoding token M after a prefill of M rows gives row M of a prefill of M + 1 rows."""
    vt = vtlib
    wl = dataclasses.replace(synthetic.WORKLOADS[1], n_layers=2)
    M, cap = 70, 96
    X = wl.hidden(M + 1, stream=9)
    with build(vt, wl, cap) as a, build(vt, wl, cap) as b:
        out_a = torch.empty((M, wl.d_model), dtype=torch.float16, device="cuda")
        vt.vt_prefill_tokens(a.part, a.kv, dev(X[:M]), M, out_a)
        y = torch.empty(wl.d_model, dtype=torch.float16, device="cuda")
        vt.vt_decode_token(a.part, a.kv, dev(X[M]), y)
        out_b = torch.empty((M + 1, wl.d_model), dtype=torch.float16, device="cuda")
        vt.vt_prefill_tokens(b.part, b.kv, dev(X), M + 1, out_b)
        assert_close(host(y), host(out_b)[M], "decode vs prefill row")
        assert_close(host(out_a), host(out_b)[:M], "shorter prefill rows")


# ------------------------------------------------------------------ the timed path at full width

def _stack_layer_reference(wl, w, X, rows, cap):
    """The oracle's one-layer prefill of X from position 0: every KV head's K/V rows for all of X,
    the layer output on `rows` (attention over the causal set of each row)."""
    kc, vc = oracle.new_cache(wl, cap)
    n = X.shape[0]
    for hr in wl.head_ranges:
        k0, k1 = oracle.kv_heads_of(wl, hr)
        if k1 > k0:
            oracle.kv_append(wl, w, (k0, k1), X, 0, kc, vc)
    rows = np.asarray(rows)
    ap = [oracle.attn_partial(wl, w, hr, X[rows], rows, kc, vc) for hr in wl.head_ranges]
    h = oracle.combine(ap, X[rows])
    fp = [oracle.ffn_partial(wl, w, cr, h) for cr in wl.ffn_ranges]
    return oracle.combine(fp, h), kc, vc


def _check_cache(vt, st, wl, layer, n, kc, vc, tag):
    for d, hr in enumerate(wl.head_ranges):
        k0, k1 = kv_range(wl, hr)
        if k1 == k0:
            continue
        kg, vg = vt.vt_kv_read(st.kv, layer, d, n, k1 - k0, wl.d_head)
        assert_close(kg, kc[k0:k1, :n], f"{tag} layer {layer} k dev {d}")
        assert_close(vg, vc[k0:k1, :n], f"{tag} layer {layer} v dev {d}")


FULL_WIDTH = {
    # config: (prompt rows, sampled rows spanning 128-row tiles and the ragged tail)
    4: (512, [0, 1, 127, 128, 255, 256, 300, 383, 384, 510, 511]),   # 7B, even 4-way (the bench's shape)
    3: (300, [0, 63, 127, 128, 200, 256, 299]),                      # 13B, heads 20/12/8, FFN 6912/4147/2765
    5: (260, [0, 1, 127, 128, 255, 259]),                           # 8B GQA, 2 KV heads per shard
}


@pytest.mark.parametrize("cid", list(FULL_WIDTH))
def test_prefill_tokens_full_width_one_layer(vtlib, cid):
    """vt_prefill_tokens (one grouped tensor-core GEMM launch per projection for all shards, split-K
    chosen by the time model) on one full-width layer, against the oracle.  The prompt's residual is
    scaled down (x ~ N(0, 0.01^2)), so the output is dominated by the shard partials and an error in
    any of them shows; every appended K/V row is compared too."""
    vt = vtlib
    n, rows = FULL_WIDTH[cid]
    wl = dataclasses.replace(synthetic.WORKLOADS[cid], n_layers=1)
    w = wl.layer_weights(0)
    X = (wl.hidden(n, stream=160 + cid).astype(np.float32) * 0.01).astype(np.float16)
    ref, kc, vc = _stack_layer_reference(wl, w, X, rows, n)
    assert np.sqrt(np.mean(X.astype(np.float64) ** 2)) < 0.05 * np.sqrt(np.mean(ref.astype(np.float64) ** 2))
    with build(vt, wl, n) as st:
        out = torch.empty((n, wl.d_model), dtype=torch.float16, device="cuda")
        vt.vt_prefill_tokens(st.part, st.kv, dev(X), n, out)
        assert_close(host(out)[rows], ref, f"{wl.name} prefill_tokens x_out")
        _check_cache(vt, st, wl, 0, n, kc, vc, wl.name)
        assert vt.vt_kv_length(st.kv, 0) == n
        assert vt.vt_kv_status(st.kv) == 0 and vt.vt_partition_status(st.part) == 0


def test_prefill_tokens_7b_two_layers_512_rows(vtlib):
    """The benchmarked prompt shape (512 rows, 7B width, even 4-way) through two layers of the
    stack: layer 0 in full on the oracle (its output feeds layer 1's K/V), layer 1 on sampled rows."""
    vt = vtlib
    n, rows = FULL_WIDTH[4]
    wl = dataclasses.replace(synthetic.WORKLOADS[4], n_layers=2)
    X = wl.hidden(n, stream=170)
    w0, w1 = wl.layer_weights(0), wl.layer_weights(1)
    kc0, vc0 = oracle.new_cache(wl, n)
    _, x1, _, _ = oracle.tp_layer(wl, w0, X, 0, kc0, vc0)
    ref, kc1, vc1 = _stack_layer_reference(wl, w1, x1, rows, n)
    with build(vt, wl, n) as st:
        out = torch.empty((n, wl.d_model), dtype=torch.float16, device="cuda")
        vt.vt_prefill_tokens(st.part, st.kv, dev(X), n, out)
        assert_close(host(out)[rows], ref, "7b two-layer prefill_tokens x_out")
        _check_cache(vt, st, wl, 0, n, kc0, vc0, "7b")
        _check_cache(vt, st, wl, 1, n, kc1, vc1, "7b")
        assert vt.vt_kv_status(st.kv) == 0 and vt.vt_partition_status(st.part) == 0
