"""Sliding-window attention (vt_model_set_window) on every attention path, against the oracle's
windowed attention (a row at position p attends to [max(0, p - W + 1), p]):
  decode per shard (vt_decode_step), the static-scratch step, the fused token (vt_decode_token),
  prefill per shard (vt_prefill) and the whole-stack prefill (vt_prefill_tokens).
Windows cover the degenerate W = 1 (each row sees only itself), windows that end inside and at the
edge of a 64-position tile, a window longer than the cache (equal to full attention), and the
gemma-3 window of 1024 at a KV length of 4096 on the 8B-GQA shapes.
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


def stack(vt, wl, capacity, windows, layer_ids=None):
    from paper_2607_07046_gb300.stack import Stack
    layer_ids = list(range(wl.n_layers)) if layer_ids is None else list(layer_ids)
    shapes = shapes_of(vt, wl, max_seq=max(wl.max_seq, capacity))
    shapes.n_layers = len(layer_ids)
    return Stack(shapes, lambda i: wl.layer_weights(layer_ids[i]), wl.head_ranges, wl.ffn_ranges, capacity,
                 windows=windows)


def fill(vt, st, layer, wl, kc, vc, L):
    for d, hr in enumerate(wl.head_ranges):
        k0, k1 = kv_range(wl, hr)
        if k1 > k0 and L > 0:
            vt.vt_kv_write_raw(st.kv, layer, d, kc[k0:k1, :L], vc[k0:k1, :L])
    vt.vt_kv_set_length(st.kv, layer, L)


# ------------------------------------------------------------------ decode, per shard

@pytest.mark.parametrize("L,W", [(0, 1), (1, 1), (200, 1), (63, 5), (200, 64), (200, 65), (127, 128),
                                 (200, 201), (200, 10000), (64, 64)])
def test_decode_step_window(vtlib, L, W):
    vt = vtlib
    wl = synthetic.WORKLOADS[1]
    w = wl.layer_weights(0)
    cap = 256
    kc, vc = wl.kv_fill(0, L, cap) if L > 0 else oracle.new_cache(wl, cap)
    with stack(vt, wl, cap, W) as st:
        assert vt.vt_model_window(st.model, 0) == W
        fill(vt, st, 0, wl, kc, vc, L)
        x = wl.hidden(1, stream=200 + L)
        D = wl.d_model
        parts = [torch.empty(D, dtype=torch.float32, device="cuda") for _ in wl.head_ranges]
        for d in range(len(wl.head_ranges)):
            vt.vt_decode_step(st.part, (0, d, ATTN), dev(x.reshape(D)), st.kv, parts[d])
        _, ap = oracle.tp_attention(wl, w, x, L, kc, vc, window=W)
        for d in range(len(wl.head_ranges)):
            assert_close(host(parts[d]), ap[d], f"L={L} W={W} windowed partial dev {d}")
        assert vt.vt_kv_status(st.kv) == 0


def test_static_step_window(vtlib):
    """The static-scratch step honours the window like vt_decode_step (GQA group 4, dh 128)."""
    vt = vtlib
    wl = synthetic.small("swa-static", n_layers=1, d_model=1024, n_heads=8, n_kv_heads=2, d_head=128, d_ffn=256,
                         head_ranges=((0, 4), (4, 8)), ffn_ranges=((0, 128), (128, 256)), kv_len=300,
                         decode_steps=1, prompt_len=0, model_id=120)
    w = wl.layer_weights(0)
    L, W, cap = 300, 100, 320
    kc, vc = wl.kv_fill(0, L, cap)
    with stack(vt, wl, cap, W) as st:
        fill(vt, st, 0, wl, kc, vc, L)
        x = wl.hidden(1, stream=210)
        part = torch.empty(wl.d_model, dtype=torch.float32, device="cuda")
        vt.vt_decode_step_static(st.part, (0, 1, ATTN), dev(x.reshape(-1)), st.kv, part)
        _, ap = oracle.tp_attention(wl, w, x, L, kc, vc, window=W)
        assert_close(host(part), ap[1], "static step windowed partial")


# ------------------------------------------------------------------ decode, fused token

def test_fused_token_per_layer_windows(vtlib):
    """Three layers with windows 1, 0 (full) and 40, three tokens from KV length 70 (the windows
    cut inside the cache and move with the position), against the oracle chained layer by layer."""
    vt = vtlib
    wl = synthetic.small("swa-fused", n_layers=3, d_model=512, n_heads=8, n_kv_heads=4, d_head=64, d_ffn=640,
                         head_ranges=((0, 2), (2, 6), (6, 8)), ffn_ranges=((0, 200), (200, 420), (420, 640)),
                         kv_len=70, decode_steps=3, prompt_len=0, model_id=121)
    windows = [1, 0, 40]
    L0, steps, cap = 70, 3, 80
    ws = [wl.layer_weights(l) for l in range(3)]
    caches = [wl.kv_fill(l, L0, cap) for l in range(3)]
    with stack(vt, wl, cap, windows) as st:
        fused = vt.vt_decode_token_fused_available(st.part)
        assert fused[0], fused[1]
        for l in range(3):
            fill(vt, st, l, wl, caches[l][0], caches[l][1], L0)
        xout = torch.empty(wl.d_model, dtype=torch.float16, device="cuda")
        for t in range(steps):
            x = wl.hidden(1, stream=220 + t)
            vt.vt_decode_token(st.part, st.kv, dev(x.reshape(-1)), xout)
            r = x.reshape(1, -1)
            for l in range(3):
                _, r, ap, fp = oracle.tp_layer(wl, ws[l], r, L0 + t, *caches[l], window=windows[l])
            assert_close(host(xout), r.reshape(-1), f"windowed fused token {t}")
            got = vt.vt_token_partials_read(st.part, ATTN, 3, wl.d_model)
            for d in range(3):
                assert_close(got[d], ap[d].reshape(-1), f"token {t} last-layer windowed partial dev {d}")
        assert vt.vt_kv_status(st.kv) == 0


def test_8b_gqa_window_1024_at_kv_4096(vtlib):
    """The gemma-3 window (1024) on a full-size 8B-GQA layer at KV length 4096: the fused token and
    the per-shard step against the oracle; the window reads a quarter of the cache."""
    vt = vtlib
    wl = synthetic.WORKLOADS[5]
    layer, L, W = wl.n_layers - 1, wl.kv_len, 1024
    cap = L + 8
    w = wl.layer_weights(layer)
    kc, vc = wl.kv_fill(layer, L, cap)
    x = (wl.hidden(1, stream=230).astype(np.float32) * 1e-3).astype(np.float16)  # partials dominate
    n = len(wl.head_ranges)
    with stack(vt, wl, cap, W, layer_ids=[layer]) as st:
        fill(vt, st, 0, wl, kc, vc, L)
        xout = torch.empty(wl.d_model, dtype=torch.float16, device="cuda")
        vt.vt_decode_token(st.part, st.kv, dev(x.reshape(-1)), xout)
        got = vt.vt_token_partials_read(st.part, ATTN, n, wl.d_model)
        k_after, v_after = kc.copy(), vc.copy()
        h_ref, ap = oracle.tp_attention(wl, w, x, L, k_after, v_after, window=W)
        xn_ref, _ = oracle.tp_ffn(wl, w, h_ref)
        for d in range(n):
            assert_close(got[d], ap[d].reshape(-1), f"8b W=1024 fused partial dev {d}")
        assert_close(host(xout), xn_ref.reshape(-1), "8b W=1024 fused x_out")
        # the per-shard path at the same position (the token advanced the length: rewind it)
        vt.vt_kv_set_length(st.kv, 0, L)
        part = torch.empty(wl.d_model, dtype=torch.float32, device="cuda")
        vt.vt_decode_step(st.part, (0, 2, ATTN), dev(x.reshape(-1)), st.kv, part)
        assert_close(host(part), ap[2], "8b W=1024 per-shard partial dev 2")
        assert vt.vt_kv_status(st.kv) == 0


# ------------------------------------------------------------------ prefill

@pytest.mark.parametrize("pos0,n,W", [(0, 300, 1), (0, 300, 37), (0, 300, 64), (0, 300, 65), (0, 300, 1000),
                                      (77, 150, 50), (77, 150, 128)])
def test_prefill_shard_window(vtlib, pos0, n, W):
    """Per-shard prefill rows at positions pos0 .. pos0 + n - 1 (after pos0 cached positions):
    windows inside one 64-position tile, across tile edges, and longer than every row's history."""
    vt = vtlib
    wl = synthetic.WORKLOADS[1]
    w = wl.layer_weights(0)
    cap = pos0 + n + 8
    kc, vc = wl.kv_fill(0, pos0, cap) if pos0 > 0 else oracle.new_cache(wl, cap)
    X = wl.hidden(n, stream=240 + W)
    D = wl.d_model
    with stack(vt, wl, cap, W) as st:
        fill(vt, st, 0, wl, kc, vc, pos0)
        parts = [torch.empty((n, D), dtype=torch.float32, device="cuda") for _ in wl.head_ranges]
        for d in range(len(wl.head_ranges)):
            vt.vt_prefill(st.part, (0, d, ATTN), dev(X), n, st.kv, parts[d])
        _, ap = oracle.tp_attention(wl, w, X, pos0, kc, vc, window=W)
        for d in range(len(wl.head_ranges)):
            assert_close(host(parts[d]), ap[d], f"pos0={pos0} W={W} prefill partial dev {d}")
        assert vt.vt_kv_status(st.kv) == 0


@pytest.mark.parametrize("cid,pos0,n,W", [(1, 1000, 300, 0), (1, 1000, 300, 700), (5, 900, 260, 0), (5, 900, 260, 300)])
def test_prefill_long_history(vtlib, cid, pos0, n, W):
    """Prompt rows after a long cached history: up to 11 blocks of 128 keys per row tile, so the
    two-slot K/V rings are refilled many times and every row's running maximum meets new blocks;
    with and without a window, at dh 64 (config 1) and dh 128 with 4 query heads per KV head
    (config 5).  Per-shard attention partials on sampled rows against the oracle."""
    vt = vtlib
    wl = dataclasses.replace(synthetic.WORKLOADS[cid], n_layers=1)
    w = wl.layer_weights(0)
    cap = pos0 + n + 8
    kc, vc = wl.kv_fill(0, pos0, cap)
    X = wl.hidden(n, stream=260 + cid + W)
    rows = np.array([0, 1, 127, 128, 200, 255, 256, n - 1])
    D = wl.d_model
    with stack(vt, wl, cap, W) as st:
        fill(vt, st, 0, wl, kc, vc, pos0)
        parts = [torch.empty((n, D), dtype=torch.float32, device="cuda") for _ in wl.head_ranges]
        for d in range(len(wl.head_ranges)):
            vt.vt_prefill(st.part, (0, d, ATTN), dev(X), n, st.kv, parts[d])
        for hr in wl.head_ranges:
            oracle.kv_append(wl, w, oracle.kv_heads_of(wl, hr), X, pos0, kc, vc)
        for d, hr in enumerate(wl.head_ranges):
            ap = oracle.attn_partial(wl, w, hr, X[rows], pos0 + rows, kc, vc, W)
            assert_close(host(parts[d])[rows], ap, f"cid {cid} pos0 {pos0} W {W} partial dev {d}")
        assert vt.vt_kv_status(st.kv) == 0


def test_prefill_tokens_windows_two_layers(vtlib):
    """The whole-stack prefill with windows 64 and 0 on two layers, and then a decode token on the
    cache it wrote, against the oracle chained layer by layer."""
    vt = vtlib
    wl = dataclasses.replace(synthetic.WORKLOADS[1], n_layers=2)
    windows = [64, 0]
    n, cap = 200, 208
    X = wl.hidden(n, stream=250)
    ws = [wl.layer_weights(l) for l in range(2)]
    caches = [oracle.new_cache(wl, cap) for _ in range(2)]
    ref = X
    for l in range(2):
        _, ref, _, _ = oracle.tp_layer(wl, ws[l], ref, 0, *caches[l], window=windows[l])
    with stack(vt, wl, cap, windows) as st:
        out = torch.empty((n, wl.d_model), dtype=torch.float16, device="cuda")
        vt.vt_prefill_tokens(st.part, st.kv, dev(X), n, out)
        assert_close(host(out), ref, "windowed two-layer prefill")
        x = wl.hidden(1, stream=251)
        y = torch.empty(wl.d_model, dtype=torch.float16, device="cuda")
        vt.vt_decode_token(st.part, st.kv, dev(x.reshape(-1)), y)
        r = x.reshape(1, -1)
        for l in range(2):
            _, r, _, _ = oracle.tp_layer(wl, ws[l], r, n, *caches[l], window=windows[l])
        assert_close(host(y), r.reshape(-1), "windowed decode after prefill")
        assert vt.vt_kv_status(st.kv) == 0 and vt.vt_partition_status(st.part) == 0


def test_prefill_tokens_8b_gqa_window(vtlib):
    """One full-width 8B-GQA layer through vt_prefill_tokens with a window of 100, sampled rows
    (before, at and past the window's length) and every appended K/V row."""
    vt = vtlib
    wl = dataclasses.replace(synthetic.WORKLOADS[5], n_layers=1)
    w = wl.layer_weights(0)
    n, W = 260, 100
    rows = np.array([0, 1, 98, 99, 100, 127, 128, 200, 259])
    X = (wl.hidden(n, stream=252).astype(np.float32) * 1e-3).astype(np.float16)
    kc, vc = oracle.new_cache(wl, n)
    for hr in wl.head_ranges:
        oracle.kv_append(wl, w, oracle.kv_heads_of(wl, hr), X, 0, kc, vc)
    ap = [oracle.attn_partial(wl, w, hr, X[rows], rows, kc, vc, W) for hr in wl.head_ranges]
    h = oracle.combine(ap, X[rows])
    fp = [oracle.ffn_partial(wl, w, cr, h) for cr in wl.ffn_ranges]
    ref = oracle.combine(fp, h)
    with stack(vt, wl, n, W) as st:
        out = torch.empty((n, wl.d_model), dtype=torch.float16, device="cuda")
        vt.vt_prefill_tokens(st.part, st.kv, dev(X), n, out)
        assert_close(host(out)[rows], ref, "8b W=100 prefill_tokens x_out")
        for d, hr in enumerate(wl.head_ranges):
            k0, k1 = kv_range(wl, hr)
            kg, vg = vt.vt_kv_read(st.kv, 0, d, n, k1 - k0, wl.d_head)
            assert_close(kg, kc[k0:k1, :n], f"k dev {d}")
            assert_close(vg, vc[k0:k1, :n], f"v dev {d}")


# ------------------------------------------------------------------ API

def test_window_api_rules(vtlib):
    vt = vtlib
    wl = synthetic.WORKLOADS[1]
    m = vt.vt_model_create(shapes_of(vt, wl), [wl.layer_weights(0)])
    try:
        for bad in [(0, -1), (1, 8), (-2, 8)]:
            with pytest.raises(vt.VtError) as e:
                vt.vt_model_set_window(m, bad[0], bad[1])
            assert e.value.status == vt.VT_ERR_INVALID_ARG
        vt.vt_model_set_window(m, -1, 512)
        assert vt.vt_model_window(m, 0) == 512
        p = vt.vt_partition_create(m, wl.head_ranges, wl.ffn_ranges)
        with pytest.raises(vt.VtError) as e:
            vt.vt_model_set_window(m, 0, 16)
        assert e.value.status == vt.VT_ERR_STATE
        vt.vt_partition_destroy(p)
        vt.vt_model_set_window(m, 0, 0)
        assert vt.vt_model_window(m, 0) == 0
    finally:
        vt.vt_model_destroy(m)
