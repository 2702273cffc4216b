"""The whole-token entry points against the CPU oracle: vt_decode_token (one fused cooperative
kernel per token when the partition supports it) and vt_decode_token_sharded (per-shard
kernels).  Each test runs several tokens in a row with the KV length advancing on the device, and
compares every token's output with the oracle chained through the same layers and caches.
"""
from __future__ import annotations

import numpy as np
import pytest

import oracle
import synthetic
from tests.parity import assert_close
from tests.test_gpu_decode import build, dev, host, write_cache

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


def run_tokens(vt, wl, layers, L0, steps, entry, graph=True, stream_id=70):
    """`steps` tokens through `layers` of the workload from KV length L0, returning the GPU
    outputs and the oracle's, token by token."""
    cap = L0 + steps + 4
    ws = [wl.layer_weights(l) for l in layers]
    caches = []
    got, ref = [], []
    with build(vt, wl, layer_ids=layers, capacity=cap) as st:
        for i, layer in enumerate(layers):
            if L0 > 0:
                kc, vc = wl.kv_fill(layer, L0, cap)
            else:
                kc, vc = oracle.new_cache(wl, cap)
            caches.append((kc, vc))
            write_cache(vt, st, i, wl, kc, vc, L0, wl.head_ranges)
        vt.vt_kv_set_length(st.kv, -1, L0)
        D = wl.d_model
        xin = torch.empty(D, dtype=torch.float16, device="cuda")
        xout = torch.empty(D, dtype=torch.float16, device="cuda")
        g = None
        if graph:
            g = torch.cuda.CUDAGraph()
            s = torch.cuda.Stream()
            s.wait_stream(torch.cuda.current_stream())
            with torch.cuda.stream(s):
                with torch.cuda.graph(g, stream=s):
                    entry(st.part, st.kv, xin, xout, stream=s)
            torch.cuda.current_stream().wait_stream(s)
        for t in range(steps):
            x = wl.hidden(1, stream=stream_id + t)
            xin.copy_(dev(x.reshape(-1)))
            if g is not None:
                g.replay()
            else:
                entry(st.part, st.kv, xin, xout)
            r = x.reshape(1, -1)
            for i in range(len(layers)):
                _, r, _, _ = oracle.tp_layer(wl, ws[i], r, L0 + t, *caches[i])
            got.append(host(xout).copy())
            ref.append(r.reshape(-1))
        torch.cuda.synchronize()
        assert vt.vt_kv_status(st.kv) == 0
        lens = [vt.vt_kv_length(st.kv, i) for i in range(len(layers))]
        assert lens == [L0 + steps] * len(layers)
        # the appended rows of the first shard's first KV head, every layer
        for i in range(len(layers)):
            g_ = wl.n_heads // wl.n_kv_heads
            h0, h1 = wl.head_ranges[0]
            if h1 == h0:
                continue
            kg, vg = vt.vt_kv_read(st.kv, i, 0, L0 + steps, h1 // g_ - h0 // g_, wl.d_head)
            kc, vc = caches[i]
            assert np.array_equal(kg[:, :L0], kc[h0 // g_:h1 // g_, :L0])
            assert_close(kg[:, L0:], kc[h0 // g_:h1 // g_, L0:L0 + steps], "appended k")
            assert_close(vg[:, L0:], vc[h0 // g_:h1 // g_, L0:L0 + steps], "appended v")
        fused = vt.vt_decode_token_fused_available(st.part)
    return got, ref, fused


SHAPES = {
    # name: (workload kwargs, layers, L0, steps)
    "mha-dh64-uneven-empty": (dict(n_layers=3, d_model=256, n_heads=4, n_kv_heads=2, d_head=64, d_ffn=320,
                                   head_ranges=((0, 2), (2, 2), (2, 4)),
                                   ffn_ranges=((0, 100), (100, 217), (217, 320)), model_id=96), [0, 1, 2], 37, 3),
    "mha-dh128-3way": (dict(n_layers=2, d_model=1024, n_heads=8, n_kv_heads=8, d_head=128, d_ffn=2752,
                            head_ranges=((0, 4), (4, 6), (6, 8)), ffn_ranges=((0, 1376), (1376, 2000), (2000, 2752)),
                            model_id=97), [0, 1], 300, 3),
    "gqa4-dh128": (dict(n_layers=2, d_model=1024, n_heads=8, n_kv_heads=2, d_head=128, d_ffn=1408,
                        head_ranges=((0, 4), (4, 8)), ffn_ranges=((0, 704), (704, 1408)), model_id=98,
                        rope_theta=5e5), [0, 1], 513, 2),
    "gqa2-dh64-L0": (dict(n_layers=2, d_model=512, n_heads=8, n_kv_heads=4, d_head=64, d_ffn=1000,
                          head_ranges=((0, 2), (2, 8)), ffn_ranges=((0, 9), (9, 1000)), model_id=99), [0, 1], 0, 3),
    "d5120-1way": (dict(n_layers=1, d_model=5120, n_heads=40, n_kv_heads=40, d_head=128, d_ffn=1024,
                        head_ranges=((0, 40),), ffn_ranges=((0, 1024),), model_id=100), [0], 100, 2),
}


@pytest.mark.parametrize("name", list(SHAPES))
def test_fused_token_matches_oracle(vtlib, name):
    kw, layers, L0, steps = SHAPES[name]
    wl = synthetic.small(name, kv_len=L0, decode_steps=steps, prompt_len=0, **kw)
    got, ref, fused = run_tokens(vtlib, wl, layers, L0, steps, vtlib.vt_decode_token)
    assert fused[0], fused[1]
    for t in range(steps):
        assert_close(got[t], ref[t], f"{name} token {t}")


@pytest.mark.parametrize("name", ["mha-dh64-uneven-empty", "gqa4-dh128"])
def test_sharded_token_matches_oracle(vtlib, name):
    kw, layers, L0, steps = SHAPES[name]
    wl = synthetic.small(name, kv_len=L0, decode_steps=steps, prompt_len=0, **kw)
    got, ref, _ = run_tokens(vtlib, wl, layers, L0, steps, vtlib.vt_decode_token_sharded)
    for t in range(steps):
        assert_close(got[t], ref[t], f"{name} sharded token {t}")


def test_fused_token_eager_calls(vtlib):
    """Without a graph: consecutive eager calls advance the device lengths themselves."""
    kw, layers, L0, steps = SHAPES["mha-dh64-uneven-empty"]
    wl = synthetic.small("eager", kv_len=L0, decode_steps=steps, prompt_len=0, **kw)
    got, ref, _ = run_tokens(vtlib, wl, layers, L0, steps, vtlib.vt_decode_token, graph=False)
    for t in range(steps):
        assert_close(got[t], ref[t], f"eager token {t}")


@pytest.mark.parametrize("cid", [2, 3, 5])
def test_fused_token_full_size_layer(vtlib, cid):
    """One full-size layer of the 7B, 13B (uneven 3-way) and 8B-GQA models at the workload's KV
    length: the fused kernel is available for the partition and matches the oracle."""
    wl = synthetic.WORKLOADS[cid]
    got, ref, fused = run_tokens(vtlib, wl, [wl.n_layers - 1], wl.kv_len, 2, vtlib.vt_decode_token)
    assert fused[0], fused[1]
    for t in range(2):
        assert_close(got[t], ref[t], f"{wl.name} fused token {t}")


def test_fused_and_sharded_agree_and_repeat(vtlib):
    """Same inputs through both entry points: the outputs agree within the parity tolerance, and
    the fused kernel repeats itself to within fp32 rounding of the atomically summed FFN partials."""
    kw, layers, L0, steps = SHAPES["mha-dh128-3way"]
    wl = synthetic.small("agree", kv_len=L0, decode_steps=steps, prompt_len=0, **kw)
    a, ref, _ = run_tokens(vtlib, wl, layers, L0, 2, vtlib.vt_decode_token, stream_id=90)
    b, _, _ = run_tokens(vtlib, wl, layers, L0, 2, vtlib.vt_decode_token_sharded, stream_id=90)
    c, _, _ = run_tokens(vtlib, wl, layers, L0, 2, vtlib.vt_decode_token, stream_id=90)
    for t in range(2):
        assert_close(a[t], b[t], f"fused vs sharded token {t}")
        d = np.abs(a[t].astype(np.float64) - c[t].astype(np.float64))
        assert d.max() <= 2e-3, f"fused run-to-run difference {d.max():.3e}"


# ------------------------------------------------------------------ partials of the fused kernel

def _one_layer_token_with_small_residual(vt, wl, layer, L0, scale=1e-3, stream_id=130):
    """One token through one layer with the input residual scaled down (x ~ N(0, scale^2)): the
    RMSNorm undoes the scale, so the partials keep their size while the residual they are added to
    becomes small, and an error in a partial is no longer hidden by the fp16 rounding of the
    residual.  Returns the GPU's x_out and fp32 partials of both blocks, and the oracle's."""
    from tests.test_gpu_decode import build as build_stack, write_cache
    cap = L0 + 8
    w = wl.layer_weights(layer)
    kc, vc = wl.kv_fill(layer, L0, cap) if L0 > 0 else oracle.new_cache(wl, cap)
    x = (wl.hidden(1, stream=stream_id).astype(np.float32) * scale).astype(np.float16)
    n = len(wl.head_ranges)
    with build_stack(vt, wl, layer_ids=[layer], capacity=cap) as st:
        write_cache(vt, st, 0, wl, kc, vc, L0, wl.head_ranges)
        vt.vt_kv_set_length(st.kv, -1, L0)
        fused = vt.vt_decode_token_fused_available(st.part)
        assert fused[0], fused[1]
        xout = torch.empty(wl.d_model, dtype=torch.float16, device="cuda")
        vt.vt_decode_token(st.part, st.kv, dev(x.reshape(-1)), xout)
        got_attn = vt.vt_token_partials_read(st.part, vt.VT_BLOCK_ATTN, n, wl.d_model)
        got_ffn = vt.vt_token_partials_read(st.part, vt.VT_BLOCK_FFN, n, wl.d_model)
        got_out = host(xout)
        assert vt.vt_kv_status(st.kv) == 0
    h_ref, ap = oracle.tp_attention(wl, w, x.reshape(1, -1), L0, kc, vc)
    xn_ref, fp = oracle.tp_ffn(wl, w, h_ref)
    return x, got_out, got_attn, got_ffn, h_ref, xn_ref, ap, fp


def _check_partials(wl, got_out, got_attn, got_ffn, x, h_ref, xn_ref, ap, fp, tag):
    n = len(wl.head_ranges)
    for d in range(n):
        h0, h1 = wl.head_ranges[d]
        if h1 > h0:
            assert_close(got_attn[d], ap[d].reshape(-1), f"{tag} fused ATTN partial dev {d}")
        c0, c1 = wl.ffn_ranges[d]
        if c1 > c0:
            assert_close(got_ffn[d], fp[d].reshape(-1), f"{tag} fused FFN partial dev {d}")
    # h from the kernel's own ATTN partials (the combine it performs: residual + partials in
    # shard order, one fp16 rounding) against the oracle's h
    used = [got_attn[d].astype(np.float64) for d in range(n) if wl.head_ranges[d][1] > wl.head_ranges[d][0]]
    h_gpu = oracle.combine(used, x.reshape(1, -1))
    assert_close(h_gpu, h_ref, f"{tag} h")
    # with the residual scaled down, x_out is dominated by the partials
    resid = np.sqrt(np.mean(x.astype(np.float64) ** 2))
    assert resid < 0.05 * np.sqrt(np.mean(xn_ref.astype(np.float64) ** 2))
    assert_close(got_out, xn_ref.reshape(-1), f"{tag} x_out")


@pytest.mark.parametrize("name", list(SHAPES))
def test_fused_token_partials_with_small_residual(vtlib, name):
    kw, layers, L0, steps = SHAPES[name]
    wl = synthetic.small(name, kv_len=L0, decode_steps=steps, prompt_len=0, **kw)
    r = _one_layer_token_with_small_residual(vtlib, wl, layers[-1], L0)
    x, got_out, got_attn, got_ffn, h_ref, xn_ref, ap, fp = r
    _check_partials(wl, got_out, got_attn, got_ffn, x, h_ref, xn_ref, ap, fp, name)


@pytest.mark.parametrize("cid", [2, 3, 5])
def test_fused_token_partials_full_size_layer(vtlib, cid):
    """The benchmarked kernel's fp32 shard partials at full width (7B 4-way, 13B uneven 3-way,
    8B GQA 4-way, at the workloads' KV lengths), with a small residual so x_out shows them."""
    wl = synthetic.WORKLOADS[cid]
    r = _one_layer_token_with_small_residual(vtlib, wl, wl.n_layers - 1, wl.kv_len, stream_id=140 + cid)
    x, got_out, got_attn, got_ffn, h_ref, xn_ref, ap, fp = r
    _check_partials(wl, got_out, got_attn, got_ffn, x, h_ref, xn_ref, ap, fp, wl.name)


def test_capture_leaves_the_host_length_mirror(vtlib):
    """Capturing vt_decode_token records device work only: with room for exactly one more token,
    an eager token after the capture is accepted (a capture that had advanced the host mirror would
    make it fail the capacity check), and the next one is refused before any launch."""
    vt = vtlib
    kw, layers, L0, steps = SHAPES["mha-dh64-uneven-empty"]
    wl = synthetic.small("capture", kv_len=L0, decode_steps=1, prompt_len=0, **kw)
    cap = L0 + 1
    with build(vt, wl, layer_ids=[0], capacity=cap) as st:
        kc, vc = wl.kv_fill(0, L0, cap)
        write_cache(vt, st, 0, wl, kc, vc, L0, wl.head_ranges)
        vt.vt_kv_set_length(st.kv, -1, L0)
        xin = dev(wl.hidden(1, stream=150).reshape(-1))
        xout = torch.empty_like(xin)
        g = torch.cuda.CUDAGraph()
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(s):
            with torch.cuda.graph(g, stream=s):
                vt.vt_decode_token(st.part, st.kv, xin, xout, stream=s)
        torch.cuda.current_stream().wait_stream(s)
        vt.vt_decode_token(st.part, st.kv, xin, xout)
        with pytest.raises(vt.VtError) as e:
            vt.vt_decode_token(st.part, st.kv, xin, xout)
        assert e.value.status == vt.VT_ERR_KV_CAPACITY
        assert vt.vt_kv_length(st.kv, 0) == L0 + 1
        assert vt.vt_kv_status(st.kv) == 0
        del g


# ------------------------------------------------------------------ bounded waits

@pytest.mark.parametrize("cta", [0, -2])
def test_grid_barrier_wait_gives_up_and_the_next_token_runs_clean(vtlib, cta):
    """The fused kernel's grid-barrier waits are bounded.  One CTA (the first, or the last of the
    grid) is made to skip its arrival at the token's first barrier and the poll limit is cut to a
    few thousand: every CTA gives up, the kernel returns (no hang), and the KV status word reports
    VT_DEV_WAIT_TIMEOUT to the host.  After the status is cleared (which also removes the test
    settings) the same token, from the same KV length, runs clean and equals the first clean run."""
    vt = vtlib
    kw, layers, L0, steps = SHAPES["mha-dh128-3way"]
    wl = synthetic.small("timeout", kv_len=L0, decode_steps=1, prompt_len=0, **kw)
    cap = L0 + 4
    with build(vt, wl, layer_ids=layers, capacity=cap) as st:
        for i, layer in enumerate(layers):
            kc, vc = wl.kv_fill(layer, L0, cap)
            write_cache(vt, st, i, wl, kc, vc, L0, wl.head_ranges)
        fused, why = vt.vt_decode_token_fused_available(st.part)
        assert fused, why
        xin = dev(wl.hidden(1, stream=160).reshape(-1))
        xout = torch.empty_like(xin)

        vt.vt_kv_set_length(st.kv, -1, L0)
        vt.vt_decode_token(st.part, st.kv, xin, xout)
        clean = host(xout).copy()
        assert vt.vt_kv_status(st.kv) == 0

        # the grid size is the partition's; -2 picks the last CTA through the hook's range check
        target = cta
        if cta < 0:
            target = 0
            while True:
                try:
                    vt.vt_token_test_barrier(st.part, target + 1, 4096)
                    target += 1
                except vt.VtError:
                    break
        vt.vt_token_test_barrier(st.part, target, 4096)
        vt.vt_kv_set_length(st.kv, -1, L0)
        xout.fill_(0)
        vt.vt_decode_token(st.part, st.kv, xin, xout)
        torch.cuda.synchronize()
        flags = vt.vt_kv_status(st.kv, clear=True)
        assert flags & vt.VT_DEV_WAIT_TIMEOUT, f"status {flags:#x}"
        assert vt.vt_kv_status(st.kv) == 0

        vt.vt_kv_set_length(st.kv, -1, L0)
        vt.vt_decode_token(st.part, st.kv, xin, xout)
        again = host(xout)
        assert vt.vt_kv_status(st.kv) == 0
        assert vt.vt_kv_length(st.kv, 0) == L0 + 1
        d = np.abs(again.astype(np.float64) - clean.astype(np.float64))
        assert d.max() <= 2e-3, f"clean run after the timeout differs by {d.max():.3e}"
        with pytest.raises(vt.VtError):
            vt.vt_token_test_barrier(st.part, -2, 0)
