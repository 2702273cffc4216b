"""Decode parity at the full sizes of the workloads (7B MHA 4-way, 13B uneven 3-way, 8B GQA 4-way).

Each test loads the first and the last layer of the model at full width, fills their KV caches
with the seeded synthetic cache at the workload's length, and checks one teacher-forced decode
token per layer (every shard's partial, both combines and the appended K/V rows) against the CPU
oracle.  The last test runs the whole-token entry point (vt_decode_token) captured in a CUDA graph,
the launch configuration the benchmark times, over a two-layer 7B-shaped stack for two tokens.
"""
from __future__ import annotations

import numpy as np
import pytest

import oracle
import synthetic
from tests.parity import assert_close
from tests.test_gpu_decode import build, decode_layer_check, dev, host, write_cache

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


def _full_layer_checks(vt, wl, layers, lengths):
    cap = max(lengths) + 8
    with build(vt, wl, layer_ids=layers, capacity=cap) as st:
        for i, layer in enumerate(layers):
            w = wl.layer_weights(layer)
            for L in lengths:
                kc, vc = wl.kv_fill(layer, L, cap)
                write_cache(vt, st, i, wl, kc, vc, L, wl.head_ranges)
                vt.vt_kv_set_length(st.kv, i, L)
                x = wl.hidden(1, stream=40 + 7 * layer + L % 5)
                decode_layer_check(vt, st, wl, w, i, x, L, kc, vc, wl.head_ranges,
                                   wl.ffn_ranges, f"{wl.name} layer {layer} L={L}")
        assert vt.vt_kv_status(st.kv) == 0 and vt.vt_partition_status(st.part) == 0


def test_7b_decode_first_and_last_layer_at_both_ends_of_the_schedule(vtlib):
    """Llama-2-7B shapes, even 4-way; KV length 1024 (first step) and 1151 (last of 128)."""
    wl = synthetic.WORKLOADS[2]
    _full_layer_checks(vtlib, wl, [0, wl.n_layers - 1], [wl.kv_len, wl.kv_len + wl.decode_steps - 1])


def test_13b_decode_uneven_three_way(vtlib):
    """Llama-2-13B shapes, heads 20/12/8 and FFN columns 6912/4147/2765, KV length 2048."""
    wl = synthetic.WORKLOADS[3]
    _full_layer_checks(vtlib, wl, [0, wl.n_layers - 1], [wl.kv_len])


def test_8b_gqa_decode_at_kv_4096(vtlib):
    """Llama-3-8B shapes (32 query / 8 KV heads, 2 KV heads per shard), KV length 4096."""
    wl = synthetic.WORKLOADS[5]
    _full_layer_checks(vtlib, wl, [0, wl.n_layers - 1], [wl.kv_len])


def test_7b_decode_token_graph_two_layer_stack(vtlib):
    """vt_decode_token over layers 0 and 31 of the 7B-shaped model, captured once as a CUDA graph
    and replayed for two tokens (positions advance on the device), against the oracle chained
    through the same two layers."""
    wl = synthetic.WORKLOADS[2]
    layers = [0, wl.n_layers - 1]
    L0, steps = wl.kv_len, 2
    cap = L0 + steps + 8
    D = wl.d_model
    ws = [wl.layer_weights(l) for l in layers]
    caches = []
    with build(vtlib, wl, layer_ids=layers, capacity=cap) as st:
        for i, layer in enumerate(layers):
            kc, vc = wl.kv_fill(layer, L0, cap)
            caches.append((kc, vc))
            write_cache(vtlib, st, i, wl, kc, vc, L0, wl.head_ranges)
        vtlib.vt_kv_set_length(st.kv, -1, L0)
        xin = torch.empty(D, dtype=torch.float16, device="cuda")
        xout = torch.empty(D, dtype=torch.float16, device="cuda")
        g = torch.cuda.CUDAGraph()
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(s):
            with torch.cuda.graph(g, stream=s):
                vtlib.vt_decode_token(st.part, st.kv, xin, xout, stream=s)
        torch.cuda.current_stream().wait_stream(s)
        # the capture recorded device work only: the device lengths and the host mirror are still L0
        assert vtlib.vt_kv_length(st.kv, 0) == L0
        for t in range(steps):
            x = wl.hidden(1, stream=60 + t)
            xin.copy_(dev(x.reshape(-1)))
            g.replay()
            ref = x.reshape(1, -1)
            for i in range(len(layers)):
                _, ref, _, _ = oracle.tp_layer(wl, ws[i], ref, L0 + t, *caches[i])
            assert_close(host(xout), ref.reshape(-1), f"7b graph step {t}")
        torch.cuda.synchronize()
        assert vtlib.vt_kv_status(st.kv) == 0
        for i in range(len(layers)):
            k0, k1 = 0, wl.n_kv_heads // len(wl.head_ranges)
            kg, vg = vtlib.vt_kv_read(st.kv, i, 0, L0 + steps, k1 - k0, wl.d_head)
            assert np.array_equal(kg[:, :L0], caches[i][0][k0:k1, :L0])
            assert_close(kg[:, L0:L0 + steps], caches[i][0][k0:k1, L0:L0 + steps], "k rows")
            assert_close(vg[:, L0:L0 + steps], caches[i][1][k0:k1, L0:L0 + steps], "v rows")
