"""Free-running whole-stack decode of the 7B-shaped model (all 32 layers, even 4-way) for three
tokens: the GPU feeds each layer its own fp16 output, the oracle its own.  Binding parity is per
layer and teacher-forced (the other tests); here the deviation accumulated over 32 layers of fp16
hidden states is measured and bounded loosely, and printed so it can be reported.
"""
from __future__ import annotations

import numpy as np
import pytest

import oracle
import synthetic
from tests.parity import errors
from tests.test_gpu_decode import build, dev, host, write_cache

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


def test_7b_free_running_32_layers_three_tokens(vtlib, capsys):
    vt = vtlib
    wl = synthetic.WORKLOADS[2]
    L0, steps = wl.kv_len, 3
    cap = L0 + steps + 5
    ws = [wl.layer_weights(l) for l in range(wl.n_layers)]
    caches = [wl.kv_fill(l, L0, cap) for l in range(wl.n_layers)]
    from paper_2607_07046_gb300.stack import Stack
    from tests.parity import shapes_of
    shapes = shapes_of(vt, wl, max_seq=max(wl.max_seq, cap))
    report = []
    with Stack(shapes, lambda l: ws[l], wl.head_ranges, wl.ffn_ranges, cap) as st:
        for l in range(wl.n_layers):
            write_cache(vt, st, l, wl, caches[l][0], caches[l][1], L0, wl.head_ranges)
        vt.vt_kv_set_length(st.kv, -1, L0)
        xout = torch.empty(wl.d_model, dtype=torch.float16, device="cuda")
        for t in range(steps):
            x = wl.hidden(1, stream=180 + t)
            vt.vt_decode_token(st.part, st.kv, dev(x.reshape(-1)), xout)
            r = x.reshape(1, -1)
            for l in range(wl.n_layers):
                _, r, _, _ = oracle.tp_layer(wl, ws[l], r, L0 + t, *caches[l])
            rel, mx = errors(host(xout), r)
            report.append((t, rel, mx))
        assert vt.vt_kv_status(st.kv) == 0
    with capsys.disabled():
        for t, rel, mx in report:
            print(f"\n7B free-running 32 layers, token {t}: rel-RMS {rel:.3e}, max-abs {mx:.3e}")
    for t, rel, mx in report:
        assert np.isfinite(rel) and rel <= 1e-2, (t, rel, mx)
