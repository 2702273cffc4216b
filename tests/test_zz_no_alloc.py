"""vt_decode_step_static (the ATTN decode step whose scratch is a fixed device array) against
vt_decode_step, through the C ABI, on two decode tokens in a row.

The file name sorts last so that the static-scratch step also runs after every other GPU test in
the same process; it must pass alone as well.  The two entry points share the QKV and O kernels and
differ in how the attention slices merge, so partials agree to fp32 rounding and the appended KV
rows agree bit for bit.
"""
from __future__ import annotations

import dataclasses

import numpy as np
import pytest

import synthetic
from tests.parity import kv_range, shapes_of

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

ATTN, FFN = 0, 1


# The first static call in a process looks the array's address up, which loads the library's
# module that holds it (the CUDA loader then places the array in device memory).  Every later call
# must leave free device memory exactly as it found it.
_setup_done = []


def _stack(vt, wl, capacity):
    from paper_2607_07046_gb300.stack import Stack
    return Stack(shapes_of(vt, wl, max_seq=max(wl.max_seq, capacity)), wl.layer_weights,
                 wl.head_ranges, wl.ffn_ranges, capacity)


def _fill(vt, st, wl, L):
    for l in range(wl.n_layers):
        kc, vc = wl.kv_fill(l, L)
        for d, hr in enumerate(wl.head_ranges):
            k0, k1 = kv_range(wl, hr)
            if k1 > k0:
                vt.vt_kv_write_raw(st.kv, l, d, kc[k0:k1], vc[k0:k1])
    vt.vt_kv_set_length(st.kv, -1, L)


def _gqa(name, n_heads, n_kv_heads):
    return synthetic.small(name, n_layers=1, d_model=512, n_heads=n_heads, n_kv_heads=n_kv_heads, d_head=64,
                           d_ffn=256, head_ranges=((0, n_heads // 2), (n_heads // 2, n_heads)),
                           ffn_ranges=((0, 128), (128, 256)), kv_len=20, decode_steps=2, prompt_len=0, model_id=150)


CASES = [
    # (workload, cached positions before the first token): 2-way MHA with dh 64 and a length that
    # leaves ragged slices; one layer of the 8B GQA model (4 query heads per KV head, dh 128);
    # 8 and 2 query heads per KV head at lengths that leave most of the 16 slices empty (the
    # merge then weighs empty slices by zero).
    ("tiny", lambda: synthetic.WORKLOADS[1], 100),
    ("8b-gqa", lambda: dataclasses.replace(synthetic.WORKLOADS[5], n_layers=1), 300),
    ("gqa8-L0", lambda: _gqa("gqa8", 16, 2), 0),
    ("gqa8-L1", lambda: _gqa("gqa8", 16, 2), 1),
    ("gqa2-L15", lambda: _gqa("gqa2", 8, 4), 15),
    ("gqa2-L17", lambda: _gqa("gqa2", 8, 4), 17),
]


@pytest.mark.parametrize("name,make,L", CASES, ids=[c[0] for c in CASES])
def test_static_step_matches_decode_step_on_two_tokens(vtlib, name, make, L):
    vt = vtlib
    wl = make()
    D = wl.d_model
    with _stack(vt, wl, L + 8) as st:
        _fill(vt, st, wl, L)
        xs = wl.hidden(2, stream=7)
        for t in range(2):
            x = torch.from_numpy(xs[t].copy()).cuda()
            for d, hr in enumerate(wl.head_ranges):
                ref = torch.full((D,), float("nan"), dtype=torch.float32, device="cuda")
                got = torch.full((D,), float("nan"), dtype=torch.float32, device="cuda")
                vt.vt_decode_step(st.part, (0, d, ATTN), x, st.kv, ref)
                torch.cuda.synchronize()
                k0, k1 = kv_range(wl, hr)
                kv_ref = vt.vt_kv_read(st.kv, 0, d, L + t + 1, k1 - k0, wl.d_head) if k1 > k0 else None
                free0 = torch.cuda.mem_get_info()[0]
                vt.vt_decode_step_static(st.part, (0, d, ATTN), x, st.kv, got)
                torch.cuda.synchronize()
                if _setup_done:
                    assert torch.cuda.mem_get_info()[0] == free0, "the static step changed free device memory"
                _setup_done.append(True)
                r, g = ref.cpu().numpy(), got.cpu().numpy()
                assert np.isfinite(g).all()
                scale = max(float(np.abs(r).max()), 1e-30)
                err = float(np.abs(g - r).max())
                assert err <= 1e-5 * scale + 1e-7, f"{name} token {t} device {d}: max |diff| {err:.3e} (scale {scale:.3e})"
                if kv_ref is not None:
                    kv_got = vt.vt_kv_read(st.kv, 0, d, L + t + 1, k1 - k0, wl.d_head)
                    assert np.array_equal(kv_got[0], kv_ref[0]) and np.array_equal(kv_got[1], kv_ref[1])
            vt.vt_kv_advance(st.kv, -1, 1)
        flags = vt.vt_kv_status(st.kv, clear=True)
        assert flags == 0, flags


def test_static_step_rejects_ffn_shards_and_oversized_shards(vtlib):
    vt = vtlib
    wl = synthetic.WORKLOADS[1]
    with _stack(vt, wl, 16) as st:
        x = torch.zeros(wl.d_model, dtype=torch.float16, device="cuda")
        out = torch.zeros(wl.d_model, dtype=torch.float32, device="cuda")
        with pytest.raises(vt.VtError, match="ATTN shards only"):
            vt.vt_decode_step_static(st.part, (0, 0, FFN), x, None, out)
    # 128 KV heads on one device: more than the array's 64 arrival counters and 1 MiB
    big = synthetic.small("wide", n_layers=1, d_model=64, n_heads=128, n_kv_heads=128, d_head=128,
                          d_ffn=64, head_ranges=((0, 128),), ffn_ranges=((0, 64),), kv_len=4)
    with _stack(vt, big, 16) as st:
        x = torch.zeros(big.d_model, dtype=torch.float16, device="cuda")
        out = torch.zeros(big.d_model, dtype=torch.float32, device="cuda")
        with pytest.raises(vt.VtError, match="bytes of static scratch"):
            vt.vt_decode_step_static(st.part, (0, 0, ATTN), x, st.kv, out)
