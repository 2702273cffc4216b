"""Sliding-window attention in the oracle (Voltron Section 2.1 lists SWA among the attention
variants of the evaluated models; the kernels for it are a next step).  Row i at position p
attends to positions [max(0, p - W + 1), p].

Pins: PyTorch's scaled_dot_product_attention with the banded causal mask (tests/torch_reference.py),
a window that covers every position equals full attention, and a window of one returns the
projected value of the row's own position.  CPU only."""
from __future__ import annotations

import numpy as np
import pytest

import oracle
import synthetic
from tests import torch_reference


def rel(a, b):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300))


def filled(wl, w, x, cap):
    """Caches with the rows of x appended at positions 0..rows-1 (every KV head)."""
    kc, vc = oracle.new_cache(wl, cap)
    oracle.kv_append(wl, w, (0, wl.n_kv_heads), x, 0, kc, vc)
    return kc, vc


@pytest.mark.parametrize("window", [1, 3, 5, 9, 40])
@pytest.mark.parametrize("kw", [dict(), dict(n_kv_heads=4)])
def test_window_matches_banded_torch_attention(window, kw):
    wl = synthetic.small("swa", **kw)
    w = wl.layer_weights(0)
    rows = 9
    x = wl.hidden(rows, stream=31)
    kc, vc = filled(wl, w, x, 16)
    got = oracle.attn_partial(wl, w, (0, wl.n_heads), x, np.arange(rows), kc, vc, window=window)
    ref = torch_reference.layer(wl, w, x, 0, None, None, window=window)["attn_out"]
    assert rel(got, ref) < 1e-12


def test_window_covering_every_position_is_full_attention():
    wl = synthetic.small("swa-full")
    w = wl.layer_weights(0)
    rows = 7
    x = wl.hidden(rows, stream=32)
    kc, vc = filled(wl, w, x, 8)
    pos = np.arange(rows)
    full = oracle.attn_partial(wl, w, (0, wl.n_heads), x, pos, kc, vc)
    for window in (rows, rows + 5):
        assert np.array_equal(oracle.attn_partial(wl, w, (0, wl.n_heads), x, pos, kc, vc, window=window), full)
    assert not np.array_equal(oracle.attn_partial(wl, w, (0, wl.n_heads), x, pos, kc, vc, window=2), full)


def test_window_of_one_returns_the_rows_own_value():
    """softmax over one position is 1: the partial is Wo[:, heads] . v(own position) per head."""
    wl = synthetic.small("swa-one", n_heads=8, n_kv_heads=4, head_ranges=((0, 8),), d_model=128)
    w = wl.layer_weights(0)
    rows = 5
    x = wl.hidden(rows, stream=33)
    kc, vc = filled(wl, w, x, 8)
    h0, h1 = 2, 6
    got = oracle.attn_partial(wl, w, (h0, h1), x, np.arange(rows), kc, vc, window=1)
    g = wl.n_heads // wl.n_kv_heads
    dh = wl.d_head
    wo = w["wo"].astype(np.float64)
    for i in range(rows):
        o = np.concatenate([vc[h // g, i].astype(np.float64) for h in range(h0, h1)])
        want = wo[:, h0 * dh:h1 * dh] @ o
        assert rel(got[i], want) < 1e-13
