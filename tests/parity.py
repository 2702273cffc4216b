"""Shared helpers of the GPU parity tests: tolerances, workload construction, oracle references."""
from __future__ import annotations

import numpy as np

import oracle
import synthetic

# Tolerance of every floating-point comparison against the oracle: relative RMS error at most 1e-3
# and largest absolute error at most 2e-2, per output tensor.
REL_RMS = 1e-3
MAX_ABS = 2e-2


def errors(got, ref):
    got = np.asarray(got, np.float64).reshape(-1)
    ref = np.asarray(ref, np.float64).reshape(-1)
    d = got - ref
    rel = float(np.sqrt(np.mean(d * d)) / max(np.sqrt(np.mean(ref * ref)), 1e-30))
    return rel, float(np.max(np.abs(d))) if d.size else 0.0


def assert_close(got, ref, what: str, rel_rms: float = REL_RMS, max_abs: float = MAX_ABS):
    got = np.asarray(got)
    assert np.all(np.isfinite(got)), f"{what}: non-finite values"
    rel, mx = errors(got, ref)
    assert rel <= rel_rms and mx <= max_abs, f"{what}: rel-RMS {rel:.3e}, max-abs {mx:.3e}"
    return rel, mx


def shapes_of(vt, wl, max_seq=None):
    return vt.make_shapes(wl.n_layers, wl.d_model, wl.n_heads, wl.n_kv_heads, wl.d_head, wl.d_ffn,
                          wl.vocab, wl.max_seq if max_seq is None else max_seq, wl.rms_eps,
                          wl.rope_theta)


def kv_range(wl, heads):
    g = wl.n_heads // wl.n_kv_heads
    return heads[0] // g, heads[1] // g
