"""Block quantization of weight shards (Voltron Sections 3.2.2 and 4.2.2, precision heterogeneity;
Section 5.1 uses k-quant formats without defining them).  Reading: per row, blocks of 32 weights,
fp16 scale d = fp16(amax / qmax) (qmax 127 for INT8, 7 for INT4), codes round-half-even(w / d)
clamped to [-qmax, qmax], decisions in fp32.

The oracle's quantizer is pinned to closed forms of that definition (exact power-of-two grids,
ties to even, the zero block, a subnormal scale that needs the clamp, the d / 2 error bound), its
dequantized matrix-vector product to numpy, and the library's own quantizer must give the same
codes and scales bit for bit.  CPU only."""
from __future__ import annotations

import numpy as np
import pytest

import oracle
import synthetic


def f16(a):
    return np.asarray(a, dtype=np.float16)


@pytest.mark.parametrize("bits,qmax", [(8, 127), (4, 7)])
def test_power_of_two_grid_returns_its_integers(bits, qmax):
    """Weights i * 2^-8 for i in [-qmax, qmax]: amax / qmax = 2^-8 exactly, so d = 2^-8 and every
    code is i."""
    i = np.arange(-qmax, qmax + 1)
    w = f16(i * 2.0 ** -8)[None, :]
    q, d = oracle.quantize_rows(w, bits, block=w.shape[1])
    assert d[0, 0] == np.float16(2.0 ** -8)
    assert np.array_equal(q[0], i.astype(np.int8))


def test_ties_round_to_even():
    """d = 2^-8 (the block's max is 127 * 2^-8); w = +-2.5 d, +-3.5 d, +-0.5 d sit exactly halfway."""
    d = 2.0 ** -8
    w = f16([127 * d, 2.5 * d, -2.5 * d, 3.5 * d, -3.5 * d, 0.5 * d, -0.5 * d, 1.5 * d])[None, :]
    q, sc = oracle.quantize_rows(w, 8, block=8)
    assert sc[0, 0] == np.float16(d)
    assert q[0].tolist() == [127, 2, -2, 4, -4, 0, 0, 2]


def test_zero_block_and_vanishing_scale():
    """A zero block has d = 0 and codes 0; so does a block whose scale rounds to zero in fp16
    (amax = 2^-20: amax / 127 is below half the smallest subnormal)."""
    w = f16([[0.0] * 32 + [2.0 ** -20, -2.0 ** -21] + [0.0] * 30])
    q, sc = oracle.quantize_rows(w, 8, block=32)
    assert sc[0].tolist() == [0.0, 0.0]
    assert not q.any()


def test_subnormal_scale_needs_the_clamp():
    """amax = 2^-15: amax / 127 = 2.40e-7 rounds to the subnormal 4 * 2^-24, so amax / d = 128,
    clamped to 127; 2^-16 gives 64."""
    w = f16([[2.0 ** -15, -(2.0 ** -15), 2.0 ** -16, 0.0]])
    q, sc = oracle.quantize_rows(w, 8, block=4)
    assert sc[0, 0] == np.float16(4 * 2.0 ** -24)
    assert q[0].tolist() == [127, -127, 64, 0]


@pytest.mark.parametrize("bits,qmax", [(8, 127), (4, 7)])
def test_error_bound_and_extremes(bits, qmax):
    """|w - q d| <= d / 2 for every weight (the scales here are normal fp16, so no clamp acts), the
    block maximum maps to +-qmax, and negating the weights negates the codes."""
    rng = np.random.default_rng(3 + bits)
    w = f16(rng.standard_normal((64, 96)) * np.exp(rng.uniform(-3, 3, (64, 1))))
    q, sc = oracle.quantize_rows(w, bits, block=32)
    d = np.repeat(sc.astype(np.float64), 32, axis=1)
    err = np.abs(w.astype(np.float64) - q.astype(np.float64) * d)
    assert np.all(err <= d / 2 * (1 + 1e-6) + 1e-30)
    blocks = np.abs(w.astype(np.float64)).reshape(64, 3, 32)
    arg = blocks.argmax(axis=2)
    for r in range(64):
        for b in range(3):
            assert abs(int(q[r, b * 32 + arg[r, b]])) == qmax
    qn, scn = oracle.quantize_rows(-w, bits, block=32)
    assert np.array_equal(qn, -q) and np.array_equal(scn, sc)


def test_ragged_last_block():
    w = f16(np.linspace(-1, 1, 70))[None, :]
    q, sc = oracle.quantize_rows(w, 8, block=32)
    assert sc.shape == (1, 3)
    q6, sc6 = oracle.quantize_rows(w[:, 64:], 8, block=32)
    assert np.array_equal(q[:, 64:], q6) and sc[0, 2] == sc6[0, 0]


def test_dequantized_gemv_equals_numpy():
    rng = np.random.default_rng(11)
    w = f16(rng.standard_normal((33, 200)) * 0.02)
    x = rng.standard_normal(200)
    for bits in (8, 4):
        q, sc = oracle.quantize_rows(w, bits, block=32)
        deq = q.astype(np.float64) * np.repeat(sc.astype(np.float64), 32, axis=1)[:, :200]
        assert np.allclose(oracle.gemv_blockq(q, sc, x), deq @ x, rtol=1e-13, atol=1e-15)


@pytest.mark.parametrize("bits", [8, 4])
@pytest.mark.parametrize("shape,block", [((37, 1000), 32), ((5, 31), 32), ((3, 4096), 32), ((9, 100), 16)])
def test_library_quantizer_matches_the_oracle_bit_for_bit(vtlib, bits, shape, block):
    rng = np.random.default_rng(sum(shape) + bits)
    w = rng.standard_normal(shape) * np.exp(rng.uniform(-8, 8, (shape[0], 1)))
    w = np.clip(w, -65504, 65504).astype(np.float16)
    w[0, : min(8, shape[1])] = 0.0                      # part of a zero block
    if shape[0] > 1:
        w[1] = f16(rng.standard_normal(shape[1]) * 2.0 ** -16)   # subnormal scales
    q1, s1 = oracle.quantize_rows(w, bits, block)
    q2, s2 = vtlib.vt_quantize_rows(w, bits, block)
    assert np.array_equal(q1, q2)
    assert np.array_equal(s1.view(np.uint16), s2.view(np.uint16))


def test_library_quantizer_rejects_bad_arguments(vtlib):
    w = np.zeros((2, 8), np.float16)
    for bits, block in ((5, 32), (8, 0), (0, 32)):
        with pytest.raises(vtlib.VtError) as e:
            vtlib.vt_quantize_rows(w, bits, block)
        assert e.value.status == vtlib.VT_ERR_INVALID_ARG


# ------------------------------------------------------------------ quantized partials (Section 4.3.2)

@pytest.mark.parametrize("bits,qmax", [(8, 127), (4, 7)])
def test_partial_grid_and_ties(bits, qmax):
    """fp32 partials on the grid i * 2^-6 return their integers; halfway values round to even."""
    i = np.arange(-qmax, qmax + 1)
    q, sc = oracle.quantize_vec((i * 2.0 ** -6).astype(np.float32), bits, block=i.size)
    assert sc[0] == np.float16(2.0 ** -6) and np.array_equal(q, i.astype(np.int8))
    d = 2.0 ** -6
    x = np.array([qmax * d, 2.5 * d, -2.5 * d, 1.5 * d, -0.5 * d], np.float32)
    q, _ = oracle.quantize_vec(x, bits, block=5)
    assert q.tolist() == [qmax, 2, -2, 2, 0]


def test_partial_error_bound_and_zero_partial():
    rng = np.random.default_rng(21)
    x = (rng.standard_normal(4096) * 3.0).astype(np.float32)
    for bits in (8, 4):
        q, sc = oracle.quantize_vec(x, bits, block=32)
        d = np.repeat(sc.astype(np.float64), 32)
        assert np.all(np.abs(x.astype(np.float64) - q * d) <= d / 2 * (1 + 1e-6))
    q, sc = oracle.quantize_vec(np.zeros(70, np.float32), 8, block=32)
    assert not q.any() and not sc.astype(np.float64).any()


def test_quantized_combine_equals_numpy_and_stays_within_the_bound():
    """The combine of quantized partials is binary16(residual + sum of q * d) (numpy, fp64 sums,
    round to nearest even), and differs from the unquantized combine by at most the partials'
    half-steps plus the output's rounding."""
    rng = np.random.default_rng(22)
    D, n = 512, 3
    parts = [(rng.standard_normal(D) * 0.5).astype(np.float32) for _ in range(n)]
    res = rng.standard_normal(D).astype(np.float16)
    for bits in (8, 4):
        qp = [oracle.quantize_vec(p, bits) for p in parts]
        got = oracle.combine_q(qp, res)
        deq = [q.astype(np.float64) * np.repeat(s.astype(np.float64), 32) for q, s in qp]
        want = (res.astype(np.float64) + sum(deq)).astype(np.float16)
        assert np.array_equal(got.view(np.uint16), want.view(np.uint16))
        exact = res.astype(np.float64) + sum(p.astype(np.float64) for p in parts)
        half_steps = sum(np.repeat(s.astype(np.float64), 32) / 2 for _, s in qp)
        ulp = np.abs(exact) * 2.0 ** -10 + 2.0 ** -24
        assert np.all(np.abs(got.astype(np.float64) - exact) <= half_steps * (1 + 1e-6) + ulp)
    # no residual and one zero partial: the other partial alone
    z = oracle.quantize_vec(np.zeros(D, np.float32), 8)
    one = oracle.quantize_vec(parts[0], 8)
    assert np.array_equal(oracle.combine_q([z, one], None), oracle.combine_q([one], None))


# ------------------------------------------------------------------ quantized shards (oracle)

def _exact_layer(wl, bits, seed=7):
    """Weights that are exactly q * d in binary16: codes drawn in [-qmax, qmax], one power-of-two
    scale per block of 32 along each matrix's input axis.  Returns the binary16 weights and, per
    matrix, its full (codes, scales)."""
    rng = np.random.default_rng(seed)
    qmax = 127 if bits == 8 else 7
    shapes = {"wq": (wl.n_heads * wl.d_head, wl.d_model), "wk": (wl.n_kv_heads * wl.d_head, wl.d_model),
              "wv": (wl.n_kv_heads * wl.d_head, wl.d_model), "wo": (wl.d_model, wl.n_heads * wl.d_head),
              "w_gate": (wl.d_ffn, wl.d_model), "w_up": (wl.d_ffn, wl.d_model), "w_down": (wl.d_model, wl.d_ffn)}
    w, qd = {}, {}
    for name, (r, k) in shapes.items():
        q = rng.integers(-qmax, qmax + 1, size=(r, k)).astype(np.int8)
        e = rng.integers(6, 10, size=(r, (k + 31) // 32))
        d = np.ldexp(1.0, -e).astype(np.float16)
        deq = q.astype(np.float64) * np.repeat(d.astype(np.float64), 32, axis=1)[:, :k]
        w[name] = deq.astype(np.float16)
        assert np.array_equal(w[name].astype(np.float64), deq)  # exact in binary16
        qd[name] = (q, d)
    w["attn_norm"] = synthetic.normal_f16((wl.d_model,), 5, 1.0, 0.02)
    w["ffn_norm"] = synthetic.normal_f16((wl.d_model,), 6, 1.0, 0.02)
    return w, qd


def _slice_q(qd, name, rows=None, cols=None):
    q, d = qd[name]
    if rows is not None:
        return (q[rows[0]:rows[1]], d[rows[0]:rows[1]], 32)
    return (np.ascontiguousarray(q[:, cols[0]:cols[1]]), np.ascontiguousarray(d[:, cols[0] // 32:(cols[1] + 31) // 32]), 32)


@pytest.mark.parametrize("bits", [8, 4])
def test_quantized_shard_functions_equal_the_binary16_ones_on_exact_weights(bits):
    """When every weight is exactly its dequantized value, the quantized-shard attention, K/V append
    and FFN functions must give bit for bit what the binary16 functions give (same sums in the same
    order): this ties the quantized path to the pinned binary16 layer."""
    wl = synthetic.small("qexact", n_layers=1, d_model=128, n_heads=4, n_kv_heads=2, d_head=32, d_ffn=96,
                         head_ranges=((0, 2), (2, 4)), ffn_ranges=((0, 64), (64, 96)))
    w, qd = _exact_layer(wl, bits)
    dh, cap, L = wl.d_head, 16, 5
    x = wl.hidden(3, stream=1)
    for (h0, h1), (c0, c1) in zip(wl.head_ranges, wl.ffn_ranges):
        k0, k1 = oracle.kv_heads_of(wl, (h0, h1))
        qw = {"wq": _slice_q(qd, "wq", rows=(h0 * dh, h1 * dh)), "wk": _slice_q(qd, "wk", rows=(k0 * dh, k1 * dh)),
              "wv": _slice_q(qd, "wv", rows=(k0 * dh, k1 * dh)), "wo": _slice_q(qd, "wo", cols=(h0 * dh, h1 * dh)),
              "w_gate": _slice_q(qd, "w_gate", rows=(c0, c1)), "w_up": _slice_q(qd, "w_up", rows=(c0, c1)),
              "w_down": _slice_q(qd, "w_down", cols=(c0, c1))}
        kc1, vc1 = wl.kv_fill(0, L, cap)
        kc2, vc2 = kc1.copy(), vc1.copy()
        oracle.kv_append(wl, w, (k0, k1), x, L, kc1, vc1)
        oracle.kv_append_q(wl, w, (k0, k1), x, L, kc2, vc2, qw)
        assert np.array_equal(kc1, kc2) and np.array_equal(vc1, vc2)
        pos = np.arange(L, L + 3)
        for window in (0, 2):
            a = oracle.attn_partial(wl, w, (h0, h1), x, pos, kc1, vc1, window)
            b = oracle.attn_partial_q(wl, w, (h0, h1), x, pos, kc1, vc1, qw, window)
            assert np.array_equal(a, b)
        a = oracle.ffn_partial(wl, w, (c0, c1), x)
        b = oracle.ffn_partial_q(wl, w, (c0, c1), x, qw)
        assert np.array_equal(a, b)


def test_mixed_layer_with_all_binary16_shards_is_the_binary16_layer():
    wl = synthetic.small("qmix16", n_layers=1)
    w = wl.layer_weights(0)
    x = wl.hidden(2, stream=3)
    kc1, vc1 = oracle.new_cache(wl, 16)
    kc2, vc2 = oracle.new_cache(wl, 16)
    ref = oracle.tp_layer(wl, w, x, 0, kc1, vc1)
    got = oracle.tp_layer_mixed(wl, w, x, 0, kc2, vc2, [16, 16], [16, 16])
    assert np.array_equal(ref[1], got[1]) and np.array_equal(kc1, kc2)


@pytest.mark.parametrize("bits,bound", [(8, 2e-2), (4, 3e-1)])
def test_mixed_layer_error_is_that_of_the_weight_rounding(bits, bound):
    """Quantizing real binary16 weights moves the layer's partials by the quantization error only:
    the relative difference stays within a loose bound set by d / 2 per weight (INT8: ~1/254 of
    a block's largest weight; INT4: ~1/14), and shrinks from INT4 to INT8."""
    wl = synthetic.small("qmixerr", n_layers=1, d_model=128, n_heads=4, n_kv_heads=2, d_head=32, d_ffn=96,
                         head_ranges=((0, 2), (2, 4)), ffn_ranges=((0, 64), (64, 96)))
    w = wl.layer_weights(0)
    x = wl.hidden(2, stream=4)
    kc1, vc1 = oracle.new_cache(wl, 16)
    kc2, vc2 = oracle.new_cache(wl, 16)
    _, _, ap, fp = oracle.tp_layer(wl, w, x, 0, kc1, vc1)
    _, _, aq, fq = oracle.tp_layer_mixed(wl, w, x, 0, kc2, vc2, [bits, bits], [bits, bits])
    for a, b in list(zip(ap, aq)) + list(zip(fp, fq)):
        rel = np.linalg.norm(a - b) / np.linalg.norm(a)
        assert 0 < rel < bound
