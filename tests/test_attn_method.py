"""The prefill attention kernel's numerical method, emulated in numpy on CPU, against the oracle's
exact softmax attention (fp64): blocks of 128 keys, a per-row reference maximum that is raised
only when a block's maximum exceeds it by more than 8 (log2 units; O and l are then rescaled),
P = 2^(s log2(e)/sqrt(dh) - m) computed in fp32 and rounded to fp16 for the P.V product, l summed
in fp32 from the unrounded P, O accumulated in fp32, and O / l rounded to fp16.  The cases include
scores built to force a rescale at every block, scores that fall far below the first block's
maximum (P underflows in fp16), and scores just under the rescale threshold (P near 2^8).  The
bar is the parity tolerance the GPU tests apply to the kernel itself."""
from __future__ import annotations

import numpy as np
import pytest

import oracle
from tests.parity import assert_close

BLOCK = 128
THRESHOLD = 8.0


def kernel_method(q16: np.ndarray, k16: np.ndarray, v16: np.ndarray, n_valid: int) -> np.ndarray:
    """Attention of one query over the first n_valid of the keys, the way k_prefill_attn_tc does it."""
    dh = q16.size
    sl2 = np.float32(np.log2(np.e) / np.sqrt(dh))
    s_all = k16.astype(np.float32) @ q16.astype(np.float32)  # fp16 products, fp32 sums (the MMA)
    m_use, l = -np.inf, np.float32(0.0)
    o = np.zeros(dh, np.float32)
    for b0 in range(0, n_valid, BLOCK):
        s = s_all[b0:min(b0 + BLOCK, n_valid)]
        bms = np.float32(s.max() * sl2)
        if bms > m_use + THRESHOLD:
            if np.isfinite(m_use):
                alpha = np.float32(np.exp2(np.float32(m_use - bms)))
                o *= alpha
                l *= alpha
            m_use = bms
        p = np.exp2((s * sl2 - np.float32(m_use)).astype(np.float32)).astype(np.float32)
        l += p.sum(dtype=np.float32)
        o += p.astype(np.float16).astype(np.float32) @ v16[b0:b0 + s.size].astype(np.float32)
    return (o / l).astype(np.float16)


def scores_to_keys(target_log2: np.ndarray, dh: int, rng) -> tuple:
    """A one-hot query and fp16 keys whose scaled scores s log2(e)/sqrt(dh) equal target_log2
    (to fp16 rounding of the keys)."""
    q = np.zeros(dh, np.float16)
    q[0] = 1.0
    k = (rng.standard_normal((target_log2.size, dh)) * 0.01).astype(np.float32)
    k[:, 0] = target_log2 * np.sqrt(dh) / np.log2(np.e)
    return q, k.astype(np.float16)


def exact(q16, k16, v16, n_valid):
    _, o = oracle.attend(q16.astype(np.float64), k16[:n_valid], v16[:n_valid])
    return o


@pytest.mark.parametrize("dh", [64, 128])
def test_random_rows_of_a_long_prompt(dh):
    rng = np.random.default_rng(11 + dh)
    n = 700
    k16 = rng.standard_normal((n, dh)).astype(np.float16)
    v16 = rng.standard_normal((n, dh)).astype(np.float16)
    got, ref = [], []
    for i in range(24):
        q16 = (rng.standard_normal(dh) * 1.5).astype(np.float16)
        n_valid = int(rng.integers(1, n + 1))
        got.append(kernel_method(q16, k16, v16, n_valid))
        ref.append(exact(q16, k16, v16, n_valid))
    assert_close(np.array(got), np.array(ref), f"random rows dh {dh}")


PATTERNS = ["rising", "falling", "under_threshold", "causal_tail"]


@pytest.mark.parametrize("pattern", PATTERNS)
def test_scores_that_stress_the_reference_maximum(pattern):
    dh = 128
    rng = np.random.default_rng(40 + PATTERNS.index(pattern))
    n = 6 * BLOCK
    blk = np.arange(n) // BLOCK
    if pattern == "rising":            # every block's maximum 10 above the last: a rescale each block
        t = 10.0 * blk + rng.standard_normal(n)
    elif pattern == "falling":         # later blocks 30 below the first: P underflows in fp16
        t = -30.0 * blk + rng.standard_normal(n)
    elif pattern == "under_threshold":  # each block 7.5 above the first: no rescale, P up to ~2^7.5
        t = np.where(blk == 0, 0.0, 7.5) + 0.1 * rng.standard_normal(n)
    else:                              # the row sees 3 blocks and 5 keys of the fourth
        t = rng.standard_normal(n) * 3.0
    n_valid = 3 * BLOCK + 5 if pattern == "causal_tail" else n
    q16, k16 = scores_to_keys(t, dh, rng)
    v16 = rng.standard_normal((n, dh)).astype(np.float16)
    got = kernel_method(q16, k16, v16, n_valid)
    ref = exact(q16, k16, v16, n_valid)
    assert np.all(np.isfinite(got))
    assert_close(got.reshape(1, -1), ref.reshape(1, -1), f"{pattern} scores")


def test_the_rescale_is_exact_in_exact_arithmetic():
    """With fp64 throughout (no fp16 rounding of P), the lazily rescaled sum equals the exact
    softmax to rounding: the reference maximum changes nothing but the scale of O and l."""
    rng = np.random.default_rng(5)
    dh, n = 64, 5 * BLOCK
    t = 10.0 * (np.arange(n) // BLOCK) + rng.standard_normal(n)
    q16, k16 = scores_to_keys(t, dh, rng)
    v = rng.standard_normal((n, dh))
    s = k16.astype(np.float64) @ q16.astype(np.float64) * (np.log2(np.e) / np.sqrt(dh))
    m_use, l, o = -np.inf, 0.0, np.zeros(dh)
    for b0 in range(0, n, BLOCK):
        bm = s[b0:b0 + BLOCK].max()
        if bm > m_use + THRESHOLD:
            if np.isfinite(m_use):
                o *= 2.0 ** (m_use - bm)
                l *= 2.0 ** (m_use - bm)
            m_use = bm
        p = 2.0 ** (s[b0:b0 + BLOCK] - m_use)
        l += p.sum()
        o += p @ v[b0:b0 + BLOCK]
    w = np.exp2(s - s.max())
    np.testing.assert_allclose(o / l, (w / w.sum()) @ v, rtol=1e-12, atol=1e-12)
