"""Python access to the CPU oracle (liboracle.so).

TEST INFRASTRUCTURE: imported only by tests/, __graft_entry__.smoke() and bench.py's CPU-baseline
leg.  The GPU library never imports or calls it.

The functions below marshal numpy arrays into the C oracle; the compositions at the bottom
(`tp_attention`, `tp_ffn`, `tp_layer`) wire the blocks together the way tensor parallelism does
in Voltron Section 3.2.1: every device gets the same layer input, computes its shard, and the
shard outputs are summed (with the residual) on the main device.
"""
from __future__ import annotations

import ctypes
from typing import Dict, List, Optional, Sequence, Tuple

import numpy as np

from . import build as _build

_lib = None
_P = ctypes.c_void_p
_I32 = ctypes.c_int32
_I64 = ctypes.c_int64
_F64 = ctypes.c_double


class OrShapes(ctypes.Structure):
    _fields_ = [("d_model", _I32), ("n_heads", _I32), ("n_kv_heads", _I32), ("d_head", _I32),
                ("d_ffn", _I32), ("rms_eps", _F64), ("rope_theta", _F64)]


class OrQMat(ctypes.Structure):
    _fields_ = [("q", _P), ("scales", _P), ("rows", _I64), ("k", _I64), ("block", _I32)]


class OrLayer(ctypes.Structure):
    _fields_ = [(n, _P) for n in ("attn_norm", "wq", "wk", "wv", "wo", "ffn_norm", "w_gate",
                                  "w_up", "w_down")]


def lib():
    global _lib
    if _lib is None:
        L = ctypes.CDLL(str(_build.build()))
        L.or_num_threads.restype = _I32
        L.or_set_threads.argtypes = [_I32]
        L.or_f16_to_f64.argtypes = [ctypes.c_uint16]
        L.or_f16_to_f64.restype = _F64
        L.or_f64_to_f16.argtypes = [_F64]
        L.or_f64_to_f16.restype = ctypes.c_uint16
        L.or_rmsnorm.argtypes = [_P, _P, _I32, _F64, _P]
        L.or_rope.argtypes = [_P, _I32, _I64, _F64]
        L.or_silu.argtypes = [_F64]
        L.or_silu.restype = _F64
        L.or_attend.argtypes = [_P, _P, _P, _I64, _I32, _P, _P]
        L.or_kv_append.argtypes = [ctypes.POINTER(OrShapes), ctypes.POINTER(OrLayer), _I32, _I32,
                                   _P, _I32, _I64, _P, _P, _I64]
        L.or_kv_append.restype = _I32
        L.or_attn_partial.argtypes = [ctypes.POINTER(OrShapes), ctypes.POINTER(OrLayer), _I32,
                                      _I32, _P, _I32, _P, _P, _P, _I64, _P]
        L.or_attn_partial.restype = _I32
        L.or_attn_partial_window.argtypes = [ctypes.POINTER(OrShapes), ctypes.POINTER(OrLayer), _I32,
                                             _I32, _P, _I32, _P, _P, _P, _I64, _I64, _P]
        L.or_attn_partial_window.restype = _I32
        L.or_ffn_partial.argtypes = [ctypes.POINTER(OrShapes), ctypes.POINTER(OrLayer), _I32,
                                     _I32, _P, _I32, _P]
        L.or_ffn_partial.restype = _I32
        L.or_combine.argtypes = [ctypes.POINTER(_P), _I32, _I64, _P, _P]
        L.or_quantize_rows.argtypes = [_P, _I64, _I64, _I32, _I32, _P, _P]
        L.or_quantize_rows.restype = _I32
        L.or_gemv_blockq.argtypes = [_P, _P, _I64, _I64, _I32, _P, _P]
        L.or_quantize_vec.argtypes = [_P, _I64, _I32, _I32, _P, _P]
        L.or_quantize_vec.restype = _I32
        L.or_combine_q.argtypes = [ctypes.POINTER(_P), ctypes.POINTER(_P), _I32, _I64, _I32, _P, _P]
        QM = ctypes.POINTER(OrQMat)
        L.or_kv_append_q.argtypes = [ctypes.POINTER(OrShapes), _P, QM, QM, _I32, _I32, _P, _I32, _I64, _P, _P, _I64]
        L.or_kv_append_q.restype = _I32
        L.or_attn_partial_q.argtypes = [ctypes.POINTER(OrShapes), _P, QM, QM, _I32, _I32, _P, _I32, _P, _P, _P,
                                         _I64, _I64, _P]
        L.or_attn_partial_q.restype = _I32
        L.or_ffn_partial_q.argtypes = [ctypes.POINTER(OrShapes), _P, QM, QM, QM, _I32, _P, _I32, _P]
        L.or_ffn_partial_q.restype = _I32
        _lib = L
    return _lib


def num_threads() -> int:
    return int(lib().or_num_threads())


def set_threads(n: int) -> None:
    lib().or_set_threads(int(n))


def _f16(a: np.ndarray) -> np.ndarray:
    a = np.ascontiguousarray(a)
    if a.dtype != np.float16:
        raise TypeError(f"expected float16, got {a.dtype}")
    return a


def _f64(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.float64)


def shapes_of(wl) -> OrShapes:
    return OrShapes(wl.d_model, wl.n_heads, wl.n_kv_heads, wl.d_head, wl.d_ffn, wl.rms_eps,
                    wl.rope_theta)


def layer_of(weights: Dict[str, np.ndarray]) -> Tuple[OrLayer, list]:
    keep = [_f16(weights[n]) for n, _ in OrLayer._fields_]
    return OrLayer(*[k.ctypes.data for k in keep]), keep


# ------------------------------------------------------------------ building blocks ---------

def f16_to_f64(bits: int) -> float:
    return float(lib().or_f16_to_f64(int(bits)))


def f64_to_f16(x: float) -> int:
    return int(lib().or_f64_to_f16(float(x)))


def rmsnorm(x, gain: np.ndarray, eps: float) -> np.ndarray:
    x = _f64(x)
    g = _f16(gain)
    y = np.empty_like(x)
    lib().or_rmsnorm(x.ctypes.data, g.ctypes.data, x.size, eps, y.ctypes.data)
    return y


def rope(v, pos: int, theta: float) -> np.ndarray:
    v = _f64(v).copy()
    lib().or_rope(v.ctypes.data, v.size, int(pos), float(theta))
    return v


def silu(z: float) -> float:
    return float(lib().or_silu(float(z)))


def attend(q, k: np.ndarray, v: np.ndarray) -> Tuple[np.ndarray, np.ndarray]:
    """q [dh] (fp64), k/v [n_pos, dh] binary16 -> (weights [n_pos], output [dh])."""
    q = _f64(q)
    k, v = _f16(k), _f16(v)
    n_pos, dh = k.shape
    w = np.empty(n_pos, np.float64)
    o = np.empty(dh, np.float64)
    lib().or_attend(q.ctypes.data, k.ctypes.data, v.ctypes.data, n_pos, dh, w.ctypes.data,
                    o.ctypes.data)
    return w, o


def kv_append(wl, weights, kv_heads: Tuple[int, int], x: np.ndarray, pos0: int,
              kcache: np.ndarray, vcache: np.ndarray) -> None:
    """In-place append into the full-layer caches [Hk, cap, dh] (binary16)."""
    x = _f16(x).reshape(-1, wl.d_model)
    assert kcache.flags.c_contiguous and vcache.flags.c_contiguous
    s = shapes_of(wl)
    L, keep = layer_of(weights)
    rc = lib().or_kv_append(ctypes.byref(s), ctypes.byref(L), kv_heads[0], kv_heads[1],
                            x.ctypes.data, x.shape[0], int(pos0), kcache.ctypes.data,
                            vcache.ctypes.data, kcache.shape[1])
    if rc != 0:
        raise ValueError("or_kv_append rejected its arguments")


def attn_partial(wl, weights, heads: Tuple[int, int], x: np.ndarray, pos: Sequence[int],
                 kcache: np.ndarray, vcache: np.ndarray, window: int = 0) -> np.ndarray:
    """ATTN partial of query heads `heads`; window > 0: sliding-window attention over the last
    `window` positions (up to and including the row's own)."""
    x = _f16(x).reshape(-1, wl.d_model)
    p = np.ascontiguousarray(pos, dtype=np.int64)
    assert p.size == x.shape[0]
    out = np.empty((x.shape[0], wl.d_model), np.float64)
    s = shapes_of(wl)
    L, keep = layer_of(weights)
    rc = lib().or_attn_partial_window(ctypes.byref(s), ctypes.byref(L), heads[0], heads[1],
                                      x.ctypes.data, x.shape[0], p.ctypes.data, _f16(kcache).ctypes.data,
                                      _f16(vcache).ctypes.data, kcache.shape[1], int(window), out.ctypes.data)
    if rc != 0:
        raise ValueError("or_attn_partial rejected its arguments")
    return out


def ffn_partial(wl, weights, cols: Tuple[int, int], h: np.ndarray) -> np.ndarray:
    h = _f16(h).reshape(-1, wl.d_model)
    out = np.empty((h.shape[0], wl.d_model), np.float64)
    s = shapes_of(wl)
    L, keep = layer_of(weights)
    rc = lib().or_ffn_partial(ctypes.byref(s), ctypes.byref(L), cols[0], cols[1], h.ctypes.data,
                              h.shape[0], out.ctypes.data)
    if rc != 0:
        raise ValueError("or_ffn_partial rejected its arguments")
    return out


def combine(partials: Sequence[np.ndarray], residual: Optional[np.ndarray]) -> np.ndarray:
    parts = [_f64(p) for p in partials]
    count = parts[0].size if parts else (residual.size if residual is not None else 0)
    arr = (_P * max(1, len(parts)))(*[p.ctypes.data for p in parts])
    out = np.empty(count, np.float16)
    res = _f16(residual).reshape(-1) if residual is not None else None
    lib().or_combine(arr, len(parts), count, res.ctypes.data if res is not None else None,
                     out.ctypes.data)
    shape = parts[0].shape if parts else residual.shape
    return out.reshape(shape)


# ------------------------------------------------------------------ compositions ------------

def kv_heads_of(wl, heads: Tuple[int, int]) -> Tuple[int, int]:
    g = wl.n_heads // wl.n_kv_heads
    return heads[0] // g, (heads[1] + g - 1) // g


def new_cache(wl, cap: int) -> Tuple[np.ndarray, np.ndarray]:
    shape = (wl.n_kv_heads, cap, wl.d_head)
    return np.zeros(shape, np.float16), np.zeros(shape, np.float16)


def tp_attention(wl, weights, x: np.ndarray, pos0: int, kcache, vcache,
                 head_ranges=None, window: int = 0) -> Tuple[np.ndarray, List[np.ndarray]]:
    """One ATTN block under tensor parallelism: every shard appends its KV heads for all rows,
    then computes its partial; returns (h = binary16(x + sum partials), partials).  window > 0:
    sliding-window attention (see attn_partial)."""
    head_ranges = wl.head_ranges if head_ranges is None else head_ranges
    x = _f16(x).reshape(-1, wl.d_model)
    rows = x.shape[0]
    for hr in head_ranges:
        kv_append(wl, weights, kv_heads_of(wl, hr), x, pos0, kcache, vcache)
    pos = np.arange(pos0, pos0 + rows)
    parts = [attn_partial(wl, weights, hr, x, pos, kcache, vcache, window) for hr in head_ranges]
    return combine(parts, x), parts


def tp_ffn(wl, weights, h: np.ndarray, ffn_ranges=None) -> Tuple[np.ndarray, List[np.ndarray]]:
    ffn_ranges = wl.ffn_ranges if ffn_ranges is None else ffn_ranges
    h = _f16(h).reshape(-1, wl.d_model)
    parts = [ffn_partial(wl, weights, cr, h) for cr in ffn_ranges]
    return combine(parts, h), parts


def tp_layer(wl, weights, x: np.ndarray, pos0: int, kcache, vcache, head_ranges=None,
             ffn_ranges=None, window: int = 0):
    """Whole decoder layer: returns (h, x_next, attn_partials, ffn_partials)."""
    h, ap = tp_attention(wl, weights, x, pos0, kcache, vcache, head_ranges, window)
    xn, fp = tp_ffn(wl, weights, h, ffn_ranges)
    return h, xn, ap, fp


def quantize_rows(w: np.ndarray, bits: int, block: int = 32) -> Tuple[np.ndarray, np.ndarray]:
    """Block quantization of binary16 weight rows [rows, k] (format in oracle.c): int8 codes
    [rows, k] and binary16 scales [rows, ceil(k / block)]."""
    w = _f16(w)
    if w.ndim != 2:
        raise ValueError("expected [rows, k]")
    rows, k = w.shape
    q = np.zeros((rows, k), np.int8)
    sc = np.zeros((rows, (k + block - 1) // block), np.float16)
    st = lib().or_quantize_rows(w.ctypes.data, rows, k, bits, block, q.ctypes.data, sc.ctypes.data)
    if st != 0:
        raise ValueError(f"or_quantize_rows failed ({st})")
    return q, sc


def gemv_blockq(q: np.ndarray, scales: np.ndarray, x, block: int = 32) -> np.ndarray:
    """Dequantized W . x in binary64."""
    q = np.ascontiguousarray(q, np.int8)
    sc = _f16(scales)
    xx = _f64(x).reshape(-1)
    rows, k = q.shape
    if xx.size != k or sc.shape != (rows, (k + block - 1) // block):
        raise ValueError("shape mismatch")
    y = np.zeros(rows, np.float64)
    lib().or_gemv_blockq(q.ctypes.data, sc.ctypes.data, rows, k, block, xx.ctypes.data, y.ctypes.data)
    return y


def quantize_vec(x, bits: int, block: int = 32) -> Tuple[np.ndarray, np.ndarray]:
    """Block quantization of a binary32 vector (a shard partial): int8 codes, binary16 scales."""
    xx = np.ascontiguousarray(x, np.float32).reshape(-1)
    q = np.zeros(xx.size, np.int8)
    sc = np.zeros((xx.size + block - 1) // block, np.float16)
    st = lib().or_quantize_vec(xx.ctypes.data, xx.size, bits, block, q.ctypes.data, sc.ctypes.data)
    if st != 0:
        raise ValueError(f"or_quantize_vec failed ({st})")
    return q, sc


def combine_q(parts: Sequence[Tuple[np.ndarray, np.ndarray]], residual: Optional[np.ndarray], block: int = 32) -> np.ndarray:
    """binary16(residual + sum of the dequantized partials), shards in order."""
    qs = [np.ascontiguousarray(q, np.int8) for q, _ in parts]
    ss = [_f16(s) for _, s in parts]
    count = qs[0].size
    qp = (_P * len(qs))(*[q.ctypes.data for q in qs])
    sp = (_P * len(ss))(*[s.ctypes.data for s in ss])
    out = np.zeros(count, np.float16)
    res = _f16(residual).reshape(-1) if residual is not None else None
    lib().or_combine_q(qp, sp, len(qs), count, block, res.ctypes.data if res is not None else None, out.ctypes.data)
    return out


# ------------------------------------------------------------------ quantized shards ---------

def _qm(m):
    """(codes int8 [rows, k], scales binary16 [rows, nb], block) -> OrQMat (arrays kept alive by the caller)."""
    q, sc, block = m
    q = np.ascontiguousarray(q, np.int8)
    sc = _f16(sc)
    return OrQMat(q.ctypes.data, sc.ctypes.data, q.shape[0], q.shape[1], int(block)), (q, sc)


def shard_qweights(wl, weights, heads: Tuple[int, int], cols: Tuple[int, int], attn_bits: int, ffn_bits: int,
                   block: int = 32) -> Dict[str, tuple]:
    """The shard's projections quantized with quantize_rows (bits 16: left out): query rows of heads,
    K / V rows of their KV heads, the heads' columns of Wo, gate / up rows of the columns and the
    columns of W_down, each as (codes, scales, block) with blocks along its contraction axis."""
    dh = wl.d_head
    (h0, h1), (c0, c1) = heads, cols
    k0, k1 = kv_heads_of(wl, heads)
    out = {}
    if attn_bits in (8, 4) and h1 > h0:
        for name, m in (("wq", weights["wq"][h0 * dh:h1 * dh]), ("wk", weights["wk"][k0 * dh:k1 * dh]),
                        ("wv", weights["wv"][k0 * dh:k1 * dh]), ("wo", weights["wo"][:, h0 * dh:h1 * dh])):
            out[name] = quantize_rows(np.ascontiguousarray(m), attn_bits, block) + (block,)
    if ffn_bits in (8, 4) and c1 > c0:
        for name, m in (("w_gate", weights["w_gate"][c0:c1]), ("w_up", weights["w_up"][c0:c1]),
                        ("w_down", weights["w_down"][:, c0:c1])):
            out[name] = quantize_rows(np.ascontiguousarray(m), ffn_bits, block) + (block,)
    return out


def kv_append_q(wl, weights, kv_heads: Tuple[int, int], x, pos0: int, kcache, vcache, qw) -> None:
    x = _f16(x).reshape(-1, wl.d_model)
    s = shapes_of(wl)
    mk, kk = _qm(qw["wk"])
    mv, kv = _qm(qw["wv"])
    g = _f16(weights["attn_norm"])
    rc = lib().or_kv_append_q(ctypes.byref(s), g.ctypes.data, ctypes.byref(mk), ctypes.byref(mv), kv_heads[0],
                              kv_heads[1], x.ctypes.data, x.shape[0], int(pos0), kcache.ctypes.data,
                              vcache.ctypes.data, kcache.shape[1])
    if rc != 0:
        raise ValueError("or_kv_append_q rejected its arguments")


def attn_partial_q(wl, weights, heads: Tuple[int, int], x, pos, kcache, vcache, qw, window: int = 0):
    x = _f16(x).reshape(-1, wl.d_model)
    p = np.ascontiguousarray(pos, dtype=np.int64)
    out = np.empty((x.shape[0], wl.d_model), np.float64)
    s = shapes_of(wl)
    empty = (np.zeros((0, 0), np.int8), np.zeros((0, 0), np.float16), 32)
    mq, k1 = _qm(qw.get("wq", empty))
    mo, k2 = _qm(qw.get("wo", empty))
    g = _f16(weights["attn_norm"])
    rc = lib().or_attn_partial_q(ctypes.byref(s), g.ctypes.data, ctypes.byref(mq), ctypes.byref(mo), heads[0],
                                 heads[1], x.ctypes.data, x.shape[0], p.ctypes.data, _f16(kcache).ctypes.data,
                                 _f16(vcache).ctypes.data, kcache.shape[1], int(window), out.ctypes.data)
    if rc != 0:
        raise ValueError("or_attn_partial_q rejected its arguments")
    return out


def ffn_partial_q(wl, weights, cols: Tuple[int, int], h, qw):
    h = _f16(h).reshape(-1, wl.d_model)
    out = np.empty((h.shape[0], wl.d_model), np.float64)
    s = shapes_of(wl)
    empty = (np.zeros((0, 0), np.int8), np.zeros((0, 0), np.float16), 32)
    mg, k1 = _qm(qw.get("w_gate", empty))
    mu, k2 = _qm(qw.get("w_up", empty))
    md, k3 = _qm(qw.get("w_down", empty))
    g = _f16(weights["ffn_norm"])
    rc = lib().or_ffn_partial_q(ctypes.byref(s), g.ctypes.data, ctypes.byref(mg), ctypes.byref(mu), ctypes.byref(md),
                                cols[1] - cols[0], h.ctypes.data, h.shape[0], out.ctypes.data)
    if rc != 0:
        raise ValueError("or_ffn_partial_q rejected its arguments")
    return out


def tp_layer_mixed(wl, weights, x, pos0: int, kcache, vcache, attn_bits, ffn_bits, window: int = 0,
                   head_ranges=None, ffn_ranges=None):
    """A decoder layer whose shards each run at their own precision (16: binary16 weights; 8 / 4:
    block-quantized by quantize_rows): returns (h, x_next, attn_partials, ffn_partials)."""
    head_ranges = wl.head_ranges if head_ranges is None else head_ranges
    ffn_ranges = wl.ffn_ranges if ffn_ranges is None else ffn_ranges
    x = _f16(x).reshape(-1, wl.d_model)
    rows = x.shape[0]
    qws = [shard_qweights(wl, weights, hr, cr, ab, fb)
           for hr, cr, ab, fb in zip(head_ranges, ffn_ranges, attn_bits, ffn_bits)]
    for hr, ab, qw in zip(head_ranges, attn_bits, qws):
        kvh = kv_heads_of(wl, hr)
        if kvh[1] > kvh[0]:
            if ab == 16:
                kv_append(wl, weights, kvh, x, pos0, kcache, vcache)
            else:
                kv_append_q(wl, weights, kvh, x, pos0, kcache, vcache, qw)
    pos = np.arange(pos0, pos0 + rows)
    ap = [attn_partial(wl, weights, hr, x, pos, kcache, vcache, window) if ab == 16 or hr[1] == hr[0]
          else attn_partial_q(wl, weights, hr, x, pos, kcache, vcache, qw, window)
          for hr, ab, qw in zip(head_ranges, attn_bits, qws)]
    h = combine(ap, x)
    fp = [ffn_partial(wl, weights, cr, h) if fb == 16 or cr[1] == cr[0] else ffn_partial_q(wl, weights, cr, h, qw)
          for cr, fb, qw in zip(ffn_ranges, ffn_bits, qws)]
    return h, combine(fp, h), ap, fp
