"""ctypes binding of libvoltron.so, with the C ABI's names (include/voltron.h).

Argument marshalling only: every step of the path runs in the library's CUDA kernels.  Device
buffers are torch CUDA tensors (their data_ptr() is passed through); the library allocates its own
buffers through torch's caching allocator, so PyTorch owns device memory.  Streams default to
torch's current stream.  There is no fallback: without the built library every call raises.
"""
from __future__ import annotations

import ctypes
from pathlib import Path
from typing import Iterable, List, Optional, Sequence, Tuple

import numpy as np

_HERE = Path(__file__).resolve().parent
LIB_PATH = _HERE / "libvoltron.so"

VT_OK = 0
VT_ERR_INVALID_ARG = 1
VT_ERR_SHAPE = 2
VT_ERR_PARTITION_OVERLAP = 3
VT_ERR_PARTITION_GAP = 4
VT_ERR_PARTITION_GQA = 5
VT_ERR_PARTITION_RANGE = 6
VT_ERR_KV_CAPACITY = 7
VT_ERR_CUDA = 8
VT_ERR_ALLOC = 9
VT_ERR_STATE = 10
VT_ERR_PLAN_MEMORY = 11
VT_ERR_PLAN_QOS = 12
VT_MAX_DEVICES = 16
VT_DEV_KV_OVERFLOW = 1
VT_DEV_WAIT_TIMEOUT = 2
VT_DEV_BAD_TOKEN = 4
VT_BLOCK_ATTN = 0
VT_BLOCK_FFN = 1
VT_PARTITION_PRUNE = 1

_P = ctypes.c_void_p
_I32 = ctypes.c_int32
_U32 = ctypes.c_uint32


class VtError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"vt status {status}: {message}")
        self.status = status


class vt_shapes(ctypes.Structure):
    _fields_ = [("n_layers", _I32), ("d_model", _I32), ("n_heads", _I32), ("n_kv_heads", _I32),
                ("d_head", _I32), ("d_ffn", _I32), ("vocab", _I32), ("max_seq", _I32),
                ("rms_eps", ctypes.c_float), ("rope_theta", ctypes.c_float)]


class vt_range(ctypes.Structure):
    _fields_ = [("begin", _I32), ("end", _I32)]


class vt_block_plan(ctypes.Structure):
    _fields_ = [("tp", _I32), ("device", _I32), ("ranges", vt_range * VT_MAX_DEVICES),
                ("compute_s", ctypes.c_double), ("comm_s", ctypes.c_double)]


ALLOC_FN = ctypes.CFUNCTYPE(_P, ctypes.c_size_t, _P)
FREE_FN = ctypes.CFUNCTYPE(None, _P, _P)


class vt_allocator(ctypes.Structure):
    _fields_ = [("alloc", ALLOC_FN), ("free", FREE_FN), ("ctx", _P)]


class vt_layer_weights(ctypes.Structure):
    _fields_ = [(n, _P) for n in ("attn_norm", "wq", "wk", "wv", "wo", "ffn_norm", "w_gate",
                                  "w_up", "w_down")]


class vt_shard(ctypes.Structure):
    _fields_ = [("layer", _I32), ("device", _I32), ("block", _I32)]


_lib = None


def lib() -> ctypes.CDLL:
    """The loaded library; raises if it has not been built (no CPU fallback exists)."""
    global _lib
    if _lib is None:
        if not LIB_PATH.exists():
            raise RuntimeError(f"{LIB_PATH} is missing: build it with "
                               "paper_2607_07046_gb300.build.build()")
        L = ctypes.CDLL(str(LIB_PATH))
        S = vt_status_t = _I32
        sig = {
            "vt_last_error": (ctypes.c_char_p, []),
            "vt_version": (ctypes.c_char_p, []),
            "vt_shapes_validate": (S, [ctypes.POINTER(vt_shapes)]),
            "vt_partition_validate": (S, [ctypes.POINTER(vt_shapes), _I32, ctypes.POINTER(vt_range),
                                          ctypes.POINTER(vt_range)]),
            "vt_plan_tp_shares": (S, [ctypes.POINTER(vt_shapes), _I32, _I32, ctypes.POINTER(ctypes.c_double),
                                      ctypes.POINTER(ctypes.c_double), _I32, ctypes.POINTER(vt_range),
                                      ctypes.POINTER(ctypes.c_double)]),
            "vt_quantize_rows": (S, [_P, ctypes.c_int64, ctypes.c_int64, _I32, _I32, _P, _P]),
            "vt_plan_precision": (S, [ctypes.POINTER(vt_shapes), _I32, ctypes.POINTER(vt_block_plan),
                                      ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_double),
                                      ctypes.POINTER(ctypes.c_double), ctypes.c_double, _I32,
                                      ctypes.POINTER(_I32), ctypes.POINTER(_I32), ctypes.POINTER(ctypes.c_double)]),
            "vt_plan_layers": (S, [ctypes.POINTER(vt_shapes), _I32, ctypes.POINTER(ctypes.c_double),
                                   ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_double),
                                   ctypes.c_double, ctypes.c_double, _I32, _I32,
                                   ctypes.POINTER(vt_block_plan), ctypes.POINTER(ctypes.c_double)]),
            "vt_model_create": (S, [ctypes.POINTER(vt_shapes), ctypes.POINTER(vt_layer_weights), _P,
                                    ctypes.POINTER(vt_allocator), _P, ctypes.POINTER(_P)]),
            "vt_model_load_layer": (S, [_P, _I32, ctypes.POINTER(vt_layer_weights), _P]),
            "vt_model_load_embedding": (S, [_P, _P, _P]),
            "vt_model_shapes": (S, [_P, ctypes.POINTER(vt_shapes)]),
            "vt_model_destroy": (None, [_P]),
            "vt_model_status": (S, [_P, ctypes.POINTER(ctypes.c_uint32), _I32]),
            "vt_model_set_window": (S, [_P, _I32, _I32]),
            "vt_model_window": (S, [_P, _I32, ctypes.POINTER(_I32)]),
            "vt_embed": (S, [_P, _P, _I32, _P, _P]),
            "vt_partition_create": (S, [_P, _I32, ctypes.POINTER(vt_range), ctypes.POINTER(vt_range),
                                        _P, ctypes.POINTER(_P)]),
            "vt_partition_devices": (_I32, [_P]),
            "vt_partition_create_layers": (S, [_P, _I32, ctypes.POINTER(vt_range), ctypes.POINTER(vt_range),
                                               ctypes.c_uint32, _P, ctypes.POINTER(_P)]),
            "vt_partition_validate_layers": (S, [ctypes.POINTER(vt_shapes), _I32, ctypes.POINTER(vt_range),
                                                 ctypes.POINTER(vt_range), ctypes.c_uint32]),
            "vt_partition_status": (S, [_P, ctypes.POINTER(ctypes.c_uint32), _I32]),
            "vt_partition_destroy": (None, [_P]),
            "vt_shard_weights_read": (S, [_P, vt_shard, _I32, _P, ctypes.c_size_t,
                                          ctypes.POINTER(ctypes.c_size_t)]),
            "vt_shard_weight_layout": (S, [_P, vt_shard, _I32, ctypes.POINTER(ctypes.c_int64),
                                           ctypes.POINTER(ctypes.c_int64)]),
            "vt_kv_create": (S, [_P, _I32, _P, ctypes.POINTER(_P)]),
            "vt_kv_destroy": (None, [_P]),
            "vt_kv_capacity": (_I32, [_P]),
            "vt_kv_advance": (S, [_P, _I32, _I32, _P]),
            "vt_kv_set_length": (S, [_P, _I32, _I32, _P]),
            "vt_kv_length": (S, [_P, _I32, _P, ctypes.POINTER(_I32)]),
            "vt_kv_status": (S, [_P, ctypes.POINTER(ctypes.c_uint32), _I32]),
            "vt_kv_read": (S, [_P, _I32, _I32, _I32, _P, _P]),
            "vt_kv_write_raw": (S, [_P, _I32, _I32, _I32, _P, _P]),
            "vt_decode_step": (S, [_P, vt_shard, _P, _P, _P, _P]),
            "vt_decode_step_static": (S, [_P, vt_shard, _P, _P, _P, _P]),
            "vt_prefill": (S, [_P, vt_shard, _P, _I32, _P, _P, _P]),
            "vt_combine": (S, [ctypes.POINTER(_P), _I32, _I32, _I32, _P, _P, _P]),
            "vt_decode_token": (S, [_P, _P, _P, _P, _P]),
            "vt_decode_token_sharded": (S, [_P, _P, _P, _P, _P]),
            "vt_decode_token_fused_available": (_I32, [_P, ctypes.POINTER(ctypes.c_char_p)]),
            "vt_prefill_tokens": (S, [_P, _P, _P, _I32, _P, _P]),
            "vt_partition_set_precision": (S, [_P, vt_shard, _I32, _P]),
            "vt_shard_precision": (_I32, [_P, vt_shard]),
            "vt_shard_qweights_read": (S, [_P, vt_shard, _I32, _P, _P]),
            "vt_partial_code_bytes": (ctypes.c_size_t, [ctypes.c_int64, _I32]),
            "vt_quantize_partial": (S, [_P, ctypes.c_int64, _I32, _P, _P, _P]),
            "vt_combine_q": (S, [ctypes.POINTER(_P), ctypes.POINTER(_P), _I32, ctypes.c_int64, _I32, _P, _P, _P]),
            "vt_partition_set_comm_bits": (S, [_P, _I32, _I32]),
            "vt_token_partials_read": (S, [_P, _I32, _P]),
            "vt_token_test_barrier": (S, [_P, _I32, _U32, _P]),
        }
        for name, (res, args) in sig.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


def vt_last_error() -> str:
    return lib().vt_last_error().decode()


def vt_version() -> str:
    return lib().vt_version().decode()


def _check(status: int) -> None:
    if status != VT_OK:
        raise VtError(status, vt_last_error())


def _stream(stream) -> int:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if hasattr(stream, "cuda_stream"):
        return stream.cuda_stream
    return int(stream)


def _ptr(t, dtype=None) -> int:
    """data_ptr of a contiguous CUDA tensor (checked), or 0 for None."""
    if t is None:
        return 0
    import torch
    if not isinstance(t, torch.Tensor):
        raise TypeError("expected a torch tensor")
    if not t.is_cuda or not t.is_contiguous():
        raise ValueError("expected a contiguous CUDA tensor")
    if dtype is not None and t.dtype != dtype:
        raise TypeError(f"expected {dtype}, got {t.dtype}")
    return t.data_ptr()


def make_shapes(n_layers, d_model, n_heads, n_kv_heads, d_head, d_ffn, vocab, max_seq,
                rms_eps=1e-5, rope_theta=1e4) -> vt_shapes:
    return vt_shapes(n_layers, d_model, n_heads, n_kv_heads, d_head, d_ffn, vocab, max_seq,
                     rms_eps, rope_theta)


def _ranges(rs: Sequence[Tuple[int, int]]):
    arr = (vt_range * max(1, len(rs)))(*[vt_range(a, b) for a, b in rs])
    return arr


# ------------------------------------------------------------------ allocator (torch-backed)

def _torch_alloc(nbytes, ctx):
    import torch
    try:
        return torch.cuda.caching_allocator_alloc(int(nbytes), torch.cuda.current_device())
    except Exception:  # out of memory: the library reports VT_ERR_ALLOC
        return None


def _torch_free(ptr, ctx):
    import torch
    torch.cuda.caching_allocator_delete(ptr)


_TORCH_ALLOCATOR = vt_allocator(ALLOC_FN(_torch_alloc), FREE_FN(_torch_free), None)


# ------------------------------------------------------------------ validation (host only)

def vt_shapes_validate(shapes: vt_shapes) -> int:
    return int(lib().vt_shapes_validate(ctypes.byref(shapes)))


def vt_partition_validate(shapes: vt_shapes, head_ranges, ffn_col_ranges) -> int:
    n = len(head_ranges)
    if len(ffn_col_ranges) != n:
        raise ValueError("one head range and one FFN range per device")
    return int(lib().vt_partition_validate(ctypes.byref(shapes), n, _ranges(head_ranges),
                                           _ranges(ffn_col_ranges)))


def vt_plan_tp_shares(shapes: vt_shapes, block: int, rate, mem_bytes=None, col_unit: int = 1):
    """Heterogeneity-aware TP shares of one block: (ranges per device, makespan in seconds).
    rate: bytes per second of each device; mem_bytes: per-device budget for the block's shard, or
    None.  Raises VtError on a failed status."""
    n = len(rate)
    r = (ctypes.c_double * max(1, n))(*[float(x) for x in rate])
    m = None
    if mem_bytes is not None:
        if len(mem_bytes) != n:
            raise ValueError("one memory budget per device")
        m = (ctypes.c_double * max(1, n))(*[float(x) for x in mem_bytes])
    out = (vt_range * max(1, n))()
    ms = ctypes.c_double(0.0)
    _check(lib().vt_plan_tp_shares(ctypes.byref(shapes), int(block), n, r, m, int(col_unit), out,
                                   ctypes.byref(ms)))
    return [(out[d].begin, out[d].end) for d in range(n)], ms.value


def vt_quantize_rows(w, bits: int, block: int = 32):
    """Host block quantization of fp16 weight rows [rows, k]: (int8 codes [rows, k], fp16 scales
    [rows, ceil(k / block)]).  Raises VtError on a failed status."""
    import numpy as np
    w = np.ascontiguousarray(w, dtype=np.float16)
    if w.ndim != 2:
        raise ValueError("expected [rows, k]")
    rows, k = w.shape
    q = np.zeros((rows, k), np.int8)
    sc = np.zeros((rows, (k + block - 1) // block if block > 0 else 1), np.float16)  # the library checks block
    _check(lib().vt_quantize_rows(w.ctypes.data, rows, k, int(bits), int(block), q.ctypes.data, sc.ctypes.data))
    return q, sc


def vt_plan_layers(shapes: vt_shapes, rate, flop_rate=None, mem_bytes=None, link_bytes_per_s=1e30,
                   link_latency_s=0.0, tokens: int = 1, kv_len: int = 0):
    """Layer-wise MP/TP plan of the stack: (list of per-block dicts, total seconds).  Blocks are
    ATTN of layer 0, FFN of layer 0, ATTN of layer 1, ...  Raises VtError on a failed status."""
    n = len(rate)

    def arr(v):
        if v is None:
            return None
        if len(v) != n:
            raise ValueError("one value per device")
        return (ctypes.c_double * max(1, n))(*[float(x) for x in v])

    out = (vt_block_plan * (2 * shapes.n_layers))()
    tot = ctypes.c_double(0.0)
    _check(lib().vt_plan_layers(ctypes.byref(shapes), n, arr(rate), arr(flop_rate), arr(mem_bytes),
                                float(link_bytes_per_s), float(link_latency_s), int(tokens), int(kv_len),
                                out, ctypes.byref(tot)))
    plans = [dict(tp=bool(p.tp), device=p.device, ranges=[(p.ranges[d].begin, p.ranges[d].end) for d in range(n)],
                  compute_s=p.compute_s, comm_s=p.comm_s) for p in out]
    return plans, tot.value


def vt_plan_precision(shapes: vt_shapes, plans, importance, rate, mem_bytes=None, qos_s: float = 0.0,
                      kv_len: int = 0):
    """Importance-aware precision of every block for a given plan (list of per-block dicts as
    vt_plan_layers returns them): (bits per block, steps, total seconds).  Raises VtError on a
    failed status (VT_ERR_PLAN_MEMORY / VT_ERR_PLAN_QOS when no configuration fits)."""
    n = len(rate)
    nb = 2 * shapes.n_layers
    if len(plans) != nb or len(importance) != nb:
        raise ValueError("one plan and one importance score per block")
    cp = (vt_block_plan * nb)()
    for i, p in enumerate(plans):
        cp[i].tp = int(p.get("tp", 0))
        cp[i].device = int(p.get("device", 0))
        for d, (a, b) in enumerate(p["ranges"]):
            cp[i].ranges[d].begin, cp[i].ranges[d].end = int(a), int(b)
        cp[i].compute_s = float(p.get("compute_s", 0.0))
        cp[i].comm_s = float(p.get("comm_s", 0.0))

    def arr(v):
        if v is None:
            return None
        if len(v) != n:
            raise ValueError("one value per device")
        return (ctypes.c_double * n)(*[float(x) for x in v])

    imp = (ctypes.c_double * nb)(*[float(x) for x in importance])
    bits = (_I32 * nb)()
    steps = _I32(0)
    tot = ctypes.c_double(0.0)
    _check(lib().vt_plan_precision(ctypes.byref(shapes), n, cp, imp, arr(rate), arr(mem_bytes), float(qos_s),
                                   int(kv_len), bits, ctypes.byref(steps), ctypes.byref(tot)))
    return list(bits), steps.value, tot.value


# ------------------------------------------------------------------ model

_WEIGHT_NAMES = ("attn_norm", "wq", "wk", "wv", "wo", "ffn_norm", "w_gate", "w_up", "w_down")


def _layer_struct(w) -> Tuple[vt_layer_weights, list]:
    keep = [np.ascontiguousarray(w[n], dtype=np.float16) for n in _WEIGHT_NAMES]
    return vt_layer_weights(*[k.ctypes.data for k in keep]), keep


def vt_model_create(shapes: vt_shapes, per_layer=None, embed: Optional[np.ndarray] = None,
                    stream=None, allocator: str = "torch") -> int:
    """per_layer: list of dicts of host fp16 arrays (nn.Linear layout), or None."""
    keep = []
    arr = None
    if per_layer is not None:
        structs = []
        for w in per_layer:
            s, k = _layer_struct(w)
            structs.append(s)
            keep.append(k)
        arr = (vt_layer_weights * len(structs))(*structs)
    emb = None if embed is None else np.ascontiguousarray(embed, dtype=np.float16)
    out = _P()
    alloc = ctypes.byref(_TORCH_ALLOCATOR) if allocator == "torch" else None
    _check(lib().vt_model_create(ctypes.byref(shapes), arr, emb.ctypes.data if emb is not None else None,
                                 alloc, _stream(stream), ctypes.byref(out)))
    return out.value


def vt_model_load_layer(model: int, layer: int, weights, stream=None) -> None:
    s, keep = _layer_struct(weights)
    _check(lib().vt_model_load_layer(model, layer, ctypes.byref(s), _stream(stream)))


def vt_model_load_embedding(model: int, embed: np.ndarray, stream=None) -> None:
    e = np.ascontiguousarray(embed, dtype=np.float16)
    _check(lib().vt_model_load_embedding(model, e.ctypes.data, _stream(stream)))


def vt_model_destroy(model: int) -> None:
    if model:
        lib().vt_model_destroy(model)


def vt_model_set_window(model: int, layer: int, window: int) -> None:
    """Sliding attention window of `layer` (-1: every layer); 0 attends to every position."""
    _check(lib().vt_model_set_window(model, int(layer), int(window)))


def vt_model_window(model: int, layer: int) -> int:
    w = _I32()
    _check(lib().vt_model_window(model, int(layer), ctypes.byref(w)))
    return int(w.value)


def vt_model_status(model: int, clear: bool = False) -> int:
    f = ctypes.c_uint32()
    _check(lib().vt_model_status(model, ctypes.byref(f), int(clear)))
    return int(f.value)


def vt_embed(model: int, ids, out, stream=None) -> None:
    import torch
    _check(lib().vt_embed(model, _ptr(ids, torch.int32), ids.numel(), _ptr(out, torch.float16),
                          _stream(stream)))


# ------------------------------------------------------------------ partition

def vt_partition_create(model: int, head_ranges, ffn_col_ranges, stream=None) -> int:
    n = len(head_ranges)
    out = _P()
    _check(lib().vt_partition_create(model, n, _ranges(head_ranges), _ranges(ffn_col_ranges),
                                     _stream(stream), ctypes.byref(out)))
    return out.value


def _layer_ranges(per_layer):
    n = len(per_layer[0])
    if any(len(r) != n for r in per_layer):
        raise ValueError("every layer needs one range per device")
    return _ranges([r for layer in per_layer for r in layer]), n


def vt_partition_create_layers(model: int, head_ranges, ffn_col_ranges, flags: int = 0, stream=None) -> int:
    """head_ranges, ffn_col_ranges: one list of per-device ranges per layer."""
    h, n = _layer_ranges(head_ranges)
    c, n2 = _layer_ranges(ffn_col_ranges)
    if n != n2:
        raise ValueError("one head range and one FFN range per device")
    out = _P()
    _check(lib().vt_partition_create_layers(model, n, h, c, int(flags), _stream(stream), ctypes.byref(out)))
    return out.value


def vt_partition_validate_layers(shapes: vt_shapes, head_ranges, ffn_col_ranges, flags: int = 0) -> int:
    h, n = _layer_ranges(head_ranges)
    c, _ = _layer_ranges(ffn_col_ranges)
    return int(lib().vt_partition_validate_layers(ctypes.byref(shapes), n, h, c, int(flags)))


def vt_partition_devices(part: int) -> int:
    return int(lib().vt_partition_devices(part))


def vt_partition_status(part: int, clear: bool = False) -> int:
    f = ctypes.c_uint32()
    _check(lib().vt_partition_status(part, ctypes.byref(f), int(clear)))
    return int(f.value)


def vt_partition_destroy(part: int) -> None:
    if part:
        lib().vt_partition_destroy(part)


def vt_shard_weight_layout(part: int, shard: Tuple[int, int, int], which: int) -> Tuple[int, int]:
    rows, stride = ctypes.c_int64(), ctypes.c_int64()
    _check(lib().vt_shard_weight_layout(part, vt_shard(*shard), which, ctypes.byref(rows),
                                        ctypes.byref(stride)))
    return int(rows.value), int(stride.value)


def vt_shard_weights_read(part: int, shard: Tuple[int, int, int], which: int) -> np.ndarray:
    rows, stride = vt_shard_weight_layout(part, shard, which)
    out = np.empty((rows, stride), np.float16)
    size = ctypes.c_size_t()
    _check(lib().vt_shard_weights_read(part, vt_shard(*shard), which, out.ctypes.data, out.nbytes,
                                       ctypes.byref(size)))
    assert size.value == out.nbytes
    return out


def vt_partition_set_precision(part: int, shard: Tuple[int, int, int], bits: int, stream=None) -> None:
    """Store one shard at 16 (fp16), 8 or 4 bits (block-quantized, blocks of 32, fp16 scales)."""
    _check(lib().vt_partition_set_precision(part, vt_shard(*shard), int(bits), _stream(stream)))


def vt_shard_precision(part: int, shard: Tuple[int, int, int]) -> int:
    return int(lib().vt_shard_precision(part, vt_shard(*shard)))


def vt_shard_qweights_read(part: int, shard: Tuple[int, int, int], which: int, rows: int, k: int):
    """Codes int8 [rows, k] and fp16 scales [rows, ceil(k / 32)] of a quantized shard tensor."""
    q = np.empty((rows, k), np.int8)
    sc = np.empty((rows, (k + 31) // 32), np.float16)
    _check(lib().vt_shard_qweights_read(part, vt_shard(*shard), int(which), q.ctypes.data, sc.ctypes.data))
    return q, sc


def vt_partial_code_bytes(count: int, bits: int) -> int:
    return int(lib().vt_partial_code_bytes(int(count), int(bits)))


def vt_quantize_partial(partial, bits: int, codes, scales, stream=None) -> None:
    """Device fp32 partial -> device codes (uint8 tensor of vt_partial_code_bytes) and fp16 scales."""
    import torch
    _check(lib().vt_quantize_partial(_ptr(partial, torch.float32), partial.numel(), int(bits), _ptr(codes, torch.uint8),
                                     _ptr(scales, torch.float16), _stream(stream)))


def vt_combine_q(codes: Sequence, scales: Sequence, bits: int, residual, out, stream=None) -> None:
    import torch
    n = len(codes)
    ca = (_P * n)(*[_ptr(c, torch.uint8) for c in codes])
    sa = (_P * n)(*[_ptr(s_, torch.float16) for s_ in scales])
    _check(lib().vt_combine_q(ca, sa, n, out.numel(), int(bits),
                              _ptr(residual, torch.float16) if residual is not None else None,
                              _ptr(out, torch.float16), _stream(stream)))


def vt_partition_set_comm_bits(part: int, device: int, bits: int) -> None:
    _check(lib().vt_partition_set_comm_bits(part, int(device), int(bits)))


# ------------------------------------------------------------------ KV cache

def vt_kv_create(part: int, capacity: int, stream=None) -> int:
    out = _P()
    _check(lib().vt_kv_create(part, capacity, _stream(stream), ctypes.byref(out)))
    return out.value


def vt_kv_destroy(kv: int) -> None:
    if kv:
        lib().vt_kv_destroy(kv)


def vt_kv_capacity(kv: int) -> int:
    return int(lib().vt_kv_capacity(kv))


def vt_kv_advance(kv: int, layer: int, n: int, stream=None) -> None:
    _check(lib().vt_kv_advance(kv, layer, n, _stream(stream)))


def vt_kv_set_length(kv: int, layer: int, length: int, stream=None) -> None:
    _check(lib().vt_kv_set_length(kv, layer, length, _stream(stream)))


def vt_kv_length(kv: int, layer: int, stream=None) -> int:
    v = _I32()
    _check(lib().vt_kv_length(kv, layer, _stream(stream), ctypes.byref(v)))
    return int(v.value)


def vt_kv_status(kv: int, clear: bool = False) -> int:
    f = ctypes.c_uint32()
    _check(lib().vt_kv_status(kv, ctypes.byref(f), int(clear)))
    return int(f.value)


def vt_kv_read(kv: int, layer: int, device: int, n_pos: int, hk: int, d_head: int):
    k = np.empty((hk, n_pos, d_head), np.float16)
    v = np.empty_like(k)
    _check(lib().vt_kv_read(kv, layer, device, n_pos, k.ctypes.data, v.ctypes.data))
    return k, v


def vt_kv_write_raw(kv: int, layer: int, device: int, k: np.ndarray, v: np.ndarray) -> None:
    k = np.ascontiguousarray(k, dtype=np.float16)
    v = np.ascontiguousarray(v, dtype=np.float16)
    assert k.shape == v.shape and k.ndim == 3
    _check(lib().vt_kv_write_raw(kv, layer, device, k.shape[1], k.ctypes.data, v.ctypes.data))


# ------------------------------------------------------------------ shard compute

def vt_decode_step(part: int, shard: Tuple[int, int, int], x, kv: Optional[int], out_partial,
                   stream=None) -> None:
    import torch
    _check(lib().vt_decode_step(part, vt_shard(*shard), _ptr(x, torch.float16), kv or None,
                                _ptr(out_partial, torch.float32), _stream(stream)))


def vt_decode_step_static(part: int, shard: Tuple[int, int, int], x, kv: Optional[int], out_partial,
                          stream=None) -> None:
    """ATTN-shard decode step that allocates nothing: every intermediate is in the library's
    fixed 1 MiB device array (for callers that cannot allocate device memory while decoding).
    Calls in flight at once race on that array; the first call on a device looks its address up
    and should come before any stream capture."""
    import torch
    _check(lib().vt_decode_step_static(part, vt_shard(*shard), _ptr(x, torch.float16), kv or None,
                                       _ptr(out_partial, torch.float32), _stream(stream)))


def vt_prefill(part: int, shard: Tuple[int, int, int], x, n: int, kv: Optional[int], out_partial,
               stream=None) -> None:
    import torch
    _check(lib().vt_prefill(part, vt_shard(*shard), _ptr(x, torch.float16), n, kv or None,
                            _ptr(out_partial, torch.float32), _stream(stream)))


def vt_combine(partials: Sequence, residual, out, rows: int, d: int, stream=None) -> None:
    import torch
    arr = (_P * len(partials))(*[_ptr(p, torch.float32) for p in partials])
    _check(lib().vt_combine(arr, len(partials), rows, d,
                            _ptr(residual, torch.float16) if residual is not None else None,
                            _ptr(out, torch.float16), _stream(stream)))


def vt_decode_token(part: int, kv: int, x_in, x_out, stream=None) -> None:
    import torch
    _check(lib().vt_decode_token(part, kv, _ptr(x_in, torch.float16), _ptr(x_out, torch.float16),
                                 _stream(stream)))


def vt_decode_token_sharded(part: int, kv: int, x_in, x_out, stream=None) -> None:
    import torch
    _check(lib().vt_decode_token_sharded(part, kv, _ptr(x_in, torch.float16),
                                         _ptr(x_out, torch.float16), _stream(stream)))


def vt_decode_token_fused_available(part: int):
    """(available, reason): whether vt_decode_token runs as one fused kernel for this partition."""
    why = ctypes.c_char_p()
    ok = lib().vt_decode_token_fused_available(part, ctypes.byref(why))
    return bool(ok), (why.value or b"").decode()


def vt_token_partials_read(part: int, block: int, n_devices: int, d_model: int) -> np.ndarray:
    """The fused decode-token kernel's fp32 shard partials [n_devices, d_model] of the last layer
    (block VT_BLOCK_ATTN or VT_BLOCK_FFN); test hook, synchronous."""
    out = np.empty((n_devices, d_model), np.float32)
    _check(lib().vt_token_partials_read(part, int(block), out.ctypes.data))
    return out


def vt_token_test_barrier(part: int, cta: int, spin_polls: int, stream=None) -> None:
    """Test hook: CTA `cta` of the next fused tokens skips its first grid-barrier arrival and
    grid-barrier waits give up after `spin_polls` polls, until a status clear."""
    _check(lib().vt_token_test_barrier(part, int(cta), int(spin_polls), _stream(stream)))


def vt_prefill_tokens(part: int, kv: int, x_in, n: int, x_out, stream=None) -> None:
    import torch
    _check(lib().vt_prefill_tokens(part, kv, _ptr(x_in, torch.float16), n,
                                   _ptr(x_out, torch.float16), _stream(stream)))
