"""Seeded synthetic workloads: shapes, partitions and input arrays for both sides of every check.

The arrays are drawn by synth.c (SplitMix64 in counter mode + Box-Muller), so any element is a
pure function of its seed and index.  This module holds no decoder-layer arithmetic.

Recipe (one stream per tensor, seed = model_id * 10**6 + layer * 100 + tensor index):
  * projection weights  W ~ N(0, 0.02^2), drawn in fp32 and rounded to fp16 (nn.Linear layout [out][in]);
  * RMSNorm gains       g ~ 1 + N(0, 0.02^2) (not exactly 1, so a dropped gain is visible);
  * embedding table     E ~ N(0, 0.02^2);
  * hidden-state inputs x ~ N(0, 1);
  * token ids           uniform over [0, vocab);
  * synthetic KV-cache  K, V ~ N(0, (0.02 sqrt(D))^2), the spread a projection of a unit-RMS
    input through N(0, 0.02^2) weights has.
"""
from __future__ import annotations

import ctypes
from dataclasses import dataclass, field
from typing import Dict, Tuple

import numpy as np

from . import build as _build

_lib = None


def _synth():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(str(_build.build()))
        i64, u64, f64 = ctypes.c_int64, ctypes.c_uint64, ctypes.c_double
        lib.synth_words.argtypes = [ctypes.c_void_p, i64, u64]
        lib.synth_normal_f16.argtypes = [ctypes.c_void_p, i64, u64, f64, f64]
        lib.synth_normal_f32.argtypes = [ctypes.c_void_p, i64, u64, f64, f64]
        lib.synth_uniform_i32.argtypes = [ctypes.c_void_p, i64, u64, ctypes.c_int32, ctypes.c_int32]
        _lib = lib
    return _lib


def words(n: int, seed: int) -> np.ndarray:
    out = np.empty(n, dtype=np.uint64)
    _synth().synth_words(out.ctypes.data, n, seed)
    return out


def normal_f16(shape, seed: int, mean: float = 0.0, std: float = 1.0) -> np.ndarray:
    out = np.empty(shape, dtype=np.float16)
    _synth().synth_normal_f16(out.ctypes.data, out.size, seed, mean, std)
    return out


def normal_f32(shape, seed: int, mean: float = 0.0, std: float = 1.0) -> np.ndarray:
    out = np.empty(shape, dtype=np.float32)
    _synth().synth_normal_f32(out.ctypes.data, out.size, seed, mean, std)
    return out


def uniform_i32(n: int, seed: int, lo: int, hi: int) -> np.ndarray:
    out = np.empty(n, dtype=np.int32)
    _synth().synth_uniform_i32(out.ctypes.data, n, seed, lo, hi)
    return out


TENSORS = ("attn_norm", "wq", "wk", "wv", "wo", "ffn_norm", "w_gate", "w_up", "w_down")


@dataclass(frozen=True)
class Workload:
    """One synthetic model + partition + decode/prefill schedule."""

    cid: int
    name: str
    n_layers: int
    d_model: int
    n_heads: int
    n_kv_heads: int
    d_head: int
    d_ffn: int
    vocab: int
    head_ranges: Tuple[Tuple[int, int], ...]
    ffn_ranges: Tuple[Tuple[int, int], ...]
    kv_len: int          # tokens already cached when decoding starts
    decode_steps: int    # teacher-forced decode steps
    prompt_len: int      # prefill prompt length (0: none)
    model_id: int        # seed namespace of the weights (7B decode and 7B prefill share one model)
    rms_eps: float = 1e-5
    rope_theta: float = 1e4
    extra: Dict[str, object] = field(default_factory=dict, compare=False)

    @property
    def n_devices(self) -> int:
        return len(self.head_ranges)

    @property
    def max_seq(self) -> int:
        return max(self.kv_len + self.decode_steps, self.prompt_len) + 8

    def seed(self, layer: int, tensor: int) -> int:
        return self.model_id * 10**6 + layer * 100 + tensor

    def shape_of(self, name: str) -> Tuple[int, ...]:
        D, H, Hk, dh, F = self.d_model, self.n_heads, self.n_kv_heads, self.d_head, self.d_ffn
        return {"attn_norm": (D,), "wq": (H * dh, D), "wk": (Hk * dh, D), "wv": (Hk * dh, D),
                "wo": (D, H * dh), "ffn_norm": (D,), "w_gate": (F, D), "w_up": (F, D),
                "w_down": (D, F)}[name]

    def layer_weights(self, layer: int) -> Dict[str, np.ndarray]:
        out = {}
        for t, name in enumerate(TENSORS):
            seed = self.seed(layer, t)
            if name.endswith("norm"):
                out[name] = normal_f16(self.shape_of(name), seed, 1.0, 0.02)
            else:
                out[name] = normal_f16(self.shape_of(name), seed, 0.0, 0.02)
        return out

    def embedding(self) -> np.ndarray:
        return normal_f16((self.vocab, self.d_model), self.model_id * 10**6 + 99_000, 0.0, 0.02)

    def token_ids(self, n: int, stream: int = 0) -> np.ndarray:
        return uniform_i32(n, self.model_id * 10**6 + 99_100 + stream, 0, self.vocab)

    def hidden(self, rows: int, stream: int = 0) -> np.ndarray:
        """N(0,1) fp16 hidden states [rows, D] (a layer's teacher-forced input)."""
        return normal_f16((rows, self.d_model), self.cid * 10**6 + 98_000 + stream, 0.0, 1.0)

    def kv_fill(self, layer: int, n_pos: int, cap: int | None = None):
        """Synthetic fp16 K and V caches [Hk, cap, dh] with positions [0, n_pos) drawn, rest 0."""
        cap = n_pos if cap is None else cap
        std = 0.02 * float(np.sqrt(self.d_model))
        shape = (self.n_kv_heads, n_pos, self.d_head)
        k = normal_f16(shape, self.model_id * 10**6 + 97_000 + 2 * layer, 0.0, std)
        v = normal_f16(shape, self.model_id * 10**6 + 97_000 + 2 * layer + 1, 0.0, std)
        if cap == n_pos:
            return k, v
        kc = np.zeros((self.n_kv_heads, cap, self.d_head), np.float16)
        vc = np.zeros_like(kc)
        kc[:, :n_pos] = k
        vc[:, :n_pos] = v
        return kc, vc


def _even(total: int, n: int) -> Tuple[Tuple[int, int], ...]:
    step = total // n
    return tuple((i * step, (i + 1) * step) for i in range(n))


WORKLOADS: Dict[int, Workload] = {
    1: Workload(1, "tiny-1layer-512", 1, 512, 8, 8, 64, 1408, 32000,
                ((0, 4), (4, 8)), ((0, 704), (704, 1408)),
                kv_len=128, decode_steps=1, prompt_len=128, model_id=1),
    2: Workload(2, "llama2-7b-decode", 32, 4096, 32, 32, 128, 11008, 32000,
                _even(32, 4), _even(11008, 4),
                kv_len=1024, decode_steps=128, prompt_len=0, model_id=2),
    3: Workload(3, "llama2-13b-decode", 40, 5120, 40, 40, 128, 13824, 32000,
                ((0, 20), (20, 32), (32, 40)), ((0, 6912), (6912, 11059), (11059, 13824)),
                kv_len=2048, decode_steps=4, prompt_len=0, model_id=3),
    4: Workload(4, "llama2-7b-prefill512", 32, 4096, 32, 32, 128, 11008, 32000,
                _even(32, 4), _even(11008, 4),
                kv_len=0, decode_steps=0, prompt_len=512, model_id=2),
    5: Workload(5, "llama3-8b-gqa-decode", 32, 4096, 32, 8, 128, 14336, 128256,
                _even(32, 4), _even(14336, 4),
                kv_len=4096, decode_steps=4, prompt_len=0, model_id=5, rope_theta=5e5),
}


def small(name: str = "mini", **kw) -> Workload:
    """A small model for CPU-side checks (defaults: D=48, 4 heads of 16, 2 KV heads, F=40)."""
    args = dict(cid=90, name=name, n_layers=2, d_model=48, n_heads=4, n_kv_heads=2, d_head=16,
                d_ffn=40, vocab=97, head_ranges=((0, 2), (2, 4)), ffn_ranges=((0, 25), (25, 40)),
                kv_len=5, decode_steps=2, prompt_len=7, model_id=90)
    args.update(kw)
    return Workload(**args)
