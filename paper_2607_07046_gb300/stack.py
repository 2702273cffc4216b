"""Owns one model + partition + KV cache built through the C ABI (marshalling only)."""
from __future__ import annotations

from typing import Callable, Dict, Optional, Sequence, Tuple

import numpy as np

from . import vt


class Stack:
    """A model loaded layer by layer from `layer_fn(l) -> dict of fp16 arrays`, split by a
    partition, with a KV cache of `capacity` positions."""

    def __init__(self, shapes: vt.vt_shapes, layer_fn: Callable[[int], Dict[str, np.ndarray]],
                 head_ranges: Sequence[Tuple[int, int]], ffn_ranges: Sequence[Tuple[int, int]],
                 capacity: int, embed: Optional[np.ndarray] = None, stream=None, windows=None,
                 precision=None, layer_ranges=None):
        """windows: None, one sliding attention window for every layer, or one per layer (0: none).
        precision: None, or a function (layer, device, block) -> bits (16, 8 or 4) applied to every
        shard before the KV cache is created.  layer_ranges: None, or (head ranges per layer, FFN
        ranges per layer, flags) for vt_partition_create_layers (head_ranges / ffn_ranges then only
        give the device count)."""
        self.shapes = shapes
        self.model = self.part = self.kv = 0
        self.model = vt.vt_model_create(shapes, None, None, stream)
        for l in range(shapes.n_layers):
            vt.vt_model_load_layer(self.model, l, layer_fn(l), stream)
        if embed is not None:
            vt.vt_model_load_embedding(self.model, embed, stream)
        if windows is not None:
            ws = [windows] * shapes.n_layers if isinstance(windows, int) else list(windows)
            for l, w in enumerate(ws):
                vt.vt_model_set_window(self.model, l, w)
        if layer_ranges is not None:  # per-layer table (head ranges per layer, FFN ranges per layer, flags)
            lh, lc, flags = layer_ranges
            self.part = vt.vt_partition_create_layers(self.model, lh, lc, flags, stream)
        else:
            self.part = vt.vt_partition_create(self.model, head_ranges, ffn_ranges, stream)
        if precision is not None:
            for l in range(shapes.n_layers):
                for d in range(len(head_ranges)):
                    for blk in (vt.VT_BLOCK_ATTN, vt.VT_BLOCK_FFN):
                        bits = precision(l, d, blk)
                        if bits != 16:
                            vt.vt_partition_set_precision(self.part, (l, d, blk), bits, stream)
        self.kv = vt.vt_kv_create(self.part, capacity, stream) if capacity > 0 else 0
        self.head_ranges = list(head_ranges)
        self.ffn_ranges = list(ffn_ranges)

    @property
    def n_devices(self) -> int:
        return len(self.head_ranges)

    def close(self) -> None:
        vt.vt_kv_destroy(self.kv)
        vt.vt_partition_destroy(self.part)
        vt.vt_model_destroy(self.model)
        self.model = self.part = self.kv = 0

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()
