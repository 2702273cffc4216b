"""An independent fp64 decoder layer built from PyTorch library routines (CPU only).

It pins the oracle: RMSNorm is torch.nn.functional.rms_norm, projections are F.linear, attention is
F.scaled_dot_product_attention with an explicit causal mask (its default scale is 1/sqrt(dh)),
SwiGLU uses F.silu, and RoPE is written in its complex-number form (each pair (v_i, v_{i+dh/2}) is
the complex number v_i + i v_{i+dh/2}, multiplied by exp(i * pos * theta^(-2i/dh))).  The fp16
rounding points match the data contract: K and V are stored as fp16, and the combined hidden state
is fp16.  numpy performs the float64 -> float16 rounding (a single round-to-nearest-even).
"""
from __future__ import annotations

import numpy as np
import torch
import torch.nn.functional as F


def _t(a: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.asarray(a, dtype=np.float64))


def _to_f16(t: torch.Tensor) -> np.ndarray:
    return t.detach().numpy().astype(np.float16)


def _rope_complex(t: torch.Tensor, pos: torch.Tensor, theta: float) -> torch.Tensor:
    """t [rows, heads, dh] -> rotated copy."""
    dh = t.shape[-1]
    half = dh // 2
    inv = theta ** (-2.0 * torch.arange(half, dtype=torch.float64) / dh)
    ang = pos[:, None] * inv[None, :]
    rot = torch.polar(torch.ones_like(ang), ang)[:, None, :]
    z = torch.complex(t[..., :half], t[..., half:]) * rot
    return torch.cat([z.real, z.imag], dim=-1)


def layer(wl, w, x: np.ndarray, pos0: int, k_prefix: np.ndarray | None, v_prefix: np.ndarray | None,
          window: int = 0):
    """Full (unpartitioned) decoder layer on rows at positions pos0..pos0+rows-1; window > 0 bands
    the causal mask to the last `window` positions of each row (sliding-window attention).

    k_prefix / v_prefix: fp16 [Hk, pos0, dh] cache content before the call (or None when pos0 = 0).
    Returns a dict with attn_out, h (fp16), ffn_out, x_next (fp16), k_new / v_new (fp16 [Hk, rows, dh]).
    """
    D, H, Hk, dh = wl.d_model, wl.n_heads, wl.n_kv_heads, wl.d_head
    x = np.asarray(x, np.float16).reshape(-1, D)
    rows = x.shape[0]
    x64 = _t(x)
    xn = F.rms_norm(x64, (D,), weight=_t(w["attn_norm"]), eps=wl.rms_eps)
    q = F.linear(xn, _t(w["wq"])).view(rows, H, dh)
    k = F.linear(xn, _t(w["wk"])).view(rows, Hk, dh)
    v = F.linear(xn, _t(w["wv"])).view(rows, Hk, dh)
    pos = torch.arange(pos0, pos0 + rows, dtype=torch.float64)
    q = _rope_complex(q, pos, wl.rope_theta)
    k = _rope_complex(k, pos, wl.rope_theta)
    k16 = _to_f16(k).transpose(1, 0, 2)  # [Hk, rows, dh]
    v16 = _to_f16(v).transpose(1, 0, 2)
    if pos0 > 0:
        K = np.concatenate([k_prefix[:, :pos0], k16], axis=1)
        V = np.concatenate([v_prefix[:, :pos0], v16], axis=1)
    else:
        K, V = k16, v16
    g = H // Hk
    Kt = _t(K).repeat_interleave(g, dim=0)[None]  # [1, H, L, dh]
    Vt = _t(V).repeat_interleave(g, dim=0)[None]
    L = pos0 + rows
    mask = torch.arange(L)[None, :] <= (pos0 + torch.arange(rows))[:, None]
    if window > 0:
        mask &= torch.arange(L)[None, :] > (pos0 + torch.arange(rows))[:, None] - window
    o = F.scaled_dot_product_attention(q.permute(1, 0, 2)[None], Kt, Vt, attn_mask=mask)
    attn = o[0].permute(1, 0, 2).reshape(rows, H * dh)
    attn_out = F.linear(attn, _t(w["wo"]))
    h16 = _to_f16(x64 + attn_out)
    h64 = _t(h16)
    hn = F.rms_norm(h64, (D,), weight=_t(w["ffn_norm"]), eps=wl.rms_eps)
    a = F.silu(F.linear(hn, _t(w["w_gate"]))) * F.linear(hn, _t(w["w_up"]))
    ffn_out = F.linear(a, _t(w["w_down"]))
    x_next = _to_f16(h64 + ffn_out)
    return dict(attn_out=attn_out.numpy(), h=h16, ffn_out=ffn_out.numpy(), x_next=x_next,
                k_new=k16, v_new=v16)
