"""Textbook Llama-style decoder in float64 from torch library calls.

An independent check of the oracle (test code only).  Each step is the
library's own routine: ``F.rms_norm``, ``F.scaled_dot_product_attention`` with
``is_causal=True`` and grouped-query heads expanded by ``repeat_interleave``
(kv head g serves query heads g*grp .. g*grp+grp-1), ``F.silu``.  RoPE is
written as a complex rotation, ``(x1 + i x2) * exp(i * pos * theta^(-2i/dh))``
on the pairs (i, i + dh/2).  That is a different formulation from the real
rotate-half code in the oracle, so a sign or index slip there shows up here.

``forward`` returns the final residual stream, the logits of every position
and, per layer, the post-RoPE q, k and the v of every position.

With ``operands="bf16"`` it is the bf16 path (every operand of a matrix
product rounded to bf16 through fp32 by torch's own conversions, sums kept in
float64): the rows entering each weight product, the queries, and the
weights of V in the attention product, taken in base 2 against the integer
ceiling of each row's largest score and normalised by the unrounded sum.
Attention is then written out (masked scores, ``torch.exp2``, one batched
product over all heads) instead of ``scaled_dot_product_attention``.
"""
from __future__ import annotations

import numpy as np
import torch
import torch.nn.functional as F

f64 = torch.float64


def as_f64(a) -> torch.Tensor:
    a = np.asarray(a)
    if a.dtype == np.uint16:
        a = (a.astype(np.uint32) << np.uint32(16)).view(np.float32)
    return torch.from_numpy(np.ascontiguousarray(a, np.float64))


def rope_complex(x: torch.Tensor, pos: torch.Tensor, theta: float) -> torch.Tensor:
    """x [n, heads, dh] rotated at positions pos [n]."""
    dh = x.shape[-1]
    half = dh // 2
    inv = float(theta) ** (-(torch.arange(half, dtype=f64) * 2.0) / dh)
    ang = pos.to(f64)[:, None] * inv[None, :]
    rot = torch.polar(torch.ones_like(ang), ang)[:, None, :]
    z = torch.complex(x[..., :half], x[..., half:]) * rot
    return torch.cat([z.real, z.imag], dim=-1)


def bf16(x: torch.Tensor) -> torch.Tensor:
    """x rounded to bf16 through fp32 (nearest even at each step), as float64."""
    return x.to(torch.float32).to(torch.bfloat16).to(f64)


def attention_bf16(q, k, v):
    """Causal attention of the bf16 path: q [H, n, dh] rounded, k, v [H, n, dh]."""
    n, dh = q.shape[1], q.shape[2]
    x = (bf16(q) @ k.transpose(1, 2)) / np.sqrt(dh) * np.log2(np.e)
    mask = torch.ones(n, n, dtype=torch.bool).triu(1)
    x = x.masked_fill(mask, -torch.inf)
    E = torch.ceil(x.max(dim=-1, keepdim=True).values)
    e = torch.exp2(x - E)
    return (bf16(e) @ v) / e.sum(dim=-1, keepdim=True)


def forward(cfg: dict, W: dict, tokens, n_layers: int | None = None,
            want_logits: bool = True, operands: str = "fp64"):
    L = cfg["n_layers"] if n_layers is None else n_layers
    d, H, G, dh = cfg["d_model"], cfg["n_heads"], cfg["n_kv_heads"], cfg["head_dim"]
    grp = H // G
    eps = cfg["rms_eps"]
    tok = torch.as_tensor(np.asarray(tokens, np.int64))
    n = tok.shape[0]
    pos = torch.arange(n)
    h = as_f64(W["embed"])[tok]
    per_layer = []
    rnd = bf16 if operands == "bf16" else (lambda x: x)
    for l in range(L):
        ly = W["layers"][l]
        a = rnd(F.rms_norm(h, (d,), weight=as_f64(ly["attn_norm"]), eps=eps))
        q = a @ as_f64(ly["wq"]).T
        k = a @ as_f64(ly["wk"]).T
        v = a @ as_f64(ly["wv"]).T
        if cfg.get("qkv_bias"):
            q = q + as_f64(ly["bq"])
            k = k + as_f64(ly["bk"])
            v = v + as_f64(ly["bv"])
        q = rope_complex(q.view(n, H, dh), pos, cfg["rope_theta"])
        k = rope_complex(k.view(n, G, dh), pos, cfg["rope_theta"])
        v = v.view(n, G, dh)
        per_layer.append(dict(q=q, k=k, v=v))
        kk = k.repeat_interleave(grp, dim=1)
        vv = v.repeat_interleave(grp, dim=1)
        if operands == "bf16":
            # the cache holds k and v in bf16
            o = attention_bf16(q.transpose(0, 1), bf16(kk).transpose(0, 1),
                               bf16(vv).transpose(0, 1))
        else:
            o = F.scaled_dot_product_attention(q.transpose(0, 1), kk.transpose(0, 1),
                                               vv.transpose(0, 1), is_causal=True)
        h = h + rnd(o.transpose(0, 1).reshape(n, H * dh)) @ as_f64(ly["wo"]).T
        b = rnd(F.rms_norm(h, (d,), weight=as_f64(ly["mlp_norm"]), eps=eps))
        act = F.silu(b @ as_f64(ly["wg"]).T) * (b @ as_f64(ly["wu"]).T)
        h = h + rnd(act) @ as_f64(ly["wd"]).T
    logits = None
    if want_logits:
        hn = rnd(F.rms_norm(h, (d,), weight=as_f64(W["final_norm"]), eps=eps))
        logits = hn @ as_f64(W["lm_head"]).T
    return dict(h=h, logits=logits, layers=per_layer)
