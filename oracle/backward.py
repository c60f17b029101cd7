"""Float64 oracle for the gradient of the chunk SDPA (§3.1 Eq. 2 with the
position mask of §3.3.1), the backward the paper's fine-tuning needs.

TEST INFRASTRUCTURE ONLY (see oracle/h2o_oracle.py): only tests/ use it.

The loss is L = sum(out * dout) for the chunk's output out = SDPA(q, [k_cache;
k_new], [v_cache; v_new]) under the mask of ``sdpa_chunk``; the gradients of L
w.r.t. q, k_cache, v_cache, k_new and v_new are taken by PyTorch autograd in
float64 on CPU, through a plain restatement of the forward (masked softmax of
scale q k^T, weights times values).  Cache slots no query row sees, and empty
slots, get zero gradient.
"""
from __future__ import annotations

import math

import numpy as np
import torch

__all__ = ["sdpa_chunk_backward"]


def sdpa_chunk_backward(q, k_cache, v_cache, k_new, v_new, slot_pos, pos0: int, dout,
                        scale: float | None = None):
    """Returns (dq (B,Hq,S,d), dk_cache, dv_cache (B,Hkv,M,d), dk_new, dv_new
    (B,Hkv,S,d)) as float64 NumPy arrays."""
    f = lambda x: torch.tensor(np.asarray(x, np.float64), requires_grad=True)
    tq, tkc, tvc, tkn, tvn = f(q), f(k_cache), f(v_cache), f(k_new), f(v_new)
    B, Hq, S, d = tq.shape
    Hkv, M = k_cache.shape[1], k_cache.shape[2]
    qg = Hq // Hkv
    if scale is None:
        scale = 1.0 / math.sqrt(d)
    g = torch.tensor(np.asarray(dout, np.float64))
    loss = torch.zeros((), dtype=torch.float64)
    qpos = pos0 + torch.arange(S)[:, None]
    for b in range(B):
        for h in range(Hkv):
            keys = torch.cat([tkc[b, h], tkn[b, h]])
            vals = torch.cat([tvc[b, h], tvn[b, h]])
            t = torch.cat([torch.as_tensor(np.asarray(slot_pos[b, h], np.int64)),
                           pos0 + torch.arange(S)])
            visible = (t[None, :] >= 0) & (t[None, :] <= qpos)
            for gg in range(qg):
                hq = h * qg + gg
                a = scale * (tq[b, hq] @ keys.T)
                a = a.masked_fill(~visible, float("-inf"))
                m = torch.softmax(a, dim=-1)
                loss = loss + (m @ vals * g[b, hq]).sum()
    loss.backward()
    z = lambda t: (t.grad if t.grad is not None else torch.zeros_like(t)).numpy()
    return z(tq), z(tkc), z(tvc), z(tkn), z(tvn)
