"""Plain fp64 CPU definition of one full backbone layer step.

TEST INFRASTRUCTURE ONLY (see the package docstring): only the tests, the
smoke check and the benchmark's CPU baseline use it.

Sec. 3.1 (Eq. 1-2): every denoising step runs the bidirectional transformer
over the step sequence [v_t || q || y^(t-1)] and reads the answer positions'
token distributions.  The paper does not print its backbones' layers; the
reading here is a pre-normalization decoder layer without a causal mask, the
layout of the 8B-class backbones it uses:

  h   = rmsnorm(x, g1)
  q,k,v = h Wq^T, h Wk^T, h Wv^T;  q, k rotated by the row's position
  x   = x + attention(q, k, v) Wo^T        (per request, all rows see all rows)
  h   = rmsnorm(x, g2)
  x   = x + (silu(h Wg^T) * (h Wu^T)) Wd^T
  logits of the answer rows = rmsnorm(x_answers, gf) Wlm^T

Every function works in float64 on numpy arrays; matrix products use numpy's
matmul (a library primitive) and nothing is blocked, fused or reordered.
"""
from __future__ import annotations

import numpy as np


def rmsnorm(x, gamma, eps: float):
    """x / sqrt(mean(x^2) + eps) * gamma, per row."""
    x = np.asarray(x, np.float64)
    return x / np.sqrt((x * x).mean(axis=-1, keepdims=True) + eps) * np.asarray(gamma, np.float64)


def rope_angles(pos, head_dim: int, theta: float):
    """angle[p, d] = pos_p * theta^(-2d/head_dim) for d < head_dim/2."""
    half = head_dim // 2
    inv = theta ** (-np.arange(half, dtype=np.float64) / half)
    return np.asarray(pos, np.float64)[:, None] * inv[None, :]


def rope(x, pos, n_heads: int, head_dim: int, theta: float):
    """Rotary position embedding of each head: the pair (d, d + D/2) of row p
    is rotated by angle(p, d).  x: [N, n_heads * head_dim]."""
    x = np.asarray(x, np.float64)
    n = x.shape[0]
    half = head_dim // 2
    ang = rope_angles(pos, head_dim, theta)[:, None, :]
    c, s = np.cos(ang), np.sin(ang)
    xh = x.reshape(n, n_heads, head_dim)
    a, b = xh[..., :half], xh[..., half:]
    return np.concatenate([a * c - b * s, b * c + a * s], axis=-1).reshape(n, n_heads * head_dim)


def silu(g):
    g = np.asarray(g, np.float64)
    return g / (1.0 + np.exp(-g))


def positions(cu):
    """Position of every row in its request: row - cu[b]."""
    cu = np.asarray(cu, np.int64)
    pos = np.empty(int(cu[-1]), np.int64)
    for b in range(len(cu) - 1):
        pos[cu[b]:cu[b + 1]] = np.arange(cu[b + 1] - cu[b])
    return pos


def attention(q, k, v, cu, n_heads: int, head_dim: int, scale: float):
    """Bidirectional attention (Eq. 1) per request and head: softmax(q k^T *
    scale) v over the request's rows."""
    n = q.shape[0]
    out = np.zeros((n, n_heads * head_dim))
    qh = q.reshape(n, n_heads, head_dim)
    kh = k.reshape(n, n_heads, head_dim)
    vh = v.reshape(n, n_heads, head_dim)
    for b in range(len(cu) - 1):
        s0, s1 = int(cu[b]), int(cu[b + 1])
        if s1 == s0:
            continue
        for h in range(n_heads):
            sc = qh[s0:s1, h] @ kh[s0:s1, h].T * scale
            sc -= sc.max(axis=1, keepdims=True)
            p = np.exp(sc)
            p /= p.sum(axis=1, keepdims=True)
            out[s0:s1, h * head_dim:(h + 1) * head_dim] = p @ vh[s0:s1, h]
    return out


def layer(x, wts: dict, cu, n_heads: int, head_dim: int, theta: float, eps: float):
    """One layer on the packed rows x [N, C] of all requests (cu: boundaries).

    wts: g1 [C], wq, wk, wv [HD, C], wo [C, HD], g2 [C], wg, wu [F, C],
    wd [C, F] (all float64 or anything numpy converts)."""
    x = np.asarray(x, np.float64)
    f = {k: np.asarray(v, np.float64) for k, v in wts.items()}
    pos = positions(cu)
    h = rmsnorm(x, f["g1"], eps)
    q = rope(h @ f["wq"].T, pos, n_heads, head_dim, theta)
    k = rope(h @ f["wk"].T, pos, n_heads, head_dim, theta)
    v = h @ f["wv"].T
    x = x + attention(q, k, v, cu, n_heads, head_dim, 1.0 / np.sqrt(head_dim)) @ f["wo"].T
    h = rmsnorm(x, f["g2"], eps)
    return x + (silu(h @ f["wg"].T) * (h @ f["wu"].T)) @ f["wd"].T


def answer_logits(x, cu, resp, gamma, w_lm, eps: float):
    """Logits of the answer rows (the last resp[b] rows of each request)."""
    x = np.asarray(x, np.float64)
    rows = np.concatenate([np.arange(int(cu[b + 1]) - int(resp[b]), int(cu[b + 1])) for b in range(len(resp))])
    return rmsnorm(x[rows], gamma, eps) @ np.asarray(w_lm, np.float64).T
