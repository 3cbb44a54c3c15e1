"""Brute-force attention in numpy fp64 for tiny inputs (test infrastructure).

A second formulation of the same operation, written independently of
``mcpu_oracle.c``: each row's keys and values are first materialised as dense
[S, H_kv, D] arrays by fancy indexing through the block table, the visibility
rule is an explicit boolean matrix [L, S], and softmax is taken over the whole
masked score matrix at once. It exists to pin the C oracle; it is far too slow
and memory-hungry for anything but small cases.
"""
from __future__ import annotations

import numpy as np


def bits_to_f64(a) -> np.ndarray:
    a = np.asarray(a, dtype=np.uint16)
    return (a.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def dense_kv(k_cache, v_cache, block_table_row, S, page_size):
    """Keys/values of one row in logical order: ([S, H_kv, D], [S, H_kv, D])."""
    pos = np.arange(S)
    pages = np.asarray(block_table_row)[pos // page_size]
    slots = pos % page_size
    k = bits_to_f64(k_cache)[pages, :, slots, :]
    v = bits_to_f64(v_cache)[pages, :, slots, :]
    return k, v


def visibility(S, L, window):
    """Boolean [L, S]: query i (position S - L + i) may see key j."""
    p = (S - L + np.arange(L))[:, None]
    j = np.arange(S)[None, :]
    vis = j <= p
    if window > 0:
        vis &= (p - j) < window
    return vis


def attention(q, k_cache, v_cache, block_table, seq_lens, query_start_loc, sliding_window,
              softmax_scale, page_size=16, sinks=None):
    """Return (out [T, Hq, D] float64, lse [T, Hq] float64), unrounded.
    sinks: optional [Hq] logits appended to every score row as one more
    column whose value row is zero."""
    qf = bits_to_f64(q)
    T, Hq, D = qf.shape
    Hkv = k_cache.shape[1]
    g = Hq // Hkv
    out = np.zeros((T, Hq, D))
    lse = np.full((T, Hq), -np.inf)
    for r in range(len(seq_lens)):
        S = int(seq_lens[r])
        t0, t1 = int(query_start_loc[r]), int(query_start_loc[r + 1])
        L = t1 - t0
        if L == 0:
            continue
        k, v = dense_kv(k_cache, v_cache, block_table[r], S, page_size)
        vis = visibility(S, L, sliding_window)
        # expand kv heads to q heads: q head h reads kv head h // g
        kq = np.repeat(k, g, axis=1)  # [S, Hq, D]
        vq = np.repeat(v, g, axis=1)
        scores = softmax_scale * np.einsum("lhd,shd->hls", qf[t0:t1], kq)  # [Hq, L, S]
        scores = np.where(vis[None], scores, -np.inf)
        if sinks is not None:
            # one extra key per head: score sigma_h, value 0, always visible
            sig = np.broadcast_to(np.asarray(sinks, np.float64)[:, None, None], (Hq, L, 1))
            scores = np.concatenate([scores, sig], axis=2)
            vq = np.concatenate([vq, np.zeros((1, Hq, D))], axis=0)
        m = scores.max(axis=2, keepdims=True)
        has = np.isfinite(m)
        m = np.where(has, m, 0.0)
        w = np.exp(scores - m)
        z = w.sum(axis=2, keepdims=True)
        with np.errstate(invalid="ignore", divide="ignore"):
            o = np.einsum("hls,shd->lhd", w / np.where(z > 0, z, 1.0), vq)
            l = np.where(has[..., 0], m[..., 0] + np.log(np.where(z[..., 0] > 0, z[..., 0], 1.0)), -np.inf)
        out[t0:t1] = o
        lse[t0:t1] = l.T
    return out, lse


def kv_append(k_new, v_new, k_cache, v_cache, block_table, seq_lens, query_start_loc, page_size=16):
    """Numpy fancy-index scatter of the new rows (bit copies)."""
    kc = np.array(k_cache, copy=True)
    vc = np.array(v_cache, copy=True)
    for r in range(len(seq_lens)):
        S = int(seq_lens[r])
        t0, t1 = int(query_start_loc[r]), int(query_start_loc[r + 1])
        pos = np.arange(S - (t1 - t0), S)
        pages = np.asarray(block_table[r])[pos // page_size]
        kc[pages, :, pos % page_size, :] = k_new[t0:t1]
        vc[pages, :, pos % page_size, :] = v_new[t0:t1]
    return kc, vc
