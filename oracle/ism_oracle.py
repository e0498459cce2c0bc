"""fp64 CPU oracle for softmax attention under the Intermittent Semi-working
Mask (ISM), arXiv 2408.00539.

TEST INFRASTRUCTURE ONLY.  This module is the independent reference that the
CUDA library is checked against.  Only ``tests/``, ``__graft_entry__.smoke()``
and the CPU-baseline / reference leg of ``bench.py`` may import it.  It shares
no code with the CUDA path and never imports it.

Everything here is the plain definition, written out slowly:

* the visibility bound f(j) of Eq. (fj) (Section 2.1), evaluated case by case
  in the paper's 1-based notation;
* the mask {(j, i) : i <= f(j)} of Eq. (e_ISM), materialised as a boolean
  matrix per sequence (no attention across packed sequences);
* softmax attention over that mask (the paper analyses the linear surrogate
  of Eq. (e_full) but applies ISM by replacing the causal mask of a softmax
  LLM, Section 2.3), with the scale exposed as a parameter because the paper
  omits it;
* the standard softmax-attention gradients;
* the KV-cache append of Section 2.3: cached keys/values of the history are
  reused, the new turn is computed and the two are concatenated;
* the tile map (empty / full / partial) by brute force over the mask;
* rotary position encoding (outside the paper's operation, which leaves
  positional encoding out): the rotation itself, the rotary append, and the
  one-pass forward / backward with queries and keys rotated at their
  positions inside their sequences.

All arithmetic is float64 on the exact input values (bf16/fp32 inputs are
upcast exactly).  Every function is pinned by ``tests/test_oracle.py``.
"""
from __future__ import annotations

from typing import Dict, Sequence, Tuple

import numpy as np

QUERY = 0
ANSWER = 1

TILE_EMPTY = 0
TILE_FULL = 1
TILE_PARTIAL = 2

ROW_BLOCK = 1024


# --------------------------------------------------------------------------
# The mask rule, Section 2.1
# --------------------------------------------------------------------------

def segment_bounds(seg_end: Sequence[int], seg_type: Sequence[int]):
    """Walk the segments of one dialogue and return (start, end, type)
    triples with 0-based half-open token ranges.  With strictly alternating
    types these are P+Q_1, A_1, Q_2, A_2, ... and the ends are the paper's
    m_{q_1}, m_{a_1}, m_{q_2}, ... (Section 2.1)."""
    out = []
    start = 0
    for e, t in zip(seg_end, seg_type):
        e = int(e)
        if e < start:
            raise ValueError("segment ends must be non-decreasing")
        out.append((start, e, int(t)))
        start = e
    return out


def f_of_j(j: int, seg_end: Sequence[int], seg_type: Sequence[int]) -> int:
    """Eq. (fj) for one 1-based token index j.

    A token in a query window m_{a_{k-1}} < j <= m_{q_k} (the prompt is part
    of the first window, first row of Eq. fj) is bounded by the end of its
    query, m_{q_k}.  A token in an answer window m_{q_k} < j <= m_{a_k} is
    bounded by itself, f(j) = j.  A query segment that directly follows
    another query segment is its own window (the equation assumes strict
    alternation; each query window keeps its own end)."""
    for start, end, kind in segment_bounds(seg_end, seg_type):
        if start < j <= end:  # 1-based j inside (start, end]
            return end if kind == QUERY else j
    raise ValueError(f"token {j} is not covered by the segments")


def f_vector(seg_end, seg_type) -> np.ndarray:
    """f(j) for j = 1..L as an int64 array (entry j-1 holds f(j)), by the
    same case rule as ``f_of_j`` applied window by window."""
    f = []
    for start, end, kind in segment_bounds(seg_end, seg_type):
        for j in range(start + 1, end + 1):
            f.append(end if kind == QUERY else j)
    return np.array(f, dtype=np.int64)


def mask_eq_fj(seg_end, seg_type, rows=None) -> np.ndarray:
    """Boolean [L, L] mask of Eq. (e_ISM): row j (0-based) may use key i
    (0-based) iff i+1 <= f(j+1), i.e. the sum of Eq. (e_ISM) runs over
    i = 1..f(j).  ``rows`` (0-based indices) selects a subset of rows."""
    f = f_vector(seg_end, seg_type)
    L = f.shape[0]
    if rows is not None:
        f = f[np.asarray(rows, dtype=np.int64)]
    i1 = np.arange(1, L + 1)[None, :]
    return i1 <= f[:, None]


def mask_from_causal(seg_end, seg_type) -> np.ndarray:
    """Second construction, Section 2.3: start from the standard causal mask
    and insert bidirectional attention over each query span."""
    L = int(seg_end[-1])
    m = np.tril(np.ones((L, L), dtype=bool))
    for start, end, kind in segment_bounds(seg_end, seg_type):
        if kind == QUERY:
            m[start:end, start:end] = True
    return m


def mask_from_prose(seg_end, seg_type) -> np.ndarray:
    """Third construction, the prose after Eq. (fj): a query token sees
    every token up to the end of its own query, prior context included; an
    answer token is strictly causal; nothing looks past the end of the
    current segment."""
    L = int(seg_end[-1])
    m = np.zeros((L, L), dtype=bool)
    for start, end, kind in segment_bounds(seg_end, seg_type):
        for j in range(start, end):
            last = end if kind == QUERY else j + 1
            m[j, :last] = True
    return m


def kv_end(seg_end, seg_type) -> np.ndarray:
    """Exclusive 0-based key bound per token: row j sees keys [0, kv_end[j]).
    Numerically kv_end[j] = f(j+1)."""
    return f_vector(seg_end, seg_type).astype(np.int32)


def packed_mask(segs) -> np.ndarray:
    """Block-diagonal [T, T] mask of a varlen batch: pairs from different
    packed sequences are never visible."""
    T = int(segs.cu_seqlens[-1])
    m = np.zeros((T, T), dtype=bool)
    for b in range(int(segs.cu_seqlens.shape[0]) - 1):
        t0, L, se, st = segs.seq(b)
        m[t0:t0 + L, t0:t0 + L] = mask_eq_fj(se, st)
    return m


# --------------------------------------------------------------------------
# Tile map (no counterpart in the paper: a classification of the mask)
# --------------------------------------------------------------------------

def tile_map_bruteforce(seg_end, seg_type, bm: int, bn: int) -> Dict[str, np.ndarray]:
    """Classify every (q-tile, k-tile) rectangle of one sequence by scanning
    the materialised mask.  A rectangle covers rows [t*bm, t*bm+bm) and
    columns [c*bn, c*bn+bn) relative to the sequence; it is FULL when it lies
    inside the sequence and every pair is visible, EMPTY when no in-bounds
    pair is visible, PARTIAL otherwise.  Also returns per q-tile the number
    of leading FULL tiles and one past the last non-empty tile, and per
    k-tile the first non-empty q-tile."""
    L = int(seg_end[-1]) if len(seg_end) else 0
    m = mask_eq_fj(seg_end, seg_type)
    nqt = -(-L // bm)
    nkt = -(-L // bn)
    cls = np.zeros((nqt, nkt), dtype=np.uint8)
    for t in range(nqt):
        r0, r1 = t * bm, t * bm + bm
        for c in range(nkt):
            c0, c1 = c * bn, c * bn + bn
            block = m[r0:min(r1, L), c0:min(c1, L)]
            if not block.any():
                cls[t, c] = TILE_EMPTY
            elif r1 <= L and c1 <= L and block.all():
                cls[t, c] = TILE_FULL
            else:
                cls[t, c] = TILE_PARTIAL
    kt_full_end = np.zeros(nqt, dtype=np.int32)
    kt_end = np.zeros(nqt, dtype=np.int32)
    for t in range(nqt):
        row = cls[t]
        n = 0
        while n < nkt and row[n] == TILE_FULL:
            n += 1
        kt_full_end[t] = n
        nz = np.nonzero(row != TILE_EMPTY)[0]
        kt_end[t] = (nz[-1] + 1) if nz.size else 0
    qt_begin = np.zeros(nkt, dtype=np.int32)
    for c in range(nkt):
        nz = np.nonzero(cls[:, c] != TILE_EMPTY)[0]
        qt_begin[c] = nz[0] if nz.size else nqt
    return {"tile_class": cls, "kt_full_end": kt_full_end, "kt_end": kt_end, "qt_begin": qt_begin}


def tile_map_packed(segs, bm: int, bn: int) -> Dict[str, np.ndarray]:
    """Concatenate the per-sequence brute-force tile maps of a varlen batch
    (row-major [nqt, nkt] per sequence, sequences in order)."""
    parts = {"tile_class": [], "kt_full_end": [], "kt_end": [], "qt_begin": [], "kv_end": []}
    for b in range(int(segs.cu_seqlens.shape[0]) - 1):
        _, _, se, st = segs.seq(b)
        tm = tile_map_bruteforce(se, st, bm, bn)
        parts["tile_class"].append(tm["tile_class"].reshape(-1))
        parts["kt_full_end"].append(tm["kt_full_end"])
        parts["kt_end"].append(tm["kt_end"])
        parts["qt_begin"].append(tm["qt_begin"])
        parts["kv_end"].append(kv_end(se, st))
    return {k: np.concatenate(v) if v else np.zeros(0) for k, v in parts.items()}


# --------------------------------------------------------------------------
# Attention, Eq. (e_ISM) with softmax (Section 2.3)
# --------------------------------------------------------------------------

def _f64(x) -> np.ndarray:
    if hasattr(x, "detach"):
        x = x.detach().to("cpu")
        import torch
        x = x.to(torch.float64).numpy()
    return np.asarray(x, dtype=np.float64)


def _group(hq: int, hkv: int, h: int) -> int:
    """Grouped-query attention: consecutive query heads share a KV head."""
    if hq % hkv:
        raise ValueError("num_heads_q must be a multiple of num_heads_kv")
    return h // (hq // hkv)


def attn_rows(q, k, v, mask, scale: float):
    """Softmax attention of query rows q [R, D] over keys k, v [N, D] under
    a boolean mask [R, N].  Returns (O [R, D], LSE [R], P [R, N]); LSE is the
    natural log of the sum of exp(scale * q.k) over visible keys."""
    s = scale * (q @ k.T)
    s = np.where(mask, s, -np.inf)
    m = s.max(axis=1, keepdims=True)
    e = np.exp(s - m)
    l = e.sum(axis=1, keepdims=True)
    p = e / l
    return p @ v, (m + np.log(l))[:, 0], p


def attn_fwd(q, k, v, segs, scale: float, heads=None, rows=None):
    """ISM attention forward over a varlen batch.

    q [T, Hq, D], k/v [T, Hkv, D] (any float type; upcast to fp64).
    Returns O [T, Hq, D] and LSE [Hq, T] as float64.  ``heads`` restricts
    the computation to a subset of query heads and ``rows`` (a sorted array
    of global token indices) to a subset of query rows; entries that are not
    computed are NaN."""
    q, k, v = _f64(q), _f64(k), _f64(v)
    T, hq, D = q.shape
    hkv = k.shape[1]
    heads = range(hq) if heads is None else heads
    o = np.full((T, hq, D), np.nan)
    lse = np.full((hq, T), np.nan)
    for b in range(int(segs.cu_seqlens.shape[0]) - 1):
        t0, L, se, st = segs.seq(b)
        if L == 0:
            continue
        if rows is None:
            want = np.arange(L)
        else:
            r = np.asarray(rows)
            want = r[(r >= t0) & (r < t0 + L)] - t0
        if want.shape[0] == 0:
            continue
        mask = mask_eq_fj(se, st, rows=want)
        for h in heads:
            g = _group(hq, hkv, h)
            kk = k[t0:t0 + L, g]
            vv = v[t0:t0 + L, g]
            for r0 in range(0, want.shape[0], ROW_BLOCK):
                idx = want[r0:r0 + ROW_BLOCK]
                ob, lb, _ = attn_rows(q[t0 + idx, h], kk, vv, mask[r0:r0 + ROW_BLOCK], scale)
                o[t0 + idx, h] = ob
                lse[h, t0 + idx] = lb
    return o, lse


def attn_bwd(q, k, v, dout, segs, scale: float):
    """Gradients of ISM attention with respect to q, k, v for the upstream
    gradient dO, from the softmax-attention chain rule:
    dV = P^T dO, dP = dO V^T, Delta = rowsum(dO * O), dS = P * (dP - Delta),
    dQ = scale * dS K, dK = scale * dS^T Q; dK and dV are summed over the
    query heads that share a KV head.  Returns float64 (dq, dk, dv)."""
    q, k, v, dout = _f64(q), _f64(k), _f64(v), _f64(dout)
    T, hq, D = q.shape
    hkv = k.shape[1]
    dq = np.zeros_like(q)
    dk = np.zeros_like(k)
    dv = np.zeros_like(v)
    for b in range(int(segs.cu_seqlens.shape[0]) - 1):
        t0, L, se, st = segs.seq(b)
        if L == 0:
            continue
        mask = mask_eq_fj(se, st)
        sl = slice(t0, t0 + L)
        for h in range(hq):
            g = _group(hq, hkv, h)
            kk, vv = k[sl, g], v[sl, g]
            for r0 in range(0, L, ROW_BLOCK):
                r1 = min(L, r0 + ROW_BLOCK)
                qq = q[t0 + r0:t0 + r1, h]
                do = dout[t0 + r0:t0 + r1, h]
                o, _, p = attn_rows(qq, kk, vv, mask[r0:r1], scale)
                dv[sl, g] += p.T @ do
                dp = do @ vv.T
                delta = (do * o).sum(axis=1, keepdims=True)
                ds = p * (dp - delta)
                dq[t0 + r0:t0 + r1, h] = scale * (ds @ kk)
                dk[sl, g] += scale * (ds.T @ qq)
    return dq, dk, dv


def attn_bwd_dq_rows(q, k, v, dout, segs, scale: float, rows):
    """dQ of ISM attention for a subset of query rows (sorted global token
    indices), every query head.  Row j of dQ needs only row j of P and of dP:
    dQ_j = scale * sum_i dS_ji k_i with dS_j = P_j * (dP_j - Delta_j),
    dP_j = dO_j V^T and Delta_j = dO_j . O_j (O_j from the same row's
    forward).  Returns float64 dq [T, Hq, D] with NaN outside ``rows``."""
    q, k, v, dout = _f64(q), _f64(k), _f64(v), _f64(dout)
    T, hq, D = q.shape
    hkv = k.shape[1]
    rows = np.asarray(rows)
    dq = np.full((T, hq, D), np.nan)
    for b in range(int(segs.cu_seqlens.shape[0]) - 1):
        t0, L, se, st = segs.seq(b)
        want = rows[(rows >= t0) & (rows < t0 + L)] - t0
        if L == 0 or want.shape[0] == 0:
            continue
        mask = mask_eq_fj(se, st, rows=want)
        for h in range(hq):
            g = _group(hq, hkv, h)
            kk, vv = k[t0:t0 + L, g], v[t0:t0 + L, g]
            qq, do = q[t0 + want, h], dout[t0 + want, h]
            o, _, p = attn_rows(qq, kk, vv, mask, scale)
            dp = do @ vv.T
            delta = (do * o).sum(axis=1, keepdims=True)
            dq[t0 + want, h] = scale * ((p * (dp - delta)) @ kk)
    return dq


def attn_bwd_dkdv_keys(q, k, v, dout, segs, scale: float, keys):
    """dK and dV of ISM attention for a subset of key rows (sorted global token
    indices), every KV head.  Key i receives contributions only from the query
    rows j that see it (i < kv_end[j], Eq. fj); each of those rows needs its
    whole softmax row (P_j over all of its visible keys, O_j, and with it
    Delta_j = dO_j . O_j), so the rows are computed in full and the
    gradients summed over them for the selected keys only:
    dV_i = sum_j P_ji dO_j, dK_i = scale * sum_j dS_ji q_j with
    dS_j = P_j * (dO_j V^T - Delta_j), summed over the query heads of the
    KV head.  Returns float64 (dk, dv) [T, Hkv, D] with NaN outside ``keys``."""
    q, k, v, dout = _f64(q), _f64(k), _f64(v), _f64(dout)
    T, hq, D = q.shape
    hkv = k.shape[1]
    keys = np.asarray(keys)
    dk = np.full((T, hkv, D), np.nan)
    dv = np.full((T, hkv, D), np.nan)
    for b in range(int(segs.cu_seqlens.shape[0]) - 1):
        t0, L, se, st = segs.seq(b)
        sel = keys[(keys >= t0) & (keys < t0 + L)] - t0
        if L == 0 or sel.shape[0] == 0:
            continue
        f = f_vector(se, st)                       # row j (0-based) sees keys [0, f[j])
        rows = np.nonzero(f > sel.min())[0]        # the rows that see at least one selected key
        mask = mask_eq_fj(se, st, rows=rows)
        dk[t0 + sel] = 0.0
        dv[t0 + sel] = 0.0
        for h in range(hq):
            g = _group(hq, hkv, h)
            kk, vv = k[t0:t0 + L, g], v[t0:t0 + L, g]
            for r0 in range(0, rows.shape[0], ROW_BLOCK):
                idx = rows[r0:r0 + ROW_BLOCK]
                qq, do = q[t0 + idx, h], dout[t0 + idx, h]
                o, _, p = attn_rows(qq, kk, vv, mask[r0:r0 + ROW_BLOCK], scale)
                delta = (do * o).sum(axis=1, keepdims=True)
                ps = p[:, sel]
                ds = ps * (do @ vv[sel].T - delta)
                dv[t0 + sel, g] += ps.T @ do
                dk[t0 + sel, g] += scale * (ds.T @ qq)
    return dk, dv


# --------------------------------------------------------------------------
# KV-cache reuse, Section 2.3
# --------------------------------------------------------------------------

def append_segments(cache_len: int, new_seg_end, new_seg_type):
    """Segments of the whole dialogue after appending a turn: the cached
    history (already complete: its rows never see past it, by the prose
    after Eq. fj) followed by the new chunk's segments shifted by the cache
    length.  The history is represented as one answer window; the rows of
    the new chunk are unaffected by how the history is segmented, since
    every new row sees all of it."""
    ends = ([cache_len] if cache_len > 0 else []) + [cache_len + int(e) for e in new_seg_end]
    types = ([ANSWER] if cache_len > 0 else []) + [int(t) for t in new_seg_type]
    return ends, types


def prefill_append(q_new, k_new, v_new, k_cache, v_cache, cache_len, new_seg_end, new_seg_type,
                   scale: float, rows=None, heads=None):
    """Append-prefill of a new turn against reused caches.

    q_new [B, Ln, Hq, D], k_new/v_new [B, Ln, Hkv, D], k_cache/v_cache
    [B, cap, Hkv, D], cache_len [B].  Keys and values of the new chunk are
    concatenated after the cached ones, [C_h; C_q], and the new rows are the
    last rows of Eq. (e_ISM) over the whole dialogue.  Returns
    (O_new [B, Ln, Hq, D], LSE_new [B, Hq, Ln]) as float64."""
    q_new, k_new, v_new = _f64(q_new), _f64(k_new), _f64(v_new)
    B, Ln, hq, D = q_new.shape
    hkv = k_new.shape[2]
    heads = range(hq) if heads is None else heads
    want = np.arange(Ln) if rows is None else np.asarray(rows)
    o = np.full((B, Ln, hq, D), np.nan)
    lse = np.full((B, hq, Ln), np.nan)
    for b in range(B):
        c = int(cache_len[b])
        kc = _f64(k_cache[b, :c])
        vc = _f64(v_cache[b, :c])
        keys = np.concatenate([kc, k_new[b]], axis=0)   # [c + Ln, Hkv, D]
        vals = np.concatenate([vc, v_new[b]], axis=0)
        ends, types = append_segments(c, new_seg_end, new_seg_type)
        mask = mask_eq_fj(ends, types, rows=c + want)   # rows of the new tokens
        for h in heads:
            g = _group(hq, hkv, h)
            ob, lb, _ = attn_rows(q_new[b, want, h], keys[:, g], vals[:, g], mask, scale)
            o[b, want, h] = ob
            lse[b, h, want] = lb
    return o, lse


def gather_pages(pool, block_table, page_size: int, n_keys: int):
    """Keys [0, n_keys) of one sequence of a paged cache, in order: key p is
    row block_table[p // page_size] * page_size + p % page_size of the pool."""
    pool = np.asarray(pool) if not hasattr(pool, "numpy") else pool
    rows = [int(block_table[p // page_size]) * page_size + p % page_size for p in range(n_keys)]
    return pool[rows]


def prefill_append_paged(q_new, k_new, v_new, k_pool, v_pool, page_size: int, block_table, cache_len,
                         new_seg_end, new_seg_type, scale: float):
    """Append-prefill against a paged cache: the same operation as
    ``prefill_append`` on the cache each sequence's block table gathers.
    block_table [B, max_pages].  Returns (O_new, LSE_new) as float64."""
    B = q_new.shape[0]
    cap = max(int(c) for c in cache_len) if B else 0
    kc = np.zeros((B, cap) + tuple(k_new.shape[2:]))
    vc = np.zeros((B, cap) + tuple(v_new.shape[2:]))
    for b in range(B):
        c = int(cache_len[b])
        kc[b, :c] = _f64(gather_pages(k_pool, block_table[b], page_size, c))
        vc[b, :c] = _f64(gather_pages(v_pool, block_table[b], page_size, c))
    return prefill_append(q_new, k_new, v_new, kc, vc, cache_len, new_seg_end, new_seg_type, scale)



# --------------------------------------------------------------------------
# Rotary position encoding of appended tokens.  Positional encoding is outside
# the paper's operation (Section 2.1 omits it; Section 2.3 applies ISM to
# models that bring their own); serving stacks rotate the new queries and
# keys by their absolute positions before the keys enter the cache.  The
# rotation is the rotary encoding of Su et al. (RoFormer) in its rotate-half
# form: coordinate k is paired with coordinate k + D/2.
# --------------------------------------------------------------------------

def rope_rotate(x, positions, cos_table, sin_table):
    """Rotate x [N, H, D] (row n at position positions[n]) pair by pair: for
    k < D/2 the pair (x_k, x_{k+D/2}) is turned by the angle whose cosine and
    sine are cos_table[p, k] and sin_table[p, k]:

        y_k       = x_k cos - x_{k+D/2} sin
        y_{k+D/2} = x_{k+D/2} cos + x_k sin

    The tables are taken as given (exact fp32 values upcast).  Returns float64."""
    x = _f64(x)
    c = _f64(cos_table)[np.asarray(positions)][:, None, :]   # [N, 1, D/2]
    s = _f64(sin_table)[np.asarray(positions)][:, None, :]
    half = x.shape[-1] // 2
    lo, hi = x[..., :half], x[..., half:]
    return np.concatenate([lo * c - hi * s, hi * c + lo * s], axis=-1)


def prefill_append_rope(q_new, k_new, v_new, k_cache, v_cache, cache_len, new_seg_end, new_seg_type,
                        cos_table, sin_table, scale: float, key_round=None):
    """Append-prefill with rotary encoding applied to the new tokens: token j
    of sequence b sits at position cache_len[b] + j; its query and key are
    rotated there (``rope_rotate``), the rotated keys are appended to the
    cache (already holding rotated keys of the history), values unchanged,
    and the new rows attend as in ``prefill_append``.  ``key_round`` maps the
    rotated keys to the values the cache stores (the cache's element type);
    None keeps them exact.  Returns (O_new, LSE_new, K_rot [B, Ln, Hkv, D])."""
    B, Ln = q_new.shape[0], q_new.shape[1]
    q_rot = np.zeros(tuple(q_new.shape))
    k_rot = np.zeros(tuple(k_new.shape))
    for b in range(B):
        pos = int(cache_len[b]) + np.arange(Ln)
        q_rot[b] = rope_rotate(q_new[b], pos, cos_table, sin_table)
        k_rot[b] = rope_rotate(k_new[b], pos, cos_table, sin_table)
    k_used = k_rot if key_round is None else _f64(key_round(k_rot))
    o, lse = prefill_append(q_rot, k_used, v_new, k_cache, v_cache, cache_len, new_seg_end, new_seg_type, scale)
    return o, lse, k_rot


# --------------------------------------------------------------------------
# Rotary position encoding on the one-pass training path.  The positions of a
# packed batch restart at every sequence: token t of sequence b (rows
# cu_seqlens[b] <= t < cu_seqlens[b+1]) sits at position t - cu_seqlens[b].
# The attention of Eq. (e_ISM) then runs on the rotated queries and keys.
# --------------------------------------------------------------------------

def seq_positions(segs) -> np.ndarray:
    """Position of every token of a varlen batch: its index inside its own
    packed sequence."""
    pos = []
    for b in range(int(segs.cu_seqlens.shape[0]) - 1):
        _, L, _, _ = segs.seq(b)
        pos.extend(range(L))
    return np.asarray(pos, dtype=np.int64)


def attn_fwd_rope(q, k, v, segs, scale: float, cos_table, sin_table, round_fn=None):
    """Forward with rotary encoding: q and k are rotated at their positions in
    their sequences (``rope_rotate``), ``round_fn`` (when given) maps the
    rotated values to those the attention is computed on (e.g. the element
    type they are stored in), then ``attn_fwd``.  Returns (O, LSE, q_rot,
    k_rot), the last two before rounding."""
    pos = seq_positions(segs)
    q_rot = rope_rotate(q, pos, cos_table, sin_table)
    k_rot = rope_rotate(k, pos, cos_table, sin_table)
    qa, ka = (q_rot, k_rot) if round_fn is None else (_f64(round_fn(q_rot)), _f64(round_fn(k_rot)))
    o, lse = attn_fwd(qa, ka, v, segs, scale)
    return o, lse, q_rot, k_rot


def attn_bwd_rope(q, k, v, dout, segs, scale: float, cos_table, sin_table, round_fn=None):
    """Gradients of the rotary forward with respect to the unrotated q, k and
    to v.  The chain rule through y = R x is dx = R^T dy, and the transpose of
    a rotation is the rotation by the opposite angle: the gradients of the
    rotated queries and keys (``attn_bwd`` on the rotated, optionally rounded,
    values) are rotated back with the sines negated."""
    pos = seq_positions(segs)
    q_rot = rope_rotate(q, pos, cos_table, sin_table)
    k_rot = rope_rotate(k, pos, cos_table, sin_table)
    if round_fn is not None:
        q_rot, k_rot = _f64(round_fn(q_rot)), _f64(round_fn(k_rot))
    dq_rot, dk_rot, dv = attn_bwd(q_rot, k_rot, v, dout, segs, scale)
    neg_sin = -_f64(sin_table)
    return rope_rotate(dq_rot, pos, cos_table, neg_sin), rope_rotate(dk_rot, pos, cos_table, neg_sin), dv
