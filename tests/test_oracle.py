"""Pins for the fp64 oracle (CPU only).

Each test ties the oracle to something other than itself: a hand-derived
worked example of Eq. (fj), the causal / prefix / full special cases that
Section 2.1 defines by separate equations, three independent constructions
of the mask, a library attention routine, brute-force scalar loops, finite
differences, and the KV-cache invariants of Section 2.3.
"""
import math
import os

import numpy as np
import pytest
import torch

from oracle import ism_oracle as orc
from paper_2408_00539_gb300 import workloads as wl

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _parse_segments(line):
    ends, types = [], []
    for tok in line.split()[1:]:
        e, t = tok.split(":")
        ends.append(int(e))
        types.append(int(t))
    return ends, types


# ---------------------------------------------------------------- mask rule

def test_fj_worked_example():
    ends = types = None
    rows = []
    with open(os.path.join(GOLDEN, "fj_worked_example.txt")) as fh:
        for line in fh:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            if line.startswith("segments"):
                ends, types = _parse_segments(line)
            else:
                j, f = line.split()
                rows.append((int(j), int(f)))
    for j, f in rows:
        assert orc.f_of_j(j, ends, types) == f
    assert orc.f_vector(ends, types).tolist() == [f for _, f in rows]


def test_tile_map_worked_example():
    spec = {}
    classes = []
    with open(os.path.join(GOLDEN, "tilemap_tiny_bm64.txt")) as fh:
        lines = [l.strip() for l in fh if l.strip() and not l.startswith("#")]
    it = iter(lines)
    for line in it:
        if line.startswith("segments"):
            spec["seg"] = _parse_segments(line)
        elif line.startswith("classes"):
            pass
        elif line[0] in "PFE":
            classes.append(["EFP".index(c) for c in line.split()])
        else:
            key, *vals = line.split()
            spec[key] = [int(v) for v in vals]
    tm = orc.tile_map_bruteforce(*spec["seg"], spec["bm"][0], spec["bn"][0])
    assert tm["tile_class"].tolist() == classes
    assert tm["kt_full_end"].tolist() == spec["kt_full_end"]
    assert tm["kt_end"].tolist() == spec["kt_end"]
    assert tm["qt_begin"].tolist() == spec["qt_begin"]


def _random_dialogues(seed, n=40, max_len=48):
    rng = np.random.Generator(np.random.PCG64(seed))
    segs = wl.random_dialogue_set(rng, n, max_len)
    return [segs.seq(b)[2:] for b in range(segs.num_seqs)]


def test_three_mask_constructions_agree():
    for se, st in _random_dialogues(11, n=200):
        a = orc.mask_eq_fj(se, st)
        assert np.array_equal(a, orc.mask_from_causal(se, st))
        assert np.array_equal(a, orc.mask_from_prose(se, st))


def test_causal_special_case():
    # Eq. (e_causal): every query segment of length 1, or every segment an
    # answer, gives the lower-triangular (diagonal included) mask.
    for L in (1, 2, 7, 33):
        tril = np.tril(np.ones((L, L), dtype=bool))
        ends = list(range(1, L + 1))
        alt = [i % 2 for i in range(L)]
        assert np.array_equal(orc.mask_eq_fj(ends, alt), tril)
        assert np.array_equal(orc.mask_eq_fj([L], [orc.ANSWER]), tril)
        assert np.array_equal(orc.mask_eq_fj(ends, [orc.QUERY] * L), tril)


def test_prefix_special_case():
    # Eq. (e_prefix): one query+answer turn, token j sees i <= max(j, m_q).
    for L, mq in ((10, 4), (17, 1), (17, 16), (64, 37)):
        m = orc.mask_eq_fj([mq, L], [orc.QUERY, orc.ANSWER])
        for j in range(1, L + 1):
            for i in range(1, L + 1):
                assert m[j - 1, i - 1] == (i <= max(j, mq))


def test_full_special_case():
    # Eq. (e_full): one query segment spanning the sequence is bidirectional.
    for L in (1, 5, 40):
        assert orc.mask_eq_fj([L], [orc.QUERY]).all()


def test_mask_properties():
    # the rule never lets a token past the end of its own segment, always
    # includes the diagonal, and kv_end is non-decreasing (what lets cached
    # keys stay valid, Section 2.3)
    for se, st in _random_dialogues(12, n=100):
        ke = orc.kv_end(se, st)
        L = int(se[-1])
        if L == 0:
            continue
        assert np.all(ke >= np.arange(1, L + 1))
        assert np.all(np.diff(ke) >= 0)
        for start, end, kind in orc.segment_bounds(se, st):
            assert np.all(ke[start:end] <= end)


# ---------------------------------------------------------------- tile map

def _tile_map_closed_form(ke, L, bm, bn):
    """Independent derivation from kv_end monotonicity: q-tile t has
    floor(kv_end[first row] / bn) leading full tiles when all its rows are
    inside the sequence, and ceil(kv_end[last row] / bn) non-empty tiles."""
    nqt, nkt = -(-L // bm), -(-L // bn)
    cls = np.zeros((nqt, nkt), dtype=np.uint8)
    for t in range(nqt):
        r0, rl = t * bm, min(L, t * bm + bm) - 1
        full = ke[r0] // bn if t * bm + bm <= L else 0
        nz = -(-int(ke[rl]) // bn)
        cls[t, :nz] = orc.TILE_PARTIAL
        cls[t, :full] = orc.TILE_FULL
    return cls


@pytest.mark.parametrize("bm,bn", [(128, 128), (128, 64), (64, 128), (64, 64), (16, 8)])
def test_tile_map_bruteforce_vs_closed_form(bm, bn):
    rng = np.random.Generator(np.random.PCG64(bm * 1000 + bn))
    segs = wl.random_dialogue_set(rng, 12, 700)
    for b in range(segs.num_seqs):
        _, L, se, st = segs.seq(b)
        tm = orc.tile_map_bruteforce(se, st, bm, bn)
        cls = tm["tile_class"]
        assert np.array_equal(cls, _tile_map_closed_form(orc.kv_end(se, st), L, bm, bn))
        # each row reads FULL* PARTIAL* EMPTY*
        for row in cls:
            seq = "".join("EFP"[c] for c in row)
            assert seq == "F" * seq.count("F") + "P" * seq.count("P") + "E" * seq.count("E")


# ---------------------------------------------------------------- forward

def _rand(rng, *shape):
    return rng.standard_normal(shape)


def _sdpa_reference(q, k, v, mask, scale):
    """torch fp64 scaled_dot_product_attention with an explicit boolean mask
    (library routine); GQA by repeating KV heads for contiguous groups."""
    hq, hkv = q.shape[1], k.shape[1]
    qt = torch.from_numpy(q).permute(1, 0, 2)
    kt = torch.from_numpy(k).repeat_interleave(hq // hkv, dim=1).permute(1, 0, 2)
    vt = torch.from_numpy(v).repeat_interleave(hq // hkv, dim=1).permute(1, 0, 2)
    o = torch.nn.functional.scaled_dot_product_attention(
        qt, kt, vt, attn_mask=torch.from_numpy(mask), scale=scale)
    return o.permute(1, 0, 2).numpy()


def test_fwd_vs_library_sdpa():
    rng = np.random.Generator(np.random.PCG64(21))
    segs = wl.random_dialogue_set(rng, 5, 90, zero_len=True)
    T = segs.total_tokens
    q, k, v = _rand(rng, T, 4, 16), _rand(rng, T, 2, 16), _rand(rng, T, 2, 16)
    scale = 0.37
    o, lse = orc.attn_fwd(q, k, v, segs, scale)
    for b in range(segs.num_seqs):
        t0, L, se, st = segs.seq(b)
        if L == 0:
            continue
        sl = slice(t0, t0 + L)
        ref = _sdpa_reference(q[sl], k[sl], v[sl], orc.mask_from_causal(se, st), scale)
        np.testing.assert_allclose(o[sl], ref, rtol=1e-12, atol=1e-12)


def test_fwd_causal_matches_library_is_causal():
    rng = np.random.Generator(np.random.PCG64(22))
    L = 50
    segs = wl.pack([(list(range(1, L + 1)), [0] * L)])  # all queries of length 1
    q, k, v = _rand(rng, L, 2, 8), _rand(rng, L, 2, 8), _rand(rng, L, 2, 8)
    o, _ = orc.attn_fwd(q, k, v, segs, 0.5)
    ref = torch.nn.functional.scaled_dot_product_attention(
        torch.from_numpy(q).permute(1, 0, 2), torch.from_numpy(k).permute(1, 0, 2),
        torch.from_numpy(v).permute(1, 0, 2), is_causal=True, scale=0.5).permute(1, 0, 2).numpy()
    np.testing.assert_allclose(o, ref, rtol=1e-12, atol=1e-12)


def test_fwd_bruteforce_scalar_loops():
    rng = np.random.Generator(np.random.PCG64(23))
    se, st = [3, 5, 6, 9, 12], [0, 1, 0, 0, 1]
    segs = wl.pack([(se, st)])
    L, D = 12, 3
    q, k, v = _rand(rng, L, 2, D), _rand(rng, L, 1, D), _rand(rng, L, 1, D)
    scale = 0.8
    o, lse = orc.attn_fwd(q, k, v, segs, scale)
    # visibility written out per segment, from the prose of Section 2.1
    vis = {j: (list(range(0, 3)) if j < 3 else list(range(0, j + 1)) if j < 5 else
               list(range(0, 6)) if j == 5 else list(range(0, 9)) if j < 9 else
               list(range(0, j + 1))) for j in range(L)}
    for h in range(2):
        for j in range(L):
            s = [scale * sum(q[j, h, d] * k[i, 0, d] for d in range(D)) for i in vis[j]]
            mx = max(s)
            den = sum(math.exp(x - mx) for x in s)
            for d in range(D):
                num = sum(math.exp(x - mx) * v[i, 0, d] for x, i in zip(s, vis[j]))
                assert abs(o[j, h, d] - num / den) < 1e-12
            assert abs(lse[h, j] - (mx + math.log(den))) < 1e-12


def test_softmax_rows_sum_to_one_and_lse():
    rng = np.random.Generator(np.random.PCG64(24))
    se, st = [20, 45, 50, 80], [0, 1, 0, 1]
    m = orc.mask_eq_fj(se, st)
    q, k, v = _rand(rng, 80, 8), _rand(rng, 80, 8), _rand(rng, 80, 8)
    o, lse, p = orc.attn_rows(q, k, v, m, 0.3)
    np.testing.assert_allclose(p.sum(axis=1), 1.0, rtol=0, atol=1e-13)
    assert np.all(p[~m] == 0)
    s = 0.3 * q @ k.T
    direct = np.array([np.log(np.exp(s[j][m[j]]).sum()) for j in range(80)])
    np.testing.assert_allclose(lse, direct, rtol=1e-13, atol=1e-13)


def test_earlier_turn_rows_unchanged_by_appended_turns():
    # Section 2.3: no row attends past its own segment end, so appending
    # turns leaves the rows of the earlier turns unchanged.
    rng = np.random.Generator(np.random.PCG64(25))
    full_e, full_t = [30, 70, 90, 150, 170, 200], [0, 1, 0, 1, 0, 1]
    q, k, v = _rand(rng, 200, 2, 8), _rand(rng, 200, 2, 8), _rand(rng, 200, 2, 8)
    o_full, lse_full = orc.attn_fwd(q, k, v, wl.pack([(full_e, full_t)]), 0.4)
    for cut in (1, 2, 4):
        L = full_e[cut - 1]
        o_pre, lse_pre = orc.attn_fwd(q[:L], k[:L], v[:L], wl.pack([(full_e[:cut], full_t[:cut])]), 0.4)
        np.testing.assert_allclose(o_pre, o_full[:L], rtol=1e-12, atol=1e-13)
        np.testing.assert_allclose(lse_pre, lse_full[:, :L], rtol=1e-12, atol=1e-13)
    # but cutting inside a query segment changes its rows (the bidirectional
    # block is truncated), which is why the invariant is stated at segment ends
    o_mid, _ = orc.attn_fwd(q[:80], k[:80], v[:80], wl.pack([([30, 70, 80], [0, 1, 0])]), 0.4)
    assert not np.allclose(o_mid[70:80], o_full[70:80])


def test_packed_sequences_do_not_interact():
    rng = np.random.Generator(np.random.PCG64(26))
    segs = wl.pack([([10, 25], [0, 1]), ([7, 7, 30], [0, 1, 0])])
    q, k, v = _rand(rng, 55, 2, 4), _rand(rng, 55, 2, 4), _rand(rng, 55, 2, 4)
    o, _ = orc.attn_fwd(q, k, v, segs, 1.0)
    o0, _ = orc.attn_fwd(q[:25], k[:25], v[:25], wl.pack([([10, 25], [0, 1])]), 1.0)
    o1, _ = orc.attn_fwd(q[25:], k[25:], v[25:], wl.pack([([7, 7, 30], [0, 1, 0])]), 1.0)
    np.testing.assert_allclose(o[:25], o0, rtol=0, atol=1e-14)
    np.testing.assert_allclose(o[25:], o1, rtol=0, atol=1e-14)


def test_row_and_head_subsets():
    rng = np.random.Generator(np.random.PCG64(27))
    segs = wl.random_dialogue_set(rng, 3, 60, min_len=5)
    T = segs.total_tokens
    q, k, v = _rand(rng, T, 4, 8), _rand(rng, T, 2, 8), _rand(rng, T, 2, 8)
    o, lse = orc.attn_fwd(q, k, v, segs, 0.5)
    rows = np.sort(rng.choice(T, size=min(T, 17), replace=False))
    o2, lse2 = orc.attn_fwd(q, k, v, segs, 0.5, heads=[1, 3], rows=rows)
    np.testing.assert_allclose(o2[rows][:, [1, 3]], o[rows][:, [1, 3]], rtol=0, atol=1e-14)
    np.testing.assert_allclose(lse2[[1, 3]][:, rows], lse[[1, 3]][:, rows], rtol=0, atol=1e-14)


# ---------------------------------------------------------------- backward

def test_bwd_vs_finite_differences():
    rng = np.random.Generator(np.random.PCG64(31))
    segs = wl.pack([([3, 6, 8, 11], [0, 1, 0, 1]), ([4, 9], [1, 0])])
    T = segs.total_tokens
    q, k, v = _rand(rng, T, 4, 3), _rand(rng, T, 2, 3), _rand(rng, T, 2, 3)
    do = _rand(rng, T, 4, 3)
    scale = 0.7
    dq, dk, dv = orc.attn_bwd(q, k, v, do, segs, scale)

    def loss(q_, k_, v_):
        o, _ = orc.attn_fwd(q_, k_, v_, segs, scale)
        return float((o * do).sum())

    eps = 1e-6
    for x, g in ((q, dq), (k, dk), (v, dv)):
        num = np.zeros_like(x)
        for idx in np.ndindex(*x.shape):
            xp, xm = x.copy(), x.copy()
            xp[idx] += eps
            xm[idx] -= eps
            args = [q, k, v]
            pos = [a is x for a in args].index(True)
            ap, am = list(args), list(args)
            ap[pos], am[pos] = xp, xm
            num[idx] = (loss(*ap) - loss(*am)) / (2 * eps)
        np.testing.assert_allclose(g, num, rtol=1e-6, atol=1e-8)


def test_bwd_vs_library_autograd():
    rng = np.random.Generator(np.random.PCG64(32))
    segs = wl.random_dialogue_set(rng, 3, 70, min_len=3)
    T = segs.total_tokens
    q, k, v = _rand(rng, T, 4, 8), _rand(rng, T, 1, 8), _rand(rng, T, 1, 8)
    do = _rand(rng, T, 4, 8)
    scale = 0.35
    dq, dk, dv = orc.attn_bwd(q, k, v, do, segs, scale)
    for b in range(segs.num_seqs):
        t0, L, se, st = segs.seq(b)
        sl = slice(t0, t0 + L)
        qt = torch.from_numpy(q[sl]).permute(1, 0, 2).requires_grad_()
        kt = torch.from_numpy(k[sl]).permute(1, 0, 2).requires_grad_()
        vt = torch.from_numpy(v[sl]).permute(1, 0, 2).requires_grad_()
        o = torch.nn.functional.scaled_dot_product_attention(
            qt, kt.repeat_interleave(4, 0), vt.repeat_interleave(4, 0),
            attn_mask=torch.from_numpy(orc.mask_from_prose(se, st)), scale=scale)
        o.backward(torch.from_numpy(do[sl]).permute(1, 0, 2))
        np.testing.assert_allclose(dq[sl], qt.grad.permute(1, 0, 2).numpy(), rtol=1e-10, atol=1e-12)
        np.testing.assert_allclose(dk[sl], kt.grad.permute(1, 0, 2).numpy(), rtol=1e-10, atol=1e-12)
        np.testing.assert_allclose(dv[sl], vt.grad.permute(1, 0, 2).numpy(), rtol=1e-10, atol=1e-12)


def test_dq_rows_vs_library_autograd():
    # independent construction: masked SDPA in torch fp64 and autograd; the
    # row-subset dQ must equal the gradient rows it selects
    rng = np.random.Generator(np.random.PCG64(33))
    segs = wl.random_dialogue_set(rng, 3, 70, min_len=3)
    T = segs.total_tokens
    q, k, v, do = _rand(rng, T, 4, 8), _rand(rng, T, 2, 8), _rand(rng, T, 2, 8), _rand(rng, T, 4, 8)
    scale = 0.4
    rows = np.sort(rng.choice(T, size=T // 3, replace=False))
    dq = orc.attn_bwd_dq_rows(q, k, v, do, segs, scale, rows)
    qt = torch.from_numpy(q).requires_grad_()
    ot = _mask_sdpa_torch(qt, torch.from_numpy(k), torch.from_numpy(v), segs, scale)
    ot.backward(torch.from_numpy(do))
    np.testing.assert_allclose(dq[rows], qt.grad.numpy()[rows], rtol=1e-10, atol=1e-12)
    others = np.setdiff1d(np.arange(T), rows)
    assert np.isnan(dq[others]).all()


def test_dkdv_keys_vs_library_autograd():
    # independent construction: masked SDPA in torch fp64 and autograd; the
    # key-subset dK / dV must equal the gradient rows it selects, GQA summed
    rng = np.random.Generator(np.random.PCG64(34))
    segs = wl.random_dialogue_set(rng, 3, 70, min_len=3)
    T = segs.total_tokens
    q, k, v, do = _rand(rng, T, 4, 8), _rand(rng, T, 2, 8), _rand(rng, T, 2, 8), _rand(rng, T, 4, 8)
    scale = 0.4
    keys = np.sort(rng.choice(T, size=T // 3, replace=False))
    dk, dv = orc.attn_bwd_dkdv_keys(q, k, v, do, segs, scale, keys)
    kt, vt = torch.from_numpy(k).requires_grad_(), torch.from_numpy(v).requires_grad_()
    ot = _mask_sdpa_torch(torch.from_numpy(q), kt, vt, segs, scale)
    ot.backward(torch.from_numpy(do))
    np.testing.assert_allclose(dk[keys], kt.grad.numpy()[keys], rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(dv[keys], vt.grad.numpy()[keys], rtol=1e-10, atol=1e-12)
    others = np.setdiff1d(np.arange(T), keys)
    assert np.isnan(dk[others]).all() and np.isnan(dv[others]).all()


# ---------------------------------------------------------------- KV cache

def test_prefill_append_equals_rows_of_full_forward():
    # Section 2.3: reuse C_h, compute C_q, concatenate -> the new rows equal
    # the corresponding rows of one pass over the whole dialogue.
    rng = np.random.Generator(np.random.PCG64(41))
    B, Ln, hq, hkv, D = 2, 9, 4, 2, 6
    hist_e, hist_t = [5, 12, 20, 33], [0, 1, 0, 1]
    new_e, new_t = [6, 9], [0, 1]
    c = hist_e[-1]
    cap = c + Ln + 3
    kc, vc = _rand(rng, B, cap, hkv, D), _rand(rng, B, cap, hkv, D)
    qh = _rand(rng, B, c, hq, D)
    qn, kn, vn = _rand(rng, B, Ln, hq, D), _rand(rng, B, Ln, hkv, D), _rand(rng, B, Ln, hkv, D)
    o, lse = orc.prefill_append(qn, kn, vn, kc, vc, np.array([c, c]), new_e, new_t, 0.45)
    for b in range(B):
        ends = hist_e + [c + e for e in new_e]
        types = hist_t + new_t
        segs = wl.pack([(ends, types)])
        qf = np.concatenate([qh[b], qn[b]])
        kf = np.concatenate([kc[b, :c], kn[b]])
        vf = np.concatenate([vc[b, :c], vn[b]])
        of, lf = orc.attn_fwd(qf, kf, vf, segs, 0.45)
        np.testing.assert_allclose(o[b], of[c:], rtol=1e-12, atol=1e-13)
        np.testing.assert_allclose(lse[b], lf[:, c:], rtol=1e-12, atol=1e-13)


def test_decode_is_causal_step_over_whole_cache():
    rng = np.random.Generator(np.random.PCG64(42))
    B, hq, hkv, D, c = 3, 4, 1, 5, 17
    kc, vc = _rand(rng, B, c + 1, hkv, D), _rand(rng, B, c + 1, hkv, D)
    qn, kn, vn = _rand(rng, B, 1, hq, D), _rand(rng, B, 1, hkv, D), _rand(rng, B, 1, hkv, D)
    o, lse = orc.prefill_append(qn, kn, vn, kc, vc, np.array([c] * B), [1], [orc.ANSWER], 0.6)
    for b in range(B):
        keys = np.concatenate([kc[b, :c, 0], kn[b, :, 0]])
        vals = np.concatenate([vc[b, :c, 0], vn[b, :, 0]])
        for h in range(hq):
            s = 0.6 * keys @ qn[b, 0, h]
            p = np.exp(s - s.max())
            np.testing.assert_allclose(o[b, 0, h], (p / p.sum()) @ vals, rtol=1e-12, atol=1e-13)


def test_paged_append_equals_contiguous_append():
    # a paged cache holding the same keys (pages scattered over a shared pool,
    # written here key by key) gives exactly the contiguous result
    rng = np.random.Generator(np.random.PCG64(43))
    B, Ln, hq, hkv, D, ps = 3, 7, 4, 2, 6, 4
    c_lens = np.array([0, 5, 13])
    cap = int(c_lens.max()) + Ln
    kc, vc = _rand(rng, B, cap, hkv, D), _rand(rng, B, cap, hkv, D)
    qn, kn, vn = _rand(rng, B, Ln, hq, D), _rand(rng, B, Ln, hkv, D), _rand(rng, B, Ln, hkv, D)
    max_pages = (cap + ps - 1) // ps
    perm = rng.permutation(B * max_pages)
    table = perm.reshape(B, max_pages)
    kpool = np.full((B * max_pages * ps, hkv, D), np.nan)
    vpool = np.full((B * max_pages * ps, hkv, D), np.nan)
    for b in range(B):
        for p in range(int(c_lens[b])):
            page, off = divmod(p, ps)
            kpool[table[b, page] * ps + off] = kc[b, p]
            vpool[table[b, page] * ps + off] = vc[b, p]
    new_e, new_t = [3, 7], [0, 1]
    o_ref, l_ref = orc.prefill_append(qn, kn, vn, kc, vc, c_lens, new_e, new_t, 0.5)
    o, l = orc.prefill_append_paged(qn, kn, vn, kpool, vpool, ps, table, c_lens, new_e, new_t, 0.5)
    np.testing.assert_array_equal(o, o_ref)
    np.testing.assert_array_equal(l, l_ref)


# ---------------------------------------------------------------- rotary encoding

def _complex_rotate(x, angles):
    # the rotary encoding as a complex product (RoFormer): coordinates k and
    # k + D/2 are the real and imaginary parts of z_k, turned by e^{i angle}
    half = x.shape[-1] // 2
    z = (x[..., :half] + 1j * x[..., half:]) * np.exp(1j * angles)
    return np.concatenate([z.real, z.imag], axis=-1)


def test_rope_rotate_is_complex_multiplication():
    rng = np.random.Generator(np.random.PCG64(51))
    N, H, D, rows = 7, 3, 10, 40
    ang = rng.uniform(-7.0, 7.0, size=(rows, D // 2))
    cos_t, sin_t = np.cos(ang), np.sin(ang)
    pos = rng.integers(0, rows, size=N)
    x = rng.standard_normal((N, H, D))
    y = orc.rope_rotate(x, pos, cos_t, sin_t)
    np.testing.assert_allclose(y, _complex_rotate(x, ang[pos][:, None, :]), rtol=1e-13, atol=1e-13)
    # position 0 of the usual schedule is the identity; rotations keep norms
    c32, s32 = wl.rope_tables(rows, D)
    np.testing.assert_array_equal(orc.rope_rotate(x, np.zeros(N, dtype=int), c32, s32), x)
    yn = orc.rope_rotate(x, pos, c32, s32)
    np.testing.assert_allclose(np.linalg.norm(yn, axis=-1), np.linalg.norm(x, axis=-1), rtol=1e-6)


def test_rope_scores_depend_on_relative_position_only():
    # <R(p) q, R(p') k> is a function of p - p' (the property rotary encoding
    # is built for); the fp32 tables hold it to about 1e-6
    rng = np.random.Generator(np.random.PCG64(52))
    D, rows = 16, 600
    cos_t, sin_t = wl.rope_tables(rows, D)
    q, k = rng.standard_normal((1, 1, D)), rng.standard_normal((1, 1, D))
    for p, pk, shift in [(5, 2, 100), (37, 37, 400), (3, 90, 250)]:
        a = orc.rope_rotate(q, [p], cos_t, sin_t)[0, 0] @ orc.rope_rotate(k, [pk], cos_t, sin_t)[0, 0]
        b = orc.rope_rotate(q, [p + shift], cos_t, sin_t)[0, 0] @ orc.rope_rotate(k, [pk + shift], cos_t, sin_t)[0, 0]
        assert abs(a - b) < 1e-4 * (np.linalg.norm(q) * np.linalg.norm(k))


def test_rope_appends_equal_one_pass_over_rotated_dialogue():
    # two turns appended one after the other (keys rotated at their absolute
    # positions, stored, reused) give the rows of one forward pass over the
    # whole dialogue with every query and key rotated at its position
    rng = np.random.Generator(np.random.PCG64(53))
    hq, hkv, D = 4, 2, 8
    t1_e, t1_t = [4, 11], [0, 1]
    t2_e, t2_t = [3, 8], [0, 1]
    L1, L2 = t1_e[-1], t2_e[-1]
    L = L1 + L2
    ang = rng.uniform(-3.0, 3.0, size=(L + 5, D // 2))
    cos_t, sin_t = np.cos(ang), np.sin(ang)
    q, k, v = _rand(rng, L, hq, D), _rand(rng, L, hkv, D), _rand(rng, L, hkv, D)
    cap = L + 2
    kc, vc = np.zeros((1, cap, hkv, D)), np.zeros((1, cap, hkv, D))
    o1, l1, kr1 = orc.prefill_append_rope(q[None, :L1], k[None, :L1], v[None, :L1], kc, vc, [0], t1_e, t1_t,
                                          cos_t, sin_t, 0.4)
    kc[0, :L1], vc[0, :L1] = kr1[0], v[:L1]
    o2, l2, _ = orc.prefill_append_rope(q[None, L1:], k[None, L1:], v[None, L1:], kc, vc, [L1], t2_e, t2_t,
                                        cos_t, sin_t, 0.4)
    pos = np.arange(L)
    qr = _complex_rotate(q, ang[pos][:, None, :])
    kr = _complex_rotate(k, ang[pos][:, None, :])
    segs = wl.pack([(t1_e + [L1 + e for e in t2_e], t1_t + t2_t)])
    of, lf = orc.attn_fwd(qr, kr, v, segs, 0.4)
    np.testing.assert_allclose(o1[0], of[:L1], rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(o2[0], of[L1:], rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(l2[0], lf[:, L1:], rtol=1e-12, atol=1e-12)


def test_workload_generator_shapes():
    for w in (wl.tiny_fp32(), wl.mha_4k(), wl.gqa_8k(), wl.packed_32k()):
        s = w.segs
        assert s.cu_seqlens[0] == 0 and np.all(np.diff(s.cu_seqlens) > 0)
        for b in range(s.num_seqs):
            _, L, se, st = s.seq(b)
            assert se[-1] == L and np.all(np.diff(se) >= 0)
    t = wl.tiny_fp32()
    assert t.segs.seg_end.tolist() == [40, 70, 100, 160, 210, 256]
    assert wl.gqa_8k().segs.cu_seqlens.tolist() == [0, 8192, 16384]
    assert wl.packed_32k().total_tokens == 32768


# ---------------------------------------------------------------- rotary encoding, one pass

def _mask_sdpa_torch(q, k, v, segs, scale):
    """Masked attention of a packed batch in plain torch fp64 ([T, H, D]
    tensors; the masks from the prose construction), for autograd."""
    outs = []
    grp = q.shape[1] // k.shape[1]
    for b in range(segs.num_seqs):
        t0, L, se, st = segs.seq(b)
        sl = slice(t0, t0 + L)
        o = torch.nn.functional.scaled_dot_product_attention(
            q[sl].permute(1, 0, 2), k[sl].permute(1, 0, 2).repeat_interleave(grp, 0),
            v[sl].permute(1, 0, 2).repeat_interleave(grp, 0),
            attn_mask=torch.from_numpy(orc.mask_from_prose(se, st)), scale=scale)
        outs.append(o.permute(1, 0, 2))
    return torch.cat(outs, 0)


def _torch_complex_rotate(x, ang):
    half = x.shape[-1] // 2
    z = torch.complex(x[..., :half], x[..., half:]) * torch.polar(torch.ones_like(ang), ang)
    return torch.cat([z.real, z.imag], -1)


def test_seq_positions_restart_per_sequence():
    segs = wl.pack([([3, 5], [0, 1]), ([1], [1]), ([4], [0])])
    assert orc.seq_positions(segs).tolist() == [0, 1, 2, 3, 4, 0, 0, 1, 2, 3]


def test_rope_fwd_bwd_vs_library_autograd_through_complex_rotation():
    # independent construction: rotation as complex multiplication in torch,
    # masked SDPA, autograd for the gradients of the unrotated inputs
    rng = np.random.Generator(np.random.PCG64(54))
    segs = wl.random_dialogue_set(rng, 3, 60, min_len=3)
    T, hq, hkv, D = segs.total_tokens, 4, 2, 8
    q, k, v, do = _rand(rng, T, hq, D), _rand(rng, T, hkv, D), _rand(rng, T, hkv, D), _rand(rng, T, hq, D)
    ang = rng.uniform(-6.0, 6.0, size=(70, D // 2))
    scale = 0.45
    o, lse, q_rot, k_rot = orc.attn_fwd_rope(q, k, v, segs, scale, np.cos(ang), np.sin(ang))
    dq, dk, dv = orc.attn_bwd_rope(q, k, v, do, segs, scale, np.cos(ang), np.sin(ang))
    pos = np.concatenate([np.arange(segs.seq(b)[1]) for b in range(segs.num_seqs)])
    a = torch.from_numpy(ang[pos])[:, None, :]
    qt, kt, vt = (torch.from_numpy(x).requires_grad_() for x in (q, k, v))
    ot = _mask_sdpa_torch(_torch_complex_rotate(qt, a), _torch_complex_rotate(kt, a), vt, segs, scale)
    ot.backward(torch.from_numpy(do))
    np.testing.assert_allclose(o, ot.detach().numpy(), rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(q_rot, _complex_rotate(q, ang[pos][:, None, :]), rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(dq, qt.grad.numpy(), rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(dk, kt.grad.numpy(), rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(dv, vt.grad.numpy(), rtol=1e-10, atol=1e-12)


def test_rope_bwd_vs_finite_differences():
    rng = np.random.Generator(np.random.PCG64(55))
    segs = wl.pack([([3, 6, 9], [0, 1, 0]), ([2, 7], [1, 0])])
    T = segs.total_tokens
    q, k, v, do = _rand(rng, T, 2, 4), _rand(rng, T, 1, 4), _rand(rng, T, 1, 4), _rand(rng, T, 2, 4)
    ang = rng.uniform(-4.0, 4.0, size=(12, 2))
    c, s = np.cos(ang), np.sin(ang)
    scale = 0.8
    dq, dk, dv = orc.attn_bwd_rope(q, k, v, do, segs, scale, c, s)

    def loss(q_, k_, v_):
        return float((orc.attn_fwd_rope(q_, k_, v_, segs, scale, c, s)[0] * do).sum())

    eps = 1e-6
    for i, (x, g) in enumerate(((q, dq), (k, dk), (v, dv))):
        num = np.zeros_like(x)
        for idx in np.ndindex(*x.shape):
            args_p, args_m = [q, k, v], [q, k, v]
            xp, xm = x.copy(), x.copy()
            xp[idx] += eps
            xm[idx] -= eps
            args_p[i], args_m[i] = xp, xm
            num[idx] = (loss(*args_p) - loss(*args_m)) / (2 * eps)
        np.testing.assert_allclose(g, num, rtol=1e-6, atol=1e-8)


def test_rope_with_zero_angles_is_plain_attention():
    rng = np.random.Generator(np.random.PCG64(56))
    segs = wl.pack([([5, 9, 14], [0, 1, 0]), ([6], [1])])
    T = segs.total_tokens
    q, k, v, do = _rand(rng, T, 4, 6), _rand(rng, T, 2, 6), _rand(rng, T, 2, 6), _rand(rng, T, 4, 6)
    c, s = np.ones((20, 3)), np.zeros((20, 3))
    o, lse, _, _ = orc.attn_fwd_rope(q, k, v, segs, 0.3, c, s)
    o0, lse0 = orc.attn_fwd(q, k, v, segs, 0.3)
    np.testing.assert_array_equal(o, o0)
    np.testing.assert_array_equal(lse, lse0)
    for g, g0 in zip(orc.attn_bwd_rope(q, k, v, do, segs, 0.3, c, s), orc.attn_bwd(q, k, v, do, segs, 0.3)):
        np.testing.assert_array_equal(g, g0)


def test_rope_output_invariant_to_a_common_position_shift():
    # scores depend only on relative positions, so shifting every position of
    # a sequence by the same amount leaves O and LSE unchanged (tables of the
    # usual schedule, fp64 angles)
    rng = np.random.Generator(np.random.PCG64(57))
    segs = wl.pack([([4, 10, 13, 20], [0, 1, 0, 1])])
    T, D = segs.total_tokens, 8
    q, k, v = _rand(rng, T, 2, D), _rand(rng, T, 1, D), _rand(rng, T, 1, D)
    inv = 10000.0 ** (-2.0 * np.arange(D // 2) / D)
    for shift in (0, 37, 500):
        ang = (np.arange(T + shift, dtype=np.float64)[:, None] * inv[None, :])[shift:]
        o, lse, _, _ = orc.attn_fwd_rope(q, k, v, segs, 0.5, np.cos(ang), np.sin(ang))
        if shift == 0:
            o_ref, lse_ref = o, lse
        np.testing.assert_allclose(o, o_ref, rtol=1e-9, atol=1e-11)
        np.testing.assert_allclose(lse, lse_ref, rtol=1e-9, atol=1e-11)
