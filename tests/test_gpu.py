"""GPU parity tests: the CUDA path through the C ABI against the fp64 oracle
on identical seeded inputs.

Tolerances: tile maps bit-exact; bf16 inputs (fp32 accumulation) max-abs
2e-2 and mean-abs 2e-3 on O, dQ, dK, dV; fp32 inputs max-abs 1e-4; LSE 1e-3
(bf16) and 1e-5 (fp32) absolute.
"""
import os

import numpy as np
import pytest
import torch

from oracle import ism_oracle as orc
from paper_2408_00539_gb300 import workloads as wl

pytestmark = pytest.mark.gpu

BF16_MAX, BF16_MEAN, FP32_MAX = 2e-2, 2e-3, 1e-4


@pytest.fixture(scope="module")
def ism():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2408_00539_gb300 import ism as m
    m.load(build_if_missing=True)
    return m


DEV = "cuda:0"


def _np(t):
    return t.detach().float().cpu().numpy().astype(np.float64) if t.dtype != torch.float64 else t.cpu().numpy()


def _cmp(name, got, ref, dtype):
    got = _np(got) if isinstance(got, torch.Tensor) else got
    assert got.shape == ref.shape, (name, got.shape, ref.shape)
    assert np.all(np.isfinite(got)), f"{name}: non-finite values"
    err = np.abs(got - ref)
    if dtype == "fp32":
        assert err.max() <= FP32_MAX, f"{name}: max abs err {err.max():.3e}"
    else:
        assert err.max() <= BF16_MAX, f"{name}: max abs err {err.max():.3e}"
        assert err.mean() <= BF16_MEAN, f"{name}: mean abs err {err.mean():.3e}"


def _cmp_lse(name, got, ref, dtype):
    got = _np(got)
    err = np.abs(got - ref)
    assert err.max() <= (1e-5 if dtype == "fp32" else 1e-3), f"{name}: max abs err {err.max():.3e}"


def _run_pass(ism, w, seed_offset=0, minimal_workspace=False):
    q, k, v, do = wl.attention_tensors(w, seed_offset=seed_offset)
    segs = ism.Segments.from_workload(w.segs, DEV)
    qd, kd, vd, dod = (t.to(DEV) for t in (q, k, v, do))
    o, lse = ism.fwd(segs, qd, kd, vd, w.softmax_scale)
    dq, dk, dv = ism.bwd(segs, qd, kd, vd, o, lse, dod, w.softmax_scale, minimal_workspace=minimal_workspace)
    ism.check_status()
    return (q, k, v, do), (o, lse, dq, dk, dv)


# ---------------------------------------------------------------- tile map

def _tile_cases():
    rng = np.random.Generator(np.random.PCG64(101))
    yield "random", wl.random_dialogue_set(rng, 40, 700)
    yield "edges", wl.pack([([1], [1]), ([0, 0, 1], [0, 1, 0]), ([5, 5, 129], [0, 0, 1]),
                            ([128, 256], [0, 1]), ([127, 128, 129], [1, 0, 0]), ([0, 0], [0, 1])])
    yield "gqa_8k", wl.gqa_8k().segs
    yield "packed_32k", wl.packed_32k().segs


@pytest.mark.parametrize("bm,bn", [(128, 128), (128, 64), (64, 128), (64, 64)])
def test_tile_map_bit_exact(ism, bm, bn):
    for name, segs_np in _tile_cases():
        segs = ism.Segments.from_workload(segs_np, DEV)
        got = ism.tile_map(segs, bm, bn)
        ref = orc.tile_map_packed(segs_np, bm, bn)
        for key in ("tile_class", "kt_full_end", "kt_end", "qt_begin", "kv_end"):
            g = got[key].cpu().numpy()
            r = np.asarray(ref[key]).astype(g.dtype)
            assert np.array_equal(g, r), f"{name} {key} bm={bm} bn={bn}"


# ---------------------------------------------------------------- one pass

def test_tiny_fp32_fwd_bwd(ism):
    w = wl.tiny_fp32()
    (q, k, v, do), (o, lse, dq, dk, dv) = _run_pass(ism, w)
    o_ref, lse_ref = orc.attn_fwd(q, k, v, w.segs, w.softmax_scale)
    dq_ref, dk_ref, dv_ref = orc.attn_bwd(q, k, v, do, w.segs, w.softmax_scale)
    _cmp("o", o, o_ref, "fp32")
    _cmp_lse("lse", lse, lse_ref, "fp32")
    _cmp("dq", dq, dq_ref, "fp32")
    _cmp("dk", dk, dk_ref, "fp32")
    _cmp("dv", dv, dv_ref, "fp32")


def _small_bf16(d, hq=8, hkv=2, seed=9):
    segs = wl.pack([([70, 150, 170, 300], [0, 1, 0, 1]),      # ragged 300
                    ([33, 90, 200, 517], [0, 1, 0, 1]),        # several tiles + tail
                    ([129], [0]),                              # one query segment: full attention
                    ([1], [1]),                                # single token
                    ([0, 64, 64, 128, 256], [1, 0, 1, 0, 1]),  # tile-aligned, zero-length segment
                    ([50, 51, 52, 383], [0, 0, 1, 0])])        # adjacent queries, long final query
    return wl.Workload(f"small_d{d}", segs, hq, hkv, d, "bf16", d ** -0.5, 0.5, seed)


@pytest.mark.parametrize("d", [128, 64])
@pytest.mark.parametrize("path", ["default", "recompute_dq", "cuda_cores"])
def test_small_bf16_fwd_bwd(ism, d, path, knobs):
    if path == "cuda_cores":
        knobs("ISM_FORCE_CUDA_CORES", "1")
    w = _small_bf16(d)
    _check_small(ism, w, path)


@pytest.mark.parametrize("hq,hkv", [(4, 4), (6, 2), (2, 1)])
def test_small_bf16_group_sizes(ism, hq, hkv):
    """Query heads per KV head 1 and 3 (one-head forward kernel) and 2."""
    _check_small(ism, _small_bf16(128, hq=hq, hkv=hkv, seed=hq * 10 + hkv), "default")


def test_small_bf16_odd_heads_odd_tokens(ism):
    """Three query heads on one KV head and an odd number of tokens: the
    backward's Delta pass pairs (row, head) items with 16-lane groups, two to
    a warp, and here the two groups of a warp run different numbers of
    rounds."""
    segs = wl.pack([([70, 150, 170, 301], [0, 1, 0, 1]), ([33, 90, 200, 517], [0, 1, 0, 1]), ([1], [1])])
    assert segs.total_tokens % 2 == 1
    w = wl.Workload("odd_heads", segs, 3, 1, 128, "bf16", 128 ** -0.5, 0.5, 23)
    _check_small(ism, w, "default")


def _check_small(ism, w, path):
    (q, k, v, do), (o, lse, dq, dk, dv) = _run_pass(ism, w, minimal_workspace=path == "recompute_dq")
    o_ref, lse_ref = orc.attn_fwd(q, k, v, w.segs, w.softmax_scale)
    dq_ref, dk_ref, dv_ref = orc.attn_bwd(q, k, v, do, w.segs, w.softmax_scale)
    _cmp("o", o, o_ref, "bf16")
    _cmp_lse("lse", lse, lse_ref, "bf16")
    _cmp("dq", dq, dq_ref, "bf16")
    _cmp("dk", dk, dk_ref, "bf16")
    _cmp("dv", dv, dv_ref, "bf16")


def test_special_cases_match_causal_and_full(ism):
    # every token its own answer -> causal; one query segment -> full attention
    L = 300
    segs_np = wl.pack([([L], [wl.ANSWER]), ([L], [wl.QUERY])])
    w = wl.Workload("special", segs_np, 4, 4, 128, "bf16", 128 ** -0.5, 0.5, 13)
    q, k, v, _ = wl.attention_tensors(w)
    segs = ism.Segments.from_workload(segs_np, DEV)
    o, _ = ism.fwd(segs, q.to(DEV), k.to(DEV), v.to(DEV), w.softmax_scale)
    qf, kf, vf = (t.double().permute(1, 0, 2) for t in (q, k, v))
    causal = torch.nn.functional.scaled_dot_product_attention(qf[:, :L], kf[:, :L], vf[:, :L], is_causal=True,
                                                              scale=w.softmax_scale)
    full = torch.nn.functional.scaled_dot_product_attention(qf[:, L:], kf[:, L:], vf[:, L:], scale=w.softmax_scale)
    _cmp("causal", o[:L], causal.permute(1, 0, 2).numpy(), "bf16")
    _cmp("full", o[L:], full.permute(1, 0, 2).numpy(), "bf16")


def test_earlier_turn_rows_unchanged(ism):
    # Section 2.3: appending turns leaves earlier rows unchanged; with the
    # history ending on a 128-token tile boundary the GPU rows are identical.
    full = wl.pack([([100, 256, 300, 512], [0, 1, 0, 1])])
    pre = wl.pack([([100, 256], [0, 1])])
    w = wl.Workload("inv", full, 4, 2, 128, "bf16", 128 ** -0.5, 0.5, 17)
    q, k, v, _ = wl.attention_tensors(w)
    o_full, l_full = ism.fwd(ism.Segments.from_workload(full, DEV), q.to(DEV), k.to(DEV), v.to(DEV), w.softmax_scale)
    o_pre, l_pre = ism.fwd(ism.Segments.from_workload(pre, DEV), q[:256].contiguous().to(DEV),
                           k[:256].contiguous().to(DEV), v[:256].contiguous().to(DEV), w.softmax_scale)
    assert torch.equal(o_full[:256], o_pre)
    assert torch.equal(l_full[:, :256], l_pre)


def test_empty_batch_is_noop(ism):
    segs = ism.Segments.from_numpy([0, 0], [0, 0], [], [], DEV)
    q = torch.zeros((0, 4, 128), dtype=torch.bfloat16, device=DEV)
    k = torch.zeros((0, 2, 128), dtype=torch.bfloat16, device=DEV)
    o, lse = ism.fwd(segs, q, k, k, 0.1)
    assert o.shape == (0, 4, 128)
    ism.check_status()


def test_bounded_wait_reports_timeout(ism):
    assert ism.debug_timeout_probe(64) == 4          # ISM_ERR_TIMEOUT read back from the status word
    ism.check_status()                               # cleared: the context is still usable
    x = torch.ones(4, device=DEV)
    assert float(x.sum()) == 4.0


# ---------------------------------------------------------------- full sizes

def _largest_seq(segs):
    lens = np.diff(segs.cu_seqlens)
    return int(np.argmax(lens))


def _check_group(w, b, g, inputs, outputs):
    """One sequence b and KV head g of a full-size launch against the oracle:
    O and LSE of the group's query heads, dQ of those heads, dK and dV of g."""
    (q, k, v, do), (o, lse, dq, dk, dv) = inputs, outputs
    t0, L, se, st = w.segs.seq(b)
    grp = w.num_heads_q // w.num_heads_kv
    hs = slice(g * grp, (g + 1) * grp)
    sub = wl.pack([(se, st)])
    sl = slice(t0, t0 + L)
    qs, dos = q[sl][:, hs].contiguous(), do[sl][:, hs].contiguous()
    ks, vs = k[sl][:, g:g + 1].contiguous(), v[sl][:, g:g + 1].contiguous()
    o_ref, lse_ref = orc.attn_fwd(qs, ks, vs, sub, w.softmax_scale)
    dq_ref, dk_ref, dv_ref = orc.attn_bwd(qs, ks, vs, dos, sub, w.softmax_scale)
    tag = f"seq {b} (rows {t0}..{t0 + L}) kv head {g}"
    _cmp(f"o {tag}", o[sl][:, hs], o_ref, "bf16")
    _cmp_lse(f"lse {tag}", lse[hs][:, sl], lse_ref, "bf16")
    _cmp(f"dq {tag}", dq[sl][:, hs], dq_ref, "bf16")
    _cmp(f"dk {tag}", dk[sl][:, g:g + 1], dk_ref, "bf16")
    _cmp(f"dv {tag}", dv[sl][:, g:g + 1], dv_ref, "bf16")


@pytest.mark.parametrize("make", [wl.mha_4k, wl.gqa_8k, wl.packed_32k], ids=["mha_4k", "gqa_8k", "packed_32k"])
def test_full_size_parity_sampled_groups(ism, make):
    """Full-size launch (all sequences, all heads, as benchmarked); the oracle
    recomputes complete GQA groups: the first and the last KV head of the
    longest sequence, and for the packed buffer also the last dialogue, which
    starts at an offset that is not a multiple of the 128-row tile; and O,
    LSE and dQ of every query head on sampled rows of every sequence.  Every
    output element of the launch must be finite."""
    w = make()
    inputs, outputs = _run_pass(ism, w)
    for name, t in zip(("o", "lse", "dq", "dk", "dv"), outputs):
        assert bool(torch.isfinite(t).all()), f"{name}: non-finite values"
    b = _largest_seq(w.segs)
    checks = [(b, 0), (b, w.num_heads_kv - 1)]
    if w.segs.num_seqs > 1 and w.name.startswith("packed"):
        last = w.segs.num_seqs - 1
        assert int(w.segs.cu_seqlens[last]) % 128 != 0, "the last dialogue should start off a tile boundary"
        checks.append((last, w.num_heads_kv // 2))
    for bb, g in dict.fromkeys(checks):
        _check_group(w, bb, g, inputs, outputs)
    _check_all_heads_sampled_rows(w, inputs, outputs)


def _sample_rows(segs, rng, n_random=24):
    """Global rows to check at full size: each sequence's first and last rows,
    the first and last row of every segment, and random rows."""
    rows = set()
    for b in range(segs.num_seqs):
        t0, L, se, st = segs.seq(b)
        start = 0
        for e in se.tolist():
            if e > start:
                rows.update((t0 + start, t0 + e - 1))
            start = e
        rows.update(int(t0 + x) for x in rng.integers(0, L, size=n_random))
    return np.array(sorted(rows), dtype=np.int64)


def _check_all_heads_sampled_rows(w, inputs, outputs):
    """Every query head of the full-size launch on sampled rows: O and LSE of
    a row need only that row's forward, and dQ of a row only that row's P and
    dP, so the oracle computes them row by row for all 32 heads."""
    (q, k, v, do), (o, lse, dq, dk, dv) = inputs, outputs
    rows = _sample_rows(w.segs, np.random.Generator(np.random.PCG64(w.seed + 99)))
    o_ref, lse_ref = orc.attn_fwd(q, k, v, w.segs, w.softmax_scale, rows=rows)
    dq_ref = orc.attn_bwd_dq_rows(q, k, v, do, w.segs, w.softmax_scale, rows)
    _cmp(f"o, all heads, {rows.size} rows", o[rows], o_ref[rows], "bf16")
    _cmp_lse(f"lse, all heads, {rows.size} rows", lse[:, rows], lse_ref[:, rows], "bf16")
    _cmp(f"dq, all heads, {rows.size} rows", dq[rows], dq_ref[rows], "bf16")


@pytest.mark.parametrize("schedule", ["stored_ds", "recompute_dq"])
def test_mid_size_every_head_gqa32_8(ism, schedule):
    """The headline head layout (32 query heads over 8 KV heads, head_dim
    128, bf16) on two dialogues of 1536 and 700 tokens packed back to back,
    every head of O, LSE, dQ, dK and dV against the oracle, under both
    backward schedules."""
    rng = np.random.Generator(np.random.PCG64(2024))
    segs = wl.pack([wl.draw_dialogue(rng, 1536, 4, 16), wl.draw_dialogue(rng, 700, 2, 8)])
    w = wl.Workload("mid_gqa32_8", segs, 32, 8, 128, "bf16", 128 ** -0.5, 0.5, 77)
    (q, k, v, do), (o, lse, dq, dk, dv) = _run_pass(ism, w, minimal_workspace=schedule == "recompute_dq")
    if schedule == "stored_ds":
        assert ism.bwd_workspace_size(ism.Segments.from_workload(segs, DEV), q, k, w.softmax_scale) > \
            ism.bwd_workspace_size(ism.Segments.from_workload(segs, DEV), q, k, w.softmax_scale, minimal=True)
    o_ref, lse_ref = orc.attn_fwd(q, k, v, w.segs, w.softmax_scale)
    dq_ref, dk_ref, dv_ref = orc.attn_bwd(q, k, v, do, w.segs, w.softmax_scale)
    for h in range(w.num_heads_q):
        _cmp(f"o head {h}", o[:, h], o_ref[:, h], "bf16")
        _cmp_lse(f"lse head {h}", lse[h], lse_ref[h], "bf16")
        _cmp(f"dq head {h}", dq[:, h], dq_ref[:, h], "bf16")
    for g in range(w.num_heads_kv):
        _cmp(f"dk kv head {g}", dk[:, g], dk_ref[:, g], "bf16")
        _cmp(f"dv kv head {g}", dv[:, g], dv_ref[:, g], "bf16")


# ---------------------------------------------------------------- KV cache

def _append_inputs(B, cap, c_lens, l_new, hq, hkv, d, seed, std=0.5):
    rng = np.random.Generator(np.random.PCG64(seed))
    kc = wl.round_to(wl.normal(rng, (B, cap, hkv, d), std), "bf16")
    vc = wl.round_to(wl.normal(rng, (B, cap, hkv, d), std), "bf16")
    qn = wl.round_to(wl.normal(rng, (B, l_new, hq, d), std), "bf16")
    kn = wl.round_to(wl.normal(rng, (B, l_new, hkv, d), std), "bf16")
    vn = wl.round_to(wl.normal(rng, (B, l_new, hkv, d), std), "bf16")
    return kc, vc, qn, kn, vn


@pytest.mark.parametrize("l_new,segs,hq,hkv", [(200, ([40, 41, 120, 200], [0, 1, 0, 1]), 8, 2),
                                                (128, ([128], [0]), 8, 2), (1, ([1], [1]), 8, 2),
                                                (37, ([37], [0]), 8, 2),
                                                (200, ([40, 41, 120, 200], [0, 1, 0, 1]), 3, 3),
                                                (200, ([40, 41, 120, 200], [0, 1, 0, 1]), 6, 2)])
def test_prefill_append_small(ism, l_new, segs, hq, hkv):
    B, d = 3, 128
    c_lens = np.array([0, 77, 300], dtype=np.int32)
    cap = 300 + l_new + 5
    kc, vc, qn, kn, vn = _append_inputs(B, cap, c_lens, l_new, hq, hkv, d, seed=l_new)
    kcd, vcd = kc.to(DEV), vc.to(DEV)
    cl = torch.from_numpy(c_lens.copy()).to(DEV)
    scale = d ** -0.5
    o, lse = ism.prefill_append(qn.to(DEV), kn.to(DEV), vn.to(DEV), kcd, vcd, cl, c_lens, segs[0], segs[1], scale)
    ism.check_status()
    assert cl.cpu().numpy().tolist() == (c_lens + l_new).tolist()
    for b in range(B):
        c = int(c_lens[b])
        assert torch.equal(kcd[b, c:c + l_new].cpu(), kn[b]) and torch.equal(vcd[b, c:c + l_new].cpu(), vn[b])
        assert torch.equal(kcd[b, :c].cpu(), kc[b, :c])
    o_ref, lse_ref = orc.prefill_append(qn, kn, vn, kc, vc, c_lens, segs[0], segs[1], scale)
    _cmp("o_new", o, o_ref, "bf16")
    _cmp_lse("lse_new", lse, np.transpose(lse_ref, (1, 0, 2)), "bf16")


def test_prefill_append_matches_one_pass_rows(ism):
    # the appended turn's rows equal the rows of one pass over the whole dialogue
    hist = ([100, 256], [0, 1])
    new = ([60, 200], [0, 1])
    c, Ln, hq, hkv, d = 256, 200, 8, 2, 128
    full = wl.pack([(hist[0] + [c + e for e in new[0]], hist[1] + new[1])])
    w = wl.Workload("app", full, hq, hkv, d, "bf16", d ** -0.5, 0.5, 23)
    q, k, v, _ = wl.attention_tensors(w)
    o_full, _ = ism.fwd(ism.Segments.from_workload(full, DEV), q.to(DEV), k.to(DEV), v.to(DEV), w.softmax_scale)
    cap = c + Ln
    kc = torch.zeros((1, cap, hkv, d), dtype=torch.bfloat16)
    vc = torch.zeros((1, cap, hkv, d), dtype=torch.bfloat16)
    kc[0, :c], vc[0, :c] = k[:c], v[:c]
    cl = torch.tensor([c], dtype=torch.int32, device=DEV)
    o_app, _ = ism.prefill_append(q[None, c:].contiguous().to(DEV), k[None, c:].contiguous().to(DEV),
                                  v[None, c:].contiguous().to(DEV), kc.to(DEV), vc.to(DEV), cl, np.array([c]),
                                  new[0], new[1], w.softmax_scale)
    diff = (o_app[0].float() - o_full[c:].float()).abs().max().item()
    assert diff <= 2e-2, diff


@pytest.mark.parametrize("path", ["tensor_cores", "cuda_cores"])
@pytest.mark.parametrize("hq,hkv", [(8, 2), (4, 4), (8, 1), (4, 2), (6, 2), (10, 2), (7, 1), (16, 1), (40, 2)])
def test_decode_steps_small(ism, hq, hkv, path, knobs):
    """Group sizes 1-16 run the decode kernels (the tensor-core kernel, or the
    CUDA-core ones padded to a power of two), 20 the forward kernels."""
    if path == "cuda_cores":
        knobs("ISM_DECODE_NO_TC", "1")
    B, d, c0, steps = 2, 128, 700, 6
    cap = c0 + steps
    kc, vc, qn, kn, vn = _append_inputs(B, cap, None, steps, hq, hkv, d, seed=31)
    kcd, vcd = kc.clone().to(DEV), vc.clone().to(DEV)
    c_start = np.array([c0, c0 - 123], dtype=np.int32)
    c_host = c_start.copy()
    cl = torch.from_numpy(c_host.copy()).to(DEV)
    scale = d ** -0.5
    for t in range(steps):
        o, lse = ism.prefill_append(qn[:, t:t + 1].contiguous().to(DEV), kn[:, t:t + 1].contiguous().to(DEV),
                                    vn[:, t:t + 1].contiguous().to(DEV), kcd, vcd, cl, c_host, [1], [1], scale)
        # the cache the oracle sees: the initial one plus the tokens of the earlier steps
        kc_now, vc_now = kc.clone(), vc.clone()
        for b in range(B):
            kc_now[b, c_start[b]:c_start[b] + t] = kn[b, :t]
            vc_now[b, c_start[b]:c_start[b] + t] = vn[b, :t]
        o_ref, lse_ref = orc.prefill_append(qn[:, t:t + 1], kn[:, t:t + 1], vn[:, t:t + 1], kc_now, vc_now,
                                            c_host, [1], [1], scale)
        _cmp(f"decode o step {t}", o, o_ref, "bf16")
        _cmp_lse(f"decode lse step {t}", lse, np.transpose(lse_ref, (1, 0, 2)), "bf16")
        c_host = c_host + 1
    ism.check_status()
    assert cl.cpu().numpy().tolist() == c_host.tolist()


def test_append_16k_prefill_and_decode(ism):
    """Cache of 16384 tokens (batch 8, 32/8 heads, d 128), a new 512-token
    query segment, then 256 answer decode steps; the oracle checks one
    (sequence, KV group) for the prefill and for a sample of decode steps."""
    a = wl.append_16k()
    B, cap, hq, hkv, d = a.batch, a.capacity, a.num_heads_q, a.num_heads_kv, a.head_dim
    rng = np.random.Generator(np.random.PCG64(a.seed))
    kcd = torch.empty((B, cap, hkv, d), dtype=torch.bfloat16, device=DEV)
    vcd = torch.empty_like(kcd)
    b, g = 5, 3
    hs = list(range(g * hq // hkv, (g + 1) * hq // hkv))
    for bb in range(B):  # generate per sequence to bound host memory
        kh = wl.round_to(wl.normal(rng, (cap, hkv, d), a.value_std), "bf16")
        vh = wl.round_to(wl.normal(rng, (cap, hkv, d), a.value_std), "bf16")
        kcd[bb], vcd[bb] = kh.to(DEV), vh.to(DEV)
        if bb == b:  # the oracle's own copy of the checked (sequence, KV head) cache
            kb = kh[:, g:g + 1].clone()
            vb = vh[:, g:g + 1].clone()
    qn = wl.round_to(wl.normal(rng, (B, a.l_new, hq, d), a.value_std), "bf16")
    kn = wl.round_to(wl.normal(rng, (B, a.l_new, hkv, d), a.value_std), "bf16")
    vn = wl.round_to(wl.normal(rng, (B, a.l_new, hkv, d), a.value_std), "bf16")
    c_host = a.cache_len.copy()
    cl = torch.from_numpy(c_host.copy()).to(DEV)
    o, lse = ism.prefill_append(qn.to(DEV), kn.to(DEV), vn.to(DEV), kcd, vcd, cl, c_host, a.new_seg_end,
                                a.new_seg_type, a.softmax_scale)
    ism.check_status()
    o_ref, lse_ref = orc.prefill_append(qn[b:b + 1, :, hs], kn[b:b + 1, :, g:g + 1], vn[b:b + 1, :, g:g + 1],
                                        kb[None], vb[None], c_host[b:b + 1], a.new_seg_end, a.new_seg_type,
                                        a.softmax_scale)
    c = int(c_host[b])
    kb[c:c + a.l_new] = kn[b, :, g:g + 1]
    vb[c:c + a.l_new] = vn[b, :, g:g + 1]
    _cmp("prefill o", o[b:b + 1, :, hs], o_ref, "bf16")
    _cmp_lse("prefill lse", lse[hs][:, b:b + 1], np.transpose(lse_ref, (1, 0, 2)), "bf16")
    c_host = c_host + a.l_new
    check = {0, 1, 127, a.decode_steps - 1}
    for t in range(a.decode_steps):
        qd = wl.round_to(wl.normal(rng, (B, 1, hq, d), a.value_std), "bf16")
        kd = wl.round_to(wl.normal(rng, (B, 1, hkv, d), a.value_std), "bf16")
        vd = wl.round_to(wl.normal(rng, (B, 1, hkv, d), a.value_std), "bf16")
        o, lse = ism.prefill_append(qd.to(DEV), kd.to(DEV), vd.to(DEV), kcd, vcd, cl, c_host, [1], [1],
                                    a.softmax_scale)
        c = int(c_host[b])
        if t in check:
            o_ref, lse_ref = orc.prefill_append(qd[b:b + 1, :, hs], kd[b:b + 1, :, g:g + 1], vd[b:b + 1, :, g:g + 1],
                                                kb[None], vb[None], np.array([c]), [1], [1], a.softmax_scale)
            _cmp(f"decode o step {t}", o[b:b + 1, :, hs], o_ref, "bf16")
            _cmp_lse(f"decode lse step {t}", lse[hs][:, b:b + 1], np.transpose(lse_ref, (1, 0, 2)), "bf16")
        kb[c] = kd[b, 0, g:g + 1]
        vb[c] = vd[b, 0, g:g + 1]
        c_host = c_host + 1
    ism.check_status()
    assert cl.cpu().numpy().tolist() == c_host.tolist()


def test_in_order_tmem_reuse_matches_drained_bit_exact(ism, knobs):
    """The tensor-core kernels issue an MMA that overwrites tensor memory
    right after the MMA that reads it, relying on MMAs of one thread
    executing in issue order.  The drained variant (each such MMA waits for
    the reader to complete) computes the same arithmetic in the same order,
    so the two must agree bit for bit, run after run."""
    w = wl.gqa_8k()
    q, k, v, do = (t.to(DEV) for t in wl.attention_tensors(w))
    segs = ism.Segments.from_workload(w.segs, DEV)

    def run():
        o, lse = ism.fwd(segs, q, k, v, w.softmax_scale)
        dq, dk, dv = ism.bwd(segs, q, k, v, o, lse, do, w.softmax_scale)
        ism.check_status()
        return o, lse, dq, dk, dv

    knobs("ISM_DRAIN_TMEM_REUSE", "1")
    ref = run()
    knobs("ISM_DRAIN_TMEM_REUSE", "0")
    for _ in range(8):
        got = run()
        for name, a_, b_ in zip(("o", "lse", "dq", "dk", "dv"), got, ref):
            assert torch.equal(a_, b_), name


def test_bwd_schedules_agree(ism):
    """The stored-dS backward (dK/dV keeps every visible dS^T tile, dQ is a
    GEMM over them) and the recompute backward run the same dK/dV arithmetic,
    so dK and dV agree bit for bit; dQ is built from the same bf16-rounded
    dS in another fp32 summation order.  The stored schedule's extra
    workspace is 32 KiB per non-empty (q-tile, k-tile) pair and query head,
    the pair count being the number of non-empty tiles of the tile map."""
    w = wl.gqa_8k()
    q, k, v, do = (t.to(DEV) for t in wl.attention_tensors(w))
    segs = ism.Segments.from_workload(w.segs, DEV)
    o, lse = ism.fwd(segs, q, k, v, w.softmax_scale)
    full = ism.bwd_workspace_size(segs, q, k, w.softmax_scale)
    low = ism.bwd_workspace_size(segs, q, k, w.softmax_scale, minimal=True)
    if ism.has_tensor_cores():
        pairs = int(orc.tile_map_packed(w.segs, 128, 128)["kt_end"].sum())
        extra = pairs * w.num_heads_q * 128 * 128 * 2
        nk = int(sum((n + 127) // 128 for n in np.diff(w.segs.cu_seqlens)))
        assert extra <= full - low <= extra + 4 * nk + 1024
    stored = ism.bwd(segs, q, k, v, o, lse, do, w.softmax_scale)
    recomputed = ism.bwd(segs, q, k, v, o, lse, do, w.softmax_scale, minimal_workspace=True)
    ism.check_status()
    assert torch.equal(stored[1], recomputed[1]), "dk"
    assert torch.equal(stored[2], recomputed[2]), "dv"
    diff = (stored[0].float() - recomputed[0].float()).abs()
    scale = recomputed[0].float().abs().max().item()
    assert diff.max().item() <= 2e-2 * max(scale, 1.0), diff.max().item()
    assert diff.mean().item() <= 1e-3, diff.mean().item()



def test_dkdv_pair_matches_single_cta_bit_exact(ism, knobs):
    """dK/dV on CTA pairs (ISM_DKDV_PAIR=1: one M = 256 MMA over two
    neighbouring key tiles, B split across the pair) runs the arithmetic of
    the single-CTA kernel row by row in the same order; the odd CTA of a pair
    also visits the query tiles the even tile sees before its own, where its
    P and dS are exact zeros.  So dQ, dK and dV agree bit for bit, for both
    backward schedules, with sequences of an odd number of key tiles (the
    last pair has one tile) and query heads 3 per KV head."""
    if not ism.has_tensor_cores():
        pytest.skip("tensor-core backward only")
    cases = [wl.gqa_8k(),
             wl.Workload("pairs", wl.pack([([70, 150, 170, 300], [0, 1, 0, 1]), ([33, 90, 200, 517], [0, 1, 0, 1]),
                                           ([129], [0]), ([1, 256, 257], [1, 0, 1])]),
                         6, 2, 128, "bf16", 128 ** -0.5, 0.5, 77)]
    for w in cases:
        q, k, v, do = (t.to(DEV) for t in wl.attention_tensors(w))
        segs = ism.Segments.from_workload(w.segs, DEV)
        o, lse = ism.fwd(segs, q, k, v, w.softmax_scale)
        for minimal in (False, True):
            knobs("ISM_DKDV_PAIR", "0")
            single = ism.bwd(segs, q, k, v, o, lse, do, w.softmax_scale, minimal_workspace=minimal)
            knobs("ISM_DKDV_PAIR", "1")
            pair = ism.bwd(segs, q, k, v, o, lse, do, w.softmax_scale, minimal_workspace=minimal)
            ism.check_status()
            for name, a_, b_ in zip(("dq", "dk", "dv"), pair, single):
                assert torch.equal(a_, b_), (w.name, minimal, name)


def test_session_turn_by_turn_matches_one_pass(ism):
    """A dialogue served turn by turn (each query appended in one call, each
    answer token decoded alone against the growing cache) gives the rows of
    one ISM pass over the whole dialogue (Section 2.3: the KV cache of earlier
    turns is reused unchanged)."""
    s = wl.SessionWorkload("session_test", 2, 3, 24, 6, 8, 2, 128, 128 ** -0.5, 0.5, 41)
    B, T, hq, hkv, d = s.batch, s.capacity, s.num_heads_q, s.num_heads_kv, s.head_dim
    rng = np.random.Generator(np.random.PCG64(s.seed))
    q = wl.round_to(wl.normal(rng, (B, T, hq, d), s.value_std), "bf16")
    k = wl.round_to(wl.normal(rng, (B, T, hkv, d), s.value_std), "bf16")
    v = wl.round_to(wl.normal(rng, (B, T, hkv, d), s.value_std), "bf16")
    kc = torch.zeros((B, T, hkv, d), dtype=torch.bfloat16, device=DEV)
    vc = torch.zeros_like(kc)
    cl = torch.zeros((B,), dtype=torch.int32, device=DEV)
    c_host = np.zeros((B,), dtype=np.int32)
    o = torch.full((B, T, hq, d), float("nan"), dtype=torch.bfloat16, device=DEV)
    pos = 0
    for _ in range(s.turns):
        sl = slice(pos, pos + s.q_len)
        o[:, sl], _ = ism.prefill_append(q[:, sl].contiguous().to(DEV), k[:, sl].contiguous().to(DEV),
                                         v[:, sl].contiguous().to(DEV), kc, vc, cl, c_host, [s.q_len], [wl.QUERY],
                                         s.softmax_scale)
        pos += s.q_len
        c_host = c_host + s.q_len
        for _ in range(s.a_len):
            sl = slice(pos, pos + 1)
            o[:, sl], _ = ism.prefill_append(q[:, sl].contiguous().to(DEV), k[:, sl].contiguous().to(DEV),
                                             v[:, sl].contiguous().to(DEV), kc, vc, cl, c_host, [1], [wl.ANSWER],
                                             s.softmax_scale)
            pos += 1
            c_host = c_host + 1
    ism.check_status()
    assert cl.cpu().numpy().tolist() == [T] * B
    assert torch.equal(kc.cpu(), k) and torch.equal(vc.cpu(), v)
    segs = wl.pack([s.dialogue()])
    for b in range(B):
        o_ref, _ = orc.attn_fwd(q[b], k[b], v[b], segs, s.softmax_scale)
        _cmp(f"session dialogue {b}", o[b], o_ref, "bf16")


def _to_pages(kc, vc, page_size, rng, spare=3):
    """Scatter contiguous caches [B, cap, Hkv, D] into shuffled pages of one pool
    (plus a few unused pages): returns (k_pool, v_pool, block_table [B, max_pages])."""
    B, cap = kc.shape[:2]
    max_pages = (cap + page_size - 1) // page_size
    n_pages = B * max_pages + spare
    table = rng.permutation(n_pages)[:B * max_pages].reshape(B, max_pages).astype(np.int32)
    kp = torch.zeros((n_pages * page_size,) + tuple(kc.shape[2:]), dtype=kc.dtype)
    vp = torch.zeros_like(kp)
    for b in range(B):
        for i in range(max_pages):
            n = min(page_size, cap - i * page_size)
            r = int(table[b, i]) * page_size
            kp[r:r + n] = kc[b, i * page_size:i * page_size + n]
            vp[r:r + n] = vc[b, i * page_size:i * page_size + n]
    return kp, vp, table


@pytest.mark.parametrize("split", ["0", "1000"])
@pytest.mark.parametrize("l_new,segs,hq,hkv,d", [(200, ([40, 41, 120, 200], [0, 1, 0, 1]), 8, 2, 128),
                                                  (128, ([128], [0]), 8, 2, 128), (1, ([1], [1]), 8, 2, 128),
                                                  (1, ([1], [1]), 8, 1, 128), (37, ([37], [0]), 3, 3, 128),
                                                  (200, ([40, 41, 120, 200], [0, 1, 0, 1]), 8, 2, 64)])
def test_prefill_append_paged_matches_contiguous(ism, l_new, segs, hq, hkv, d, split, knobs):
    """The paged cache gives bit for bit the contiguous result (same kernels,
    rows through the block table) and the oracle's result on the gathered
    cache, with every prefill item split into key-range halves or none."""
    knobs("ISM_PREFILL_SPLIT", split)
    B, ps = 3, 128
    c_lens = np.array([0, 77, 300], dtype=np.int32)
    cap = int(c_lens.max()) + l_new
    kc, vc, qn, kn, vn = _append_inputs(B, cap, c_lens, l_new, hq, hkv, d, seed=100 + l_new + d)
    rng = np.random.Generator(np.random.PCG64(7 + l_new))
    kp, vp, table = _to_pages(kc, vc, ps, rng)
    scale = d ** -0.5
    kcd, vcd = kc.to(DEV), vc.to(DEV)
    cl = torch.from_numpy(c_lens.copy()).to(DEV)
    o_c, l_c = ism.prefill_append(qn.to(DEV), kn.to(DEV), vn.to(DEV), kcd, vcd, cl, c_lens, segs[0], segs[1], scale)
    kpd, vpd = kp.to(DEV), vp.to(DEV)
    clp = torch.from_numpy(c_lens.copy()).to(DEV)
    o_p, l_p = ism.prefill_append_paged(qn.to(DEV), kn.to(DEV), vn.to(DEV), kpd, vpd, ps,
                                        torch.from_numpy(table).to(DEV), table, clp, c_lens, segs[0], segs[1], scale)
    ism.check_status()
    assert torch.equal(o_p, o_c) and torch.equal(l_p, l_c)
    assert clp.cpu().numpy().tolist() == (c_lens + l_new).tolist()
    # the new keys / values sit in the sequences' pages
    kpc = kpd.cpu()
    for b in range(B):
        for j in range(l_new):
            p = int(c_lens[b]) + j
            r = int(table[b, p // ps]) * ps + p % ps
            assert torch.equal(kpc[r], kn[b, j])
    o_ref, lse_ref = orc.prefill_append_paged(qn, kn, vn, kp, vp, ps, table, c_lens, segs[0], segs[1], scale)
    _cmp("paged o_new", o_p, o_ref, "bf16")
    _cmp_lse("paged lse_new", l_p, np.transpose(lse_ref, (1, 0, 2)), "bf16")


def test_paged_append_rejects_bad_tables(ism):
    B, ps, hq, hkv, d = 2, 128, 8, 2, 128
    c_lens = np.array([100, 200], dtype=np.int32)
    kc, vc, qn, kn, vn = _append_inputs(B, 256, c_lens, 8, hq, hkv, d, seed=5)
    kp, vp, table = _to_pages(kc, vc, ps, np.random.Generator(np.random.PCG64(1)))
    cl = torch.from_numpy(c_lens.copy()).to(DEV)
    args = (qn.to(DEV), kn.to(DEV), vn.to(DEV), kp.to(DEV), vp.to(DEV))
    bad = table.copy()
    bad[1, 1] = kp.shape[0] // ps  # one past the pool
    with pytest.raises(ism.IsmError):
        ism.prefill_append_paged(*args, ps, torch.from_numpy(bad).to(DEV), bad, cl, c_lens, [8], [0], d ** -0.5)
    with pytest.raises(ism.IsmError):  # a page size that splits a 128-key tile
        ism.prefill_append_paged(*args, 64, torch.from_numpy(table).to(DEV), table, cl, c_lens, [8], [0], d ** -0.5)
    ism.check_status()
    assert cl.cpu().numpy().tolist() == c_lens.tolist()  # nothing ran


# ---------------------------------------------------------------- e4m3 forward

def _e4m3_pass(ism, w):
    """e4m3 copies of the workload's Q, K, V (per-tensor scales), the GPU
    forward on them, and their exact dequantised values for the oracle."""
    q, k, v, _ = wl.attention_tensors(w)
    (q8, qs), (k8, ks), (v8, vs) = (wl.quantize_e4m3(t) for t in (q, k, v))
    segs = ism.Segments.from_workload(w.segs, DEV)
    o, lse = ism.fwd_e4m3(segs, q8.to(DEV), k8.to(DEV), v8.to(DEV), qs, ks, vs, w.softmax_scale)
    ism.check_status()
    deq = [t.double() * s for t, s in ((q8, qs), (k8, ks), (v8, vs))]
    return deq, o, lse


def _cmp_e4m3(name, got, ref, vmax):
    """P is rounded to e4m3 for O = P V / l (relative error at most 2^-4 per
    term), O to bf16 (2^-9): |O - O_ref| <= (2^-4 + 2^-9) max|V| bounds every
    element; the errors are independent across keys, so their mean is far
    smaller (mean-abs 4e-3, twice the bf16 bound)."""
    got = _np(got)
    assert np.all(np.isfinite(got)), f"{name}: non-finite values"
    err = np.abs(got - ref)
    assert err.max() <= (2 ** -4 + 2 ** -9) * vmax, f"{name}: max abs err {err.max():.3e} (max|V| {vmax:.3f})"
    assert err.mean() <= 4e-3, f"{name}: mean abs err {err.mean():.3e}"


@pytest.mark.parametrize("hq,hkv", [(8, 2), (3, 3), (6, 2)])
def test_small_e4m3_fwd(ism, hq, hkv):
    """Paired heads (even group) and paired query tiles (odd group sizes)."""
    w = _small_bf16(128, hq=hq, hkv=hkv, seed=50 + hq)
    (q, k, v), o, lse = _e4m3_pass(ism, w)
    o_ref, lse_ref = orc.attn_fwd(q, k, v, w.segs, w.softmax_scale)
    _cmp_e4m3("o", o, o_ref, float(v.abs().max()))
    _cmp_lse("lse", lse, lse_ref, "bf16")


@pytest.mark.parametrize("make", [wl.gqa_8k, wl.mha_4k], ids=["gqa_8k", "mha_4k"])
def test_full_size_e4m3_fwd_sampled_group(ism, make):
    w = make()
    (q, k, v), o, lse = _e4m3_pass(ism, w)
    b = _largest_seq(w.segs)
    t0, L, se, st = w.segs.seq(b)
    grp = w.num_heads_q // w.num_heads_kv
    g = 1 if w.num_heads_kv > 1 else 0
    hs = slice(g * grp, (g + 1) * grp)
    sl = slice(t0, t0 + L)
    o_ref, lse_ref = orc.attn_fwd(q[sl][:, hs], k[sl][:, g:g + 1], v[sl][:, g:g + 1], wl.pack([(se, st)]),
                                  w.softmax_scale)
    _cmp_e4m3("o", o[sl][:, hs], o_ref, float(v.abs().max()))
    _cmp_lse("lse", lse[hs][:, sl], lse_ref, "bf16")


def test_e4m3_rejects_other_entry_points(ism):
    w = _small_bf16(128)
    q, k, v, _ = wl.attention_tensors(w)
    q8, k8, v8 = (wl.quantize_e4m3(t)[0].to(DEV) for t in (q, k, v))
    segs = ism.Segments.from_workload(w.segs, DEV)
    with pytest.raises(ism.IsmError):  # e4m3 only through ism_attn_fwd_e4m3
        ism.fwd(segs, q8, k8, v8, w.softmax_scale)
    with pytest.raises(ism.IsmError):  # descales must be positive
        ism.fwd_e4m3(segs, q8, k8, v8, 0.0, 1.0, 1.0, w.softmax_scale)
    ism.check_status()


@pytest.mark.parametrize("path", ["tensor_cores", "cuda_cores"])
@pytest.mark.parametrize("l_new,segs,hq,hkv", [(200, ([40, 41, 120, 200], [0, 1, 0, 1]), 8, 2),
                                                (200, ([40, 41, 120, 200], [0, 1, 0, 1]), 3, 3),
                                                (1, ([1], [1]), 8, 2), (1, ([1], [1]), 6, 2),
                                                (1, ([1], [1]), 16, 1), (1, ([1], [1]), 4, 4),
                                                (1, ([1], [1]), 10, 2), (1, ([1], [1]), 8, 1)])
def test_prefill_append_e4m3(ism, l_new, segs, hq, hkv, path, knobs):
    """e4m3 queries and caches (cache factors shared by the new keys / values)
    against the oracle on the dequantised values; single-token steps on the
    tensor-core decode or the CUDA-core one."""
    if path == "cuda_cores":
        if l_new != 1:
            pytest.skip("the decode path choice applies to single-token steps")
        knobs("ISM_DECODE_NO_TC", "1")
    B, d = 3, 128
    c_lens = np.array([0, 77, 300], dtype=np.int32)
    cap = 300 + l_new + 5
    kc, vc, qn, kn, vn = _append_inputs(B, cap, c_lens, l_new, hq, hkv, d, seed=60 + l_new + hq)
    _, ks = wl.quantize_e4m3(torch.cat([kc.reshape(-1), kn.reshape(-1)]))
    _, vs = wl.quantize_e4m3(torch.cat([vc.reshape(-1), vn.reshape(-1)]))
    q8, qs = wl.quantize_e4m3(qn)
    k8c, k8n = ((t.float() / ks).to(torch.float8_e4m3fn) for t in (kc, kn))
    v8c, v8n = ((t.float() / vs).to(torch.float8_e4m3fn) for t in (vc, vn))
    kcd, vcd = k8c.to(DEV), v8c.to(DEV)
    cl = torch.from_numpy(c_lens.copy()).to(DEV)
    o, lse = ism.prefill_append_e4m3(q8.to(DEV), k8n.to(DEV), v8n.to(DEV), kcd, vcd, cl, c_lens, segs[0], segs[1],
                                     qs, ks, vs, d ** -0.5)
    ism.check_status()
    assert cl.cpu().numpy().tolist() == (c_lens + l_new).tolist()
    for b in range(B):
        c = int(c_lens[b])
        assert torch.equal(kcd[b, c:c + l_new].cpu().view(torch.uint8), k8n[b].view(torch.uint8))
    deq = lambda t, s: t.double() * s  # noqa: E731
    o_ref, lse_ref = orc.prefill_append(deq(q8, qs), deq(k8n, ks), deq(v8n, vs), deq(k8c, ks), deq(v8c, vs), c_lens,
                                        segs[0], segs[1], d ** -0.5)
    vmax = max(float(deq(v8c, vs).abs().max()), float(deq(v8n, vs).abs().max()))
    _cmp_e4m3("o_new", o, o_ref, vmax)
    _cmp_lse("lse_new", lse, np.transpose(lse_ref, (1, 0, 2)), "bf16")


def test_append_step_matches_prefill_append(ism):
    """The prepared call (arguments marshalled once, host lengths advanced in
    place) gives the results of prefill_append step by step."""
    B, d, c0, steps, hq, hkv = 2, 128, 300, 4, 8, 2
    cap = c0 + steps
    kc, vc, qn, kn, vn = _append_inputs(B, cap, None, steps, hq, hkv, d, seed=77)
    outs = []
    for prepared in (False, True):
        kcd, vcd = kc.clone().to(DEV), vc.clone().to(DEV)
        c_host = np.array([c0, c0 - 50], dtype=np.int32)
        cl = torch.from_numpy(c_host.copy()).to(DEV)
        qb, kb, vb = (torch.empty((B, 1) + tuple(t.shape[2:]), dtype=t.dtype, device=DEV) for t in (qn, kn, vn))
        step = ism.AppendStep(qb, kb, vb, kcd, vcd, cl, c_host, [1], [1], d ** -0.5) if prepared else None
        got = []
        for t in range(steps):
            qb.copy_(qn[:, t:t + 1]); kb.copy_(kn[:, t:t + 1]); vb.copy_(vn[:, t:t + 1])
            if prepared:
                o, _ = step()
            else:
                o, _ = ism.prefill_append(qb, kb, vb, kcd, vcd, cl, c_host, [1], [1], d ** -0.5)
            got.append(o.clone())
            c_host += 1
        ism.check_status()
        outs.append(torch.stack(got))
    assert torch.equal(outs[0], outs[1])


# ---------------------------------------------------------------- rotary encoding on append

def _bf16_round(x):
    return torch.from_numpy(np.ascontiguousarray(x)).to(torch.bfloat16).to(torch.float64).numpy()


def _rope_tables(rows, d, kind, seed):
    if kind == "schedule":
        c, s = wl.rope_tables(rows, d)
    else:  # any angles: the kernel reads the tables, it assumes no schedule
        rng = np.random.Generator(np.random.PCG64(seed))
        ang = rng.uniform(-np.pi, np.pi, size=(rows, d // 2))
        c, s = np.cos(ang).astype(np.float32), np.sin(ang).astype(np.float32)
    return torch.from_numpy(c), torch.from_numpy(s)


def _check_rotated_keys(name, got, ref):
    # the kernel rotates in fp32 and rounds once to bf16; the oracle rotates in
    # fp64, so the two differ by at most half a bf16 ulp of the result (2^-8
    # relative) plus the fp32 rotation error
    got = _np(got)
    err = np.abs(got - ref)
    bound = 2.0 ** -8 * np.abs(ref) + 2e-6
    assert np.all(err <= bound), f"{name}: worst excess {np.max(err - bound):.3e}"


@pytest.mark.parametrize("l_new,segs,hq,hkv,d,kind", [
    (200, ([40, 41, 120, 200], [0, 1, 0, 1]), 8, 2, 128, "schedule"),
    (200, ([40, 41, 120, 200], [0, 1, 0, 1]), 8, 2, 128, "random"),
    (37, ([37], [0]), 6, 2, 128, "random"),
    (150, ([50, 150], [0, 1]), 4, 2, 64, "random"),
    (1, ([1], [1]), 8, 2, 128, "schedule"),
    (1, ([1], [1]), 32, 8, 64, "random")])
def test_prefill_append_rope(ism, l_new, segs, hq, hkv, d, kind):
    B = 3
    c_lens = np.array([0, 77, 300], dtype=np.int32)
    cap = 300 + l_new + 5
    kc, vc, qn, kn, vn = _append_inputs(B, cap, c_lens, l_new, hq, hkv, d, seed=l_new + 100)
    cos_t, sin_t = _rope_tables(300 + l_new, d, kind, seed=l_new + d)   # exactly the positions written
    kcd, vcd = kc.to(DEV), vc.to(DEV)
    cl = torch.from_numpy(c_lens.copy()).to(DEV)
    scale = d ** -0.5
    o, lse = ism.prefill_append_rope(qn.to(DEV), kn.to(DEV), vn.to(DEV), kcd, vcd, cl, c_lens, segs[0], segs[1],
                                     cos_t.to(DEV), sin_t.to(DEV), scale)
    ism.check_status()
    assert cl.cpu().numpy().tolist() == (c_lens + l_new).tolist()
    o_ref, lse_ref, k_rot = orc.prefill_append_rope(qn, kn, vn, kc, vc, c_lens, segs[0], segs[1], cos_t.numpy(),
                                                    sin_t.numpy(), scale, key_round=_bf16_round)
    for b in range(B):
        c = int(c_lens[b])
        _check_rotated_keys(f"cached keys of sequence {b}", kcd[b, c:c + l_new], k_rot[b])
        assert torch.equal(vcd[b, c:c + l_new].cpu(), vn[b])
        assert torch.equal(kcd[b, :c].cpu(), kc[b, :c]) and torch.equal(kcd[b, c + l_new:].cpu(), kc[b, c + l_new:])
    _cmp("o_new", o, o_ref, "bf16")
    _cmp_lse("lse_new", lse, np.transpose(lse_ref, (1, 0, 2)), "bf16")


def test_rope_turns_equal_one_pass_over_rotated_dialogue(ism):
    # a prefill of the first turn and then single-token decode steps, all with
    # rotary encoding, give the rows the one-pass forward computes on the
    # dialogue whose queries and keys the oracle rotated at their positions
    hq, hkv, d = 8, 2, 128
    t1 = ([70, 300], [0, 1])
    steps = 5
    L = t1[0][-1] + steps
    full = wl.pack([(t1[0] + [L], t1[1] + [1])])
    w = wl.Workload("rope", full, hq, hkv, d, "bf16", d ** -0.5, 0.5, 29)
    q, k, v, _ = wl.attention_tensors(w)
    cos_t, sin_t = _rope_tables(L, d, "schedule", 0)
    pos = np.arange(L)
    qr = torch.from_numpy(_bf16_round(orc.rope_rotate(q, pos, cos_t.numpy(), sin_t.numpy()))).to(torch.bfloat16)
    kr = torch.from_numpy(_bf16_round(orc.rope_rotate(k, pos, cos_t.numpy(), sin_t.numpy()))).to(torch.bfloat16)
    o_full, _ = ism.fwd(ism.Segments.from_workload(full, DEV), qr.to(DEV), kr.to(DEV), v.to(DEV), w.softmax_scale)
    kcd = torch.zeros((1, L, hkv, d), dtype=torch.bfloat16, device=DEV)
    vcd = torch.zeros_like(kcd)
    c_host = np.zeros(1, dtype=np.int32)
    cl = torch.zeros(1, dtype=torch.int32, device=DEV)
    cd, sd = cos_t.to(DEV), sin_t.to(DEV)
    chunks = [(0, t1[0][-1], t1)] + [(t1[0][-1] + i, 1, ([1], [1])) for i in range(steps)]
    for s0, n, sg in chunks:
        o, _ = ism.prefill_append_rope(q[None, s0:s0 + n].contiguous().to(DEV), k[None, s0:s0 + n].contiguous().to(DEV),
                                       v[None, s0:s0 + n].contiguous().to(DEV), kcd, vcd, cl, c_host, sg[0], sg[1],
                                       cd, sd, w.softmax_scale)
        diff = (o[0].float() - o_full[s0:s0 + n].float()).abs().max().item()
        assert diff <= 2e-2, (s0, diff)
        c_host = c_host + n
    ism.check_status()
    assert (kcd[0].float() - kr.to(DEV).float()).abs().max().item() <= 2.0 ** -6   # at most one bf16 ulp at |x| < 4


def test_append_16k_rope_prefill_sampled(ism):
    """The 8 x 16K cache with a 512-token query appended under rotary
    encoding: every stored key against the oracle's rotation, and the
    attention rows of one (sequence, KV group)."""
    a = wl.append_16k()
    B, cap, hq, hkv, d = a.batch, a.capacity, a.num_heads_q, a.num_heads_kv, a.head_dim
    rng = np.random.Generator(np.random.PCG64(a.seed + 50))
    kcd = torch.empty((B, cap, hkv, d), dtype=torch.bfloat16, device=DEV)
    vcd = torch.empty_like(kcd)
    b, g = 6, 5
    hs = list(range(g * hq // hkv, (g + 1) * hq // hkv))
    for bb in range(B):
        kh = wl.round_to(wl.normal(rng, (cap, hkv, d), a.value_std), "bf16")
        vh = wl.round_to(wl.normal(rng, (cap, hkv, d), a.value_std), "bf16")
        kcd[bb], vcd[bb] = kh.to(DEV), vh.to(DEV)
        if bb == b:
            kb = kh[:, g:g + 1].clone()
            vb = vh[:, g:g + 1].clone()
    qn = wl.round_to(wl.normal(rng, (B, a.l_new, hq, d), a.value_std), "bf16")
    kn = wl.round_to(wl.normal(rng, (B, a.l_new, hkv, d), a.value_std), "bf16")
    vn = wl.round_to(wl.normal(rng, (B, a.l_new, hkv, d), a.value_std), "bf16")
    cos_t, sin_t = _rope_tables(cap, d, "schedule", 0)
    c_host = a.cache_len.copy()
    cl = torch.from_numpy(c_host.copy()).to(DEV)
    o, lse = ism.prefill_append_rope(qn.to(DEV), kn.to(DEV), vn.to(DEV), kcd, vcd, cl, c_host, a.new_seg_end,
                                     a.new_seg_type, cos_t.to(DEV), sin_t.to(DEV), a.softmax_scale)
    ism.check_status()
    c = int(c_host[0])
    pos = c + np.arange(a.l_new)
    for bb in range(B):
        _check_rotated_keys(f"stored keys of sequence {bb}", kcd[bb, c:c + a.l_new],
                            orc.rope_rotate(kn[bb], pos, cos_t.numpy(), sin_t.numpy()))
    o_ref, lse_ref, _ = orc.prefill_append_rope(qn[b:b + 1, :, hs], kn[b:b + 1, :, g:g + 1], vn[b:b + 1, :, g:g + 1],
                                                kb[None], vb[None], c_host[b:b + 1], a.new_seg_end, a.new_seg_type,
                                                cos_t.numpy(), sin_t.numpy(), a.softmax_scale, key_round=_bf16_round)
    _cmp("prefill o", o[b:b + 1, :, hs], o_ref, "bf16")
    _cmp_lse("prefill lse", lse[hs][:, b:b + 1], np.transpose(lse_ref, (1, 0, 2)), "bf16")


# ---------------------------------------------------------------- garbage past the cached keys

def _poison_past(cache, c_lens, extra_cols=0):
    # NaN and Inf bit patterns in every row at or past cache_len[b] (unwritten
    # cache memory may hold anything)
    bad = torch.tensor([float("nan"), float("inf"), float("-inf")], dtype=cache.dtype)
    for b in range(cache.shape[0]):
        c = int(c_lens[b])
        n = cache.shape[1] - c
        if n > 0:
            idx = torch.arange(n * int(np.prod(cache.shape[2:]))) % 3
            cache[b, c:] = bad[idx].reshape((n,) + tuple(cache.shape[2:]))
    return cache


@pytest.mark.parametrize("l_new,segs,hq,hkv,d,cap_extra", [
    (200, ([40, 41, 120, 200], [0, 1, 0, 1]), 8, 2, 128, 5),     # capacity not a multiple of 128
    (64, ([64], [0]), 4, 4, 128, 100),
    (1, ([1], [1]), 8, 2, 128, 3),
    (1, ([1], [1]), 4, 4, 128, 60),                                # one query head per KV head
    (1, ([1], [1]), 40, 2, 128, 7),                                # forward kernels for the step
    (150, ([50, 150], [0, 1]), 4, 2, 64, 9)])
def test_append_ignores_garbage_past_cache_len(ism, l_new, segs, hq, hkv, d, cap_extra):
    B = 3
    c_lens = np.array([0, 77, 300], dtype=np.int32)
    cap = 300 + l_new + cap_extra
    kc, vc, qn, kn, vn = _append_inputs(B, cap, c_lens, l_new, hq, hkv, d, seed=l_new + 7)
    kc, vc = _poison_past(kc.clone(), c_lens), _poison_past(vc.clone(), c_lens)
    kcd, vcd = kc.to(DEV), vc.to(DEV)
    cl = torch.from_numpy(c_lens.copy()).to(DEV)
    scale = d ** -0.5
    o, lse = ism.prefill_append(qn.to(DEV), kn.to(DEV), vn.to(DEV), kcd, vcd, cl, c_lens, segs[0], segs[1], scale)
    ism.check_status()
    o_ref, lse_ref = orc.prefill_append(qn, kn, vn, kc, vc, c_lens, segs[0], segs[1], scale)
    _cmp("o_new", o, o_ref, "bf16")
    _cmp_lse("lse_new", lse, np.transpose(lse_ref, (1, 0, 2)), "bf16")
    # the documented side effect: value rows up to the next 128-key boundary
    # are zeroed, every other row past the new end is left as it was
    for b in range(B):
        e = int(c_lens[b]) + l_new
        stop = min((e + 127) // 128 * 128, cap)
        assert bool((vcd[b, e:stop] == 0).all())
        assert torch.equal(vcd[b, stop:].cpu().view(torch.int16), vc[b, stop:].view(torch.int16))
        assert torch.equal(kcd[b, e:].cpu().view(torch.int16), kc[b, e:].view(torch.int16))


def test_paged_and_e4m3_appends_ignore_garbage(ism):
    B, hq, hkv, d, l_new, ps = 2, 8, 2, 128, 90, 256
    c_lens = np.array([30, 300], dtype=np.int32)
    cap = 512
    kc, vc, qn, kn, vn = _append_inputs(B, cap, c_lens, l_new, hq, hkv, d, seed=77)
    segs = ([20, 90], [0, 1])
    scale = d ** -0.5
    o_ref, _ = orc.prefill_append(qn, kn, vn, kc, vc, c_lens, segs[0], segs[1], scale)
    # paged: pages of the two sequences interleaved in one pool, garbage past each length
    kcp, vcp = _poison_past(kc.clone(), c_lens), _poison_past(vc.clone(), c_lens)
    table = np.array([[3, 0], [1, 2]], dtype=np.int32)
    kp = torch.empty((4 * ps, hkv, d), dtype=torch.bfloat16)
    vp = torch.empty_like(kp)
    for b in range(B):
        for pg in range(2):
            kp[table[b, pg] * ps:(table[b, pg] + 1) * ps] = kcp[b, pg * ps:(pg + 1) * ps]
            vp[table[b, pg] * ps:(table[b, pg] + 1) * ps] = vcp[b, pg * ps:(pg + 1) * ps]
    cl = torch.from_numpy(c_lens.copy()).to(DEV)
    o, _ = ism.prefill_append_paged(qn.to(DEV), kn.to(DEV), vn.to(DEV), kp.to(DEV), vp.to(DEV), ps,
                                    torch.from_numpy(table).to(DEV), table, cl, c_lens, segs[0], segs[1], scale)
    ism.check_status()
    _cmp("paged o_new", o, o_ref, "bf16")
    # e4m3 caches: the e4m3 NaN pattern (0x7f) past each length
    k8, kd_ = wl.quantize_e4m3(torch.cat([kc, kn], 1))
    v8, vd_ = wl.quantize_e4m3(torch.cat([vc, vn], 1))
    q8, qd_ = wl.quantize_e4m3(qn)
    kc8, kn8 = k8[:, :cap].contiguous(), k8[:, cap:].contiguous()
    vc8, vn8 = v8[:, :cap].contiguous(), v8[:, cap:].contiguous()
    for b in range(B):
        kc8.view(torch.uint8)[b, c_lens[b]:] = 0x7F
        vc8.view(torch.uint8)[b, c_lens[b]:] = 0x7F
    deq = lambda t, s: t.float() * s
    o8_ref, _ = orc.prefill_append(deq(q8, qd_), deq(kn8, kd_), deq(vn8, vd_), deq(kc8, kd_), deq(vc8, vd_), c_lens,
                                   segs[0], segs[1], scale)
    cl = torch.from_numpy(c_lens.copy()).to(DEV)
    o8, _ = ism.prefill_append_e4m3(q8.to(DEV), kn8.to(DEV), vn8.to(DEV), kc8.to(DEV), vc8.to(DEV), cl, c_lens,
                                    segs[0], segs[1], qd_, kd_, vd_, scale)
    ism.check_status()
    _cmp_e4m3("e4m3 o_new", o8, o8_ref, float(torch.cat([vc, vn], 1).float().abs().max()))


# ---------------------------------------------------------------- limits

@pytest.mark.parametrize("n_seqs", [2500, 8192])
def test_max_sequences_fwd_bwd_sampled(ism, n_seqs):
    """8192 sequences (the most one call takes; and 2500, whose per-sequence
    offsets fill 40 KB of the metadata pass's shared memory) of 1-40 tokens
    with random segments (empty and same-type neighbours included) in one
    fwd + bwd call; the oracle checks every 517th sequence and the last."""
    rng = np.random.Generator(np.random.PCG64(81))
    segs = wl.random_dialogue_set(rng, n_seqs, 40)
    w = wl.Workload("many_short", segs, 4, 2, 128, "bf16", 128 ** -0.5, 0.5, 82)
    (q, k, v, do), (o, lse, dq, dk, dv) = _run_pass(ism, w)
    for b in list(range(0, n_seqs, 517)) + [n_seqs - 1]:
        t0, L, se, st = segs.seq(b)
        sub = wl.pack([(se, st)])
        sl = slice(t0, t0 + L)
        o_ref, lse_ref = orc.attn_fwd(q[sl], k[sl], v[sl], sub, w.softmax_scale)
        dq_ref, dk_ref, dv_ref = orc.attn_bwd(q[sl], k[sl], v[sl], do[sl], sub, w.softmax_scale)
        _cmp(f"o of sequence {b}", o[sl], o_ref, "bf16")
        _cmp_lse(f"lse of sequence {b}", lse[:, sl], lse_ref, "bf16")
        _cmp(f"dq of sequence {b}", dq[sl], dq_ref, "bf16")
        _cmp(f"dk of sequence {b}", dk[sl], dk_ref, "bf16")
        _cmp(f"dv of sequence {b}", dv[sl], dv_ref, "bf16")


def test_append_max_segments(ism):
    """A chunk of 256 segments (the most one append takes): alternating query
    and answer runs of 0-3 tokens."""
    rng = np.random.Generator(np.random.PCG64(83))
    lens = rng.integers(0, 4, size=256)
    lens[-1] = max(int(lens[-1]), 1)
    ends = np.cumsum(lens).astype(np.int32)
    types = np.array([i % 2 for i in range(256)], dtype=np.uint8)
    l_new = int(ends[-1])
    B, hq, hkv, d = 2, 8, 2, 128
    c_lens = np.array([0, 333], dtype=np.int32)
    cap = 333 + l_new + 4
    kc, vc, qn, kn, vn = _append_inputs(B, cap, c_lens, l_new, hq, hkv, d, seed=84)
    cl = torch.from_numpy(c_lens.copy()).to(DEV)
    o, lse = ism.prefill_append(qn.to(DEV), kn.to(DEV), vn.to(DEV), kc.to(DEV), vc.to(DEV), cl, c_lens, ends, types,
                                d ** -0.5)
    ism.check_status()
    o_ref, lse_ref = orc.prefill_append(qn, kn, vn, kc, vc, c_lens, ends, types, d ** -0.5)
    _cmp("o_new", o, o_ref, "bf16")
    _cmp_lse("lse_new", lse, np.transpose(lse_ref, (1, 0, 2)), "bf16")


@pytest.mark.parametrize("keys", [150000, 200000])
def test_decode_long_cache(ism, keys):
    """Single-token steps over one cache of 150 000 keys (the tensor-core
    decode with close to its 64 splits of at most 3072 keys) and of 200 000
    (past 64 x 3072 keys: the CUDA-core decode takes it); the oracle checks
    one KV head's group."""
    B, hq, hkv, d, steps = 1, 8, 2, 128, 2
    cap = keys + steps
    kc, vc, qn, kn, vn = _append_inputs(B, cap, None, steps, hq, hkv, d, seed=85)
    kcd, vcd = kc.clone().to(DEV), vc.clone().to(DEV)
    c_host = np.array([keys], dtype=np.int32)
    cl = torch.from_numpy(c_host.copy()).to(DEV)
    g, grp = 1, hq // hkv
    hs = list(range(g * grp, (g + 1) * grp))
    for t in range(steps):
        o, lse = ism.prefill_append(qn[:, t:t + 1].contiguous().to(DEV), kn[:, t:t + 1].contiguous().to(DEV),
                                    vn[:, t:t + 1].contiguous().to(DEV), kcd, vcd, cl, c_host, [1], [1], d ** -0.5)
        kref = kc[:, :, g:g + 1].clone()
        vref = vc[:, :, g:g + 1].clone()
        kref[0, keys:keys + t] = kn[0, :t, g:g + 1]
        vref[0, keys:keys + t] = vn[0, :t, g:g + 1]
        o_ref, lse_ref = orc.prefill_append(qn[:, t:t + 1, hs], kn[:, t:t + 1, g:g + 1], vn[:, t:t + 1, g:g + 1],
                                            kref, vref, c_host, [1], [1], d ** -0.5)
        _cmp(f"decode o step {t}", o[:, :, hs], o_ref, "bf16")
        _cmp_lse(f"decode lse step {t}", lse[hs], np.transpose(lse_ref, (1, 0, 2)), "bf16")
        c_host = c_host + 1
    ism.check_status()


# ---------------------------------------------------------------- key-range split of the prefill

@pytest.mark.parametrize("dtype", ["bf16", "e4m3"])
@pytest.mark.parametrize("n_split", ["0", "2", "1000"])
def test_prefill_key_split(ism, dtype, n_split, knobs):
    """Prefill items that run as two halves of their key range (the last ones,
    or all of them with 1000: some halves then have no key tile at all) give
    the oracle's result; ISM_PREFILL_SPLIT forces the count."""
    knobs("ISM_PREFILL_SPLIT", n_split)
    B, d, hq, hkv, l_new = 3, 128, 8, 2, 200
    segs = ([40, 41, 120, 200], [0, 1, 0, 1])
    c_lens = np.array([0, 77, 300], dtype=np.int32)
    cap = 300 + l_new + 5
    kc, vc, qn, kn, vn = _append_inputs(B, cap, c_lens, l_new, hq, hkv, d, seed=91)
    cl = torch.from_numpy(c_lens.copy()).to(DEV)
    scale = d ** -0.5
    if dtype == "bf16":
        o, lse = ism.prefill_append(qn.to(DEV), kn.to(DEV), vn.to(DEV), kc.to(DEV), vc.to(DEV), cl, c_lens, segs[0],
                                    segs[1], scale)
        ism.check_status()
        o_ref, lse_ref = orc.prefill_append(qn, kn, vn, kc, vc, c_lens, segs[0], segs[1], scale)
        _cmp("o_new", o, o_ref, "bf16")
    else:
        _, ks = wl.quantize_e4m3(torch.cat([kc.reshape(-1), kn.reshape(-1)]))
        _, vs = wl.quantize_e4m3(torch.cat([vc.reshape(-1), vn.reshape(-1)]))
        q8, qs = wl.quantize_e4m3(qn)
        k8c, k8n = ((t.float() / ks).to(torch.float8_e4m3fn) for t in (kc, kn))
        v8c, v8n = ((t.float() / vs).to(torch.float8_e4m3fn) for t in (vc, vn))
        o, lse = ism.prefill_append_e4m3(q8.to(DEV), k8n.to(DEV), v8n.to(DEV), k8c.to(DEV), v8c.to(DEV), cl, c_lens,
                                         segs[0], segs[1], qs, ks, vs, scale)
        ism.check_status()
        deq = lambda t, s: t.double() * s  # noqa: E731
        o_ref, lse_ref = orc.prefill_append(deq(q8, qs), deq(k8n, ks), deq(v8n, vs), deq(k8c, ks), deq(v8c, vs),
                                            c_lens, segs[0], segs[1], scale)
        vmax = max(float(deq(v8c, vs).abs().max()), float(deq(v8n, vs).abs().max()))
        _cmp_e4m3("o_new", o, o_ref, vmax)
    _cmp_lse("lse_new", lse, np.transpose(lse_ref, (1, 0, 2)), "bf16")


# ---------------------------------------------------------------- maximum size: one long dialogue

def test_long_context_128k_minimum_workspace(ism):
    """One 131072-token dialogue of a few hundred turns (8 query / 2 KV
    heads, head_dim 128, bf16) through the forward and the minimum-workspace
    backward (the stored-dS workspace would need about 137 GB here; long
    contexts run the recompute schedule).  The oracle checks O, LSE and dQ of
    every head on sampled rows, and dK / dV of two whole key tiles near the
    end of the dialogue (the last one and the one 640 keys before the end)
    for both KV heads, from the full softmax rows of every query that sees
    those keys."""
    L = 131072
    rng = np.random.Generator(np.random.PCG64(128))
    segs_np = wl.pack([wl.draw_dialogue(rng, L, 300, 400)])
    w = wl.Workload("long_128k", segs_np, 8, 2, 128, "bf16", 128 ** -0.5, 0.5, 128)
    (q, k, v, do), (o, lse, dq, dk, dv) = _run_pass(ism, w, minimal_workspace=True)
    for name, t in zip(("o", "lse", "dq", "dk", "dv"), (o, lse, dq, dk, dv)):
        assert bool(torch.isfinite(t).all()), f"{name}: non-finite values"
    # O, LSE, dQ: every head, 32 segment boundaries and 16 random rows
    ends = segs_np.seg_end
    bounds = np.unique(np.concatenate([ends[ends < L], np.maximum(ends - 1, 0)]))
    rows = np.unique(np.concatenate([rng.choice(bounds, size=32, replace=False), rng.integers(0, L, size=16),
                                     [0, L - 1]])).astype(np.int64)
    o_ref, lse_ref = orc.attn_fwd(q, k, v, segs_np, w.softmax_scale, rows=rows)
    dq_ref = orc.attn_bwd_dq_rows(q, k, v, do, segs_np, w.softmax_scale, rows)
    _cmp(f"o, all heads, {rows.size} rows", o[rows], o_ref[rows], "bf16")
    _cmp_lse(f"lse, all heads, {rows.size} rows", lse[:, rows], lse_ref[:, rows], "bf16")
    _cmp(f"dq, all heads, {rows.size} rows", dq[rows], dq_ref[rows], "bf16")
    # dK, dV: two key tiles near the end, both KV heads
    keys = np.concatenate([np.arange(L - 640, L - 512), np.arange(L - 128, L)])
    dk_ref, dv_ref = orc.attn_bwd_dkdv_keys(q, k, v, do, segs_np, w.softmax_scale, keys)
    _cmp(f"dk, {keys.size} keys", dk[keys], dk_ref[keys], "bf16")
    _cmp(f"dv, {keys.size} keys", dv[keys], dv_ref[keys], "bf16")
