"""GPU parity of the one-pass forward and backward with rotary encoding
(ism_attn_fwd_rope / ism_attn_bwd_rope) against the fp64 oracle's
attn_fwd_rope / attn_bwd_rope on the same seeded inputs.

The kernels rotate in fp32 and round the rotated queries and keys once to the
input type before the attention; the oracle rotates in fp64 and computes on
its own rotated values rounded to the same type.  Tolerances are those of the
plain one-pass path: bf16 max-abs 2e-2, mean-abs 2e-3 (LSE 1e-3); fp32
max-abs 1e-4 (LSE 1e-5)."""
import numpy as np
import pytest
import torch

from oracle import ism_oracle as orc
from paper_2408_00539_gb300 import workloads as wl

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
BF16_MAX, BF16_MEAN, FP32_MAX = 2e-2, 2e-3, 1e-4


@pytest.fixture(scope="module")
def ism():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2408_00539_gb300 import ism as m
    m.load(build_if_missing=True)
    return m


def _np(t):
    return t.detach().to(torch.float64).cpu().numpy()


def _cmp(name, got, ref, dtype):
    got = _np(got)
    assert got.shape == ref.shape, (name, got.shape, ref.shape)
    assert np.all(np.isfinite(got)), f"{name}: non-finite values"
    err = np.abs(got - ref)
    if dtype == "fp32":
        assert err.max() <= FP32_MAX, f"{name}: max abs err {err.max():.3e}"
    else:
        assert err.max() <= BF16_MAX, f"{name}: max abs err {err.max():.3e}"
        assert err.mean() <= BF16_MEAN, f"{name}: mean abs err {err.mean():.3e}"


def _cmp_lse(name, got, ref, dtype):
    err = np.abs(_np(got) - ref)
    assert err.max() <= (1e-5 if dtype == "fp32" else 1e-3), f"{name}: max abs err {err.max():.3e}"


def _round_fn(dtype):
    tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
    return lambda x: torch.from_numpy(np.ascontiguousarray(x)).to(tdt).to(torch.float64).numpy()


def _tables(rows, d, kind, seed):
    if kind == "schedule":
        c, s = wl.rope_tables(rows, d)
    else:  # any angles: the kernels read the tables and assume no schedule
        rng = np.random.Generator(np.random.PCG64(seed))
        ang = rng.uniform(-np.pi, np.pi, size=(rows, d // 2))
        c, s = np.cos(ang).astype(np.float32), np.sin(ang).astype(np.float32)
    return torch.from_numpy(c), torch.from_numpy(s)


def _check_rotated(name, got, ref, dtype):
    # fp32 rotation rounded once against the fp64 rotation: at most half an ulp
    # of the result's type (2^-8 relative for bf16, 2^-24 for fp32) plus the
    # fp32 rotation error
    got = _np(got)
    rel = 2.0 ** -8 if dtype == "bf16" else 2.0 ** -23
    bound = rel * np.abs(ref) + 4e-6
    err = np.abs(got - ref)
    assert np.all(err <= bound), f"{name}: worst excess {np.max(err - bound):.3e}"


def _small_segs():
    return wl.pack([([70, 150, 170, 300], [0, 1, 0, 1]),      # ragged
                    ([33, 90, 200, 517], [0, 1, 0, 1]),        # several tiles + tail
                    ([1], [1]),                                # single token
                    ([0, 64, 64, 128, 256], [1, 0, 1, 0, 1]),  # tile-aligned, zero-length segment
                    ([50, 51, 52, 383], [0, 0, 1, 0])])        # adjacent queries


def _run(ism, w, cos_t, sin_t, minimal_workspace=False, in_place=False):
    q, k, v, do = wl.attention_tensors(w)
    segs = ism.Segments.from_workload(w.segs, DEV)
    qd, kd, vd, dod = (t.to(DEV) for t in (q, k, v, do))
    cd, sd = cos_t.to(DEV), sin_t.to(DEV)
    if in_place:
        o, lse, qr, kr = ism.fwd_rope(segs, qd, kd, vd, cd, sd, w.softmax_scale, q_rot=qd, k_rot=kd)
        assert qr.data_ptr() == qd.data_ptr() and kr.data_ptr() == kd.data_ptr()
    else:
        o, lse, qr, kr = ism.fwd_rope(segs, qd, kd, vd, cd, sd, w.softmax_scale)
    dq, dk, dv = ism.bwd_rope(segs, qr, kr, vd, o, lse, dod, cd, sd, w.softmax_scale,
                              minimal_workspace=minimal_workspace)
    ism.check_status()
    return (q, k, v, do), (o, lse, qr, kr, dq, dk, dv)


def _check_all(w, cos_t, sin_t, inputs, outputs):
    q, k, v, do = inputs
    o, lse, qr, kr, dq, dk, dv = outputs
    c, s = cos_t.numpy(), sin_t.numpy()
    rnd = _round_fn(w.dtype)
    o_ref, lse_ref, qr_ref, kr_ref = orc.attn_fwd_rope(q, k, v, w.segs, w.softmax_scale, c, s, round_fn=rnd)
    dq_ref, dk_ref, dv_ref = orc.attn_bwd_rope(q, k, v, do, w.segs, w.softmax_scale, c, s, round_fn=rnd)
    _check_rotated("q_rot", qr, qr_ref, w.dtype)
    _check_rotated("k_rot", kr, kr_ref, w.dtype)
    _cmp("o", o, o_ref, w.dtype)
    _cmp_lse("lse", lse, lse_ref, w.dtype)
    _cmp("dq", dq, dq_ref, w.dtype)
    _cmp("dk", dk, dk_ref, w.dtype)
    _cmp("dv", dv, dv_ref, w.dtype)


@pytest.mark.parametrize("d,kind,schedule", [(128, "schedule", "stored_ds"), (128, "random", "stored_ds"),
                                             (128, "random", "recompute_dq"), (64, "random", "default"),
                                             (64, "schedule", "default")])
def test_rope_fwd_bwd_small_bf16(ism, d, kind, schedule):
    """head_dim 128 runs the tensor-core kernels (the inverse rotation inside
    the dQ and dK epilogues, for both backward schedules); head_dim 64 the
    CUDA-core kernels and a separate inverse-rotation pass."""
    segs = _small_segs()
    w = wl.Workload(f"rope_d{d}", segs, 8, 2, d, "bf16", d ** -0.5, 0.5, 61 + d)
    cos_t, sin_t = _tables(600, d, kind, seed=d)
    inputs, outputs = _run(ism, w, cos_t, sin_t, minimal_workspace=schedule == "recompute_dq")
    _check_all(w, cos_t, sin_t, inputs, outputs)


@pytest.mark.parametrize("hq,hkv", [(4, 4), (6, 2)])
def test_rope_fwd_bwd_group_sizes(ism, hq, hkv):
    """One and three query heads per KV head (the forward pairs query tiles
    of one head instead of two heads)."""
    w = wl.Workload("rope_grp", _small_segs(), hq, hkv, 128, "bf16", 128 ** -0.5, 0.5, 70 + hq)
    cos_t, sin_t = _tables(520, 128, "random", seed=hq)
    inputs, outputs = _run(ism, w, cos_t, sin_t)
    _check_all(w, cos_t, sin_t, inputs, outputs)


def test_rope_fwd_bwd_tiny_fp32(ism):
    w = wl.tiny_fp32()
    cos_t, sin_t = _tables(256, 64, "random", seed=5)
    inputs, outputs = _run(ism, w, cos_t, sin_t)
    _check_all(w, cos_t, sin_t, inputs, outputs)


def test_rope_in_place_equals_separate_outputs(ism):
    """q_rot / k_rot may be q / k themselves: the same results bit for bit."""
    w = wl.Workload("rope_inplace", _small_segs(), 8, 2, 128, "bf16", 128 ** -0.5, 0.5, 81)
    cos_t, sin_t = _tables(600, 128, "schedule", 0)
    _, a = _run(ism, w, cos_t, sin_t)
    _, b = _run(ism, w, cos_t, sin_t, in_place=True)
    for name, x, y in zip(("o", "lse", "q_rot", "k_rot", "dq", "dk", "dv"), a, b):
        assert torch.equal(x, y), name


def test_rope_zero_angles_equal_plain_pass(ism):
    """cos = 1, sin = 0 leaves every row as it is: the results equal the plain
    forward and backward bit for bit (same kernels, same inputs)."""
    w = wl.Workload("rope_zero", _small_segs(), 8, 2, 128, "bf16", 128 ** -0.5, 0.5, 82)
    ones, zeros = torch.ones((600, 64)), torch.zeros((600, 64))
    (q, k, v, do), (o, lse, qr, kr, dq, dk, dv) = _run(ism, w, ones, zeros)
    segs = ism.Segments.from_workload(w.segs, DEV)
    qd, kd, vd, dod = (t.to(DEV) for t in (q, k, v, do))
    o0, lse0 = ism.fwd(segs, qd, kd, vd, w.softmax_scale)
    dq0, dk0, dv0 = ism.bwd(segs, qd, kd, vd, o0, lse0, dod, w.softmax_scale)
    ism.check_status()
    assert torch.equal(qr, qd) and torch.equal(kr, kd)
    for name, x, y in zip(("o", "lse", "dq", "dk", "dv"), (o, lse, dq, dk, dv), (o0, lse0, dq0, dk0, dv0)):
        assert torch.equal(x, y), name


def test_rope_full_size_gqa_8k_sampled_group(ism):
    """The 2 x 8192 GQA workload with the usual rotary schedule, all heads
    launched; the oracle recomputes the last KV head's group of sequence 1
    (positions 0..8191 of that sequence)."""
    w = wl.gqa_8k()
    cos_t, sin_t = _tables(8192, 128, "schedule", 0)
    (q, k, v, do), (o, lse, qr, kr, dq, dk, dv) = _run(ism, w, cos_t, sin_t)
    for name, t in zip(("o", "lse", "dq", "dk", "dv"), (o, lse, dq, dk, dv)):
        assert bool(torch.isfinite(t).all()), name
    b, g = 1, w.num_heads_kv - 1
    t0, L, se, st = w.segs.seq(b)
    grp = w.num_heads_q // w.num_heads_kv
    hs, sl = slice(g * grp, (g + 1) * grp), slice(t0, t0 + L)
    sub = wl.Workload("sub", wl.pack([(se, st)]), grp, 1, 128, "bf16", w.softmax_scale, 0.5, 0)
    ins = (q[sl][:, hs].contiguous(), k[sl][:, g:g + 1].contiguous(), v[sl][:, g:g + 1].contiguous(),
           do[sl][:, hs].contiguous())
    outs = (o[sl][:, hs], lse[hs][:, sl], qr[sl][:, hs], kr[sl][:, g:g + 1], dq[sl][:, hs], dk[sl][:, g:g + 1],
            dv[sl][:, g:g + 1])
    _check_all(sub, cos_t, sin_t, ins, outs)


def test_rope_tables_too_short_rejected(ism):
    w = wl.Workload("rope_short", _small_segs(), 8, 2, 128, "bf16", 128 ** -0.5, 0.5, 83)
    q, k, v, _ = (t.to(DEV) for t in wl.attention_tensors(w))
    segs = ism.Segments.from_workload(w.segs, DEV)
    cos_t, sin_t = _tables(516, 128, "schedule", 0)  # the longest sequence has 517 tokens
    launches = ism.kernel_launches()
    with pytest.raises(ism.IsmError, match="cover 516 positions"):
        ism.fwd_rope(segs, q, k, v, cos_t.to(DEV), sin_t.to(DEV), w.softmax_scale)
    assert ism.kernel_launches() == launches


# ---------------------------------------------------------------- rotary append on paged and e4m3 caches

def _append_inputs(B, cap, l_new, hq, hkv, d, seed, std=0.5):
    rng = np.random.Generator(np.random.PCG64(seed))
    kc = wl.round_to(wl.normal(rng, (B, cap, hkv, d), std), "bf16")
    vc = wl.round_to(wl.normal(rng, (B, cap, hkv, d), std), "bf16")
    qn = wl.round_to(wl.normal(rng, (B, l_new, hq, d), std), "bf16")
    kn = wl.round_to(wl.normal(rng, (B, l_new, hkv, d), std), "bf16")
    vn = wl.round_to(wl.normal(rng, (B, l_new, hkv, d), std), "bf16")
    return kc, vc, qn, kn, vn


def _to_pages(kc, vc, page_size, rng, spare=3):
    """Contiguous caches [B, cap, Hkv, D] scattered into shuffled pages of one
    pool: (k_pool, v_pool, block_table [B, max_pages])."""
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


@pytest.mark.parametrize("l_new,segs,hq,hkv,d", [(200, ([40, 41, 120, 200], [0, 1, 0, 1]), 8, 2, 128),
                                                  (1, ([1], [1]), 8, 2, 128), (37, ([37], [0]), 3, 3, 128),
                                                  (150, ([50, 150], [0, 1]), 4, 2, 64)])
def test_paged_rope_append_matches_contiguous(ism, l_new, segs, hq, hkv, d):
    """The rotary append against a paged cache gives bit for bit the
    contiguous rotary append's outputs and stored rows (same kernels, rows
    through the block table)."""
    B, ps = 3, 128
    c_lens = np.array([0, 77, 300], dtype=np.int32)
    cap = int(c_lens.max()) + l_new
    kc, vc, qn, kn, vn = _append_inputs(B, cap, l_new, hq, hkv, d, seed=300 + l_new + d)
    cos_t, sin_t = _tables(cap, d, "random", seed=l_new)
    cd, sd = cos_t.to(DEV), sin_t.to(DEV)
    kcd, vcd = kc.to(DEV), vc.to(DEV)
    cl = torch.from_numpy(c_lens.copy()).to(DEV)
    scale = d ** -0.5
    o_c, lse_c = ism.prefill_append_rope(qn.to(DEV), kn.to(DEV), vn.to(DEV), kcd, vcd, cl, c_lens, segs[0], segs[1],
                                         cd, sd, scale)
    kp, vp, table = _to_pages(kc, vc, ps, np.random.Generator(np.random.PCG64(9 + l_new)))
    kpd, vpd = kp.to(DEV), vp.to(DEV)
    cl2 = torch.from_numpy(c_lens.copy()).to(DEV)
    o_p, lse_p = ism.prefill_append_paged_rope(qn.to(DEV), kn.to(DEV), vn.to(DEV), kpd, vpd, ps,
                                               torch.from_numpy(table).to(DEV), table, cl2, c_lens, segs[0], segs[1],
                                               cd, sd, scale)
    ism.check_status()
    assert torch.equal(o_p, o_c) and torch.equal(lse_p, lse_c)
    assert torch.equal(cl2, cl)
    kc_after, vc_after = kcd.cpu(), vcd.cpu()
    kp_after, vp_after = kpd.cpu(), vpd.cpu()
    for b in range(B):
        for p in range(int(c_lens[b]) + l_new):
            r = int(table[b, p // ps]) * ps + p % ps
            assert torch.equal(kp_after[r], kc_after[b, p]) and torch.equal(vp_after[r], vc_after[b, p]), (b, p)


def _q8(x, s):
    """Round x / s to e4m3 (round to nearest even).  A torch tensor (bf16 or
    fp32 values) is divided in fp32, as the kernels do; fp64 numpy values
    (the oracle's rotations) in fp64."""
    if torch.is_tensor(x):
        return (x.float() / s).to(torch.float8_e4m3fn)
    return torch.from_numpy(np.asarray(x, dtype=np.float64) / s).to(torch.float32).to(torch.float8_e4m3fn)


@pytest.mark.parametrize("l_new,segs,hq,hkv", [(200, ([40, 41, 120, 200], [0, 1, 0, 1]), 8, 2),
                                                (1, ([1], [1]), 8, 2), (37, ([37], [0]), 6, 2)])
def test_e4m3_rope_append(ism, l_new, segs, hq, hkv):
    """bf16 unrotated queries and keys rotated and quantised into e4m3 caches:
    the stored keys and values are the oracle's rotated values quantised with
    the caller's factors (the fp32 rotation may move a value across an e4m3
    rounding boundary: such elements differ by one step), and the outputs
    match the oracle's append on the dequantised values within the e4m3
    forward's derived bound."""
    B, d = 3, 128
    c_lens = np.array([0, 77, 300], dtype=np.int32)
    cap = 300 + l_new + 5
    kc, vc, qn, kn, vn = _append_inputs(B, cap, l_new, hq, hkv, d, seed=400 + l_new)
    cos_t, sin_t = _tables(cap, d, "schedule", 0)
    c_np, s_np = cos_t.numpy(), sin_t.numpy()
    # factors with room for the growth a rotation can cause (at most sqrt 2)
    # (fp32 numbers: the library takes the factors as fp32)
    ks = float(np.float32(max(float(kc.abs().max()), 1.5 * float(kn.abs().max())) / 448.0))
    vs = float(np.float32(max(float(vc.abs().max()), float(vn.abs().max())) / 448.0))
    qs = float(np.float32(1.5 * float(qn.abs().max()) / 448.0))
    k8c, v8c = _q8(kc, ks), _q8(vc, vs)
    k8d, v8d = k8c.to(DEV), v8c.to(DEV)
    cl = torch.from_numpy(c_lens.copy()).to(DEV)
    scale = d ** -0.5
    o, lse = ism.prefill_append_e4m3_rope(qn.to(DEV), kn.to(DEV), vn.to(DEV), k8d, v8d, cl, c_lens, segs[0], segs[1],
                                          qs, ks, vs, cos_t.to(DEV), sin_t.to(DEV), scale)
    ism.check_status()
    assert cl.cpu().numpy().tolist() == (c_lens + l_new).tolist()
    q8n = torch.empty((B, l_new, hq, d), dtype=torch.float8_e4m3fn)
    k8n = torch.empty((B, l_new, hkv, d), dtype=torch.float8_e4m3fn)
    k_after, v_after = k8d.cpu(), v8d.cpu()
    for b in range(B):
        c = int(c_lens[b])
        pos = c + np.arange(l_new)
        q8n[b] = _q8(orc.rope_rotate(qn[b], pos, c_np, s_np), qs)
        k8n[b] = _q8(orc.rope_rotate(kn[b], pos, c_np, s_np), ks)
        got, ref = k_after[b, c:c + l_new].float(), k8n[b].float()
        step = 2.0 ** (torch.floor(torch.log2(ref.abs().clamp_min(2.0 ** -6))) - 3)  # one e4m3 step at |ref|
        assert bool(((got - ref).abs() <= step).all()), f"stored keys of sequence {b}"
        assert float((got != ref).float().mean()) < 1e-3, f"stored keys of sequence {b}: too many rounding moves"
        assert torch.equal(v_after[b, c:c + l_new], _q8(vn[b], vs)), f"stored values of sequence {b}"
        assert torch.equal(k_after[b, :c], k8c[b, :c])
    deq = lambda t, s: t.double() * s  # noqa: E731
    # the oracle attends with its own quantised keys for the new rows
    o_ref, lse_ref = orc.prefill_append(deq(q8n, qs), deq(k8n, ks), deq(_q8(vn, vs), vs), deq(k8c, ks), deq(v8c, vs),
                                        c_lens, segs[0], segs[1], scale)
    vmax = max(float(deq(v8c, vs).abs().max()), float(deq(_q8(vn, vs), vs).abs().max()))
    got = _np(o)
    assert np.all(np.isfinite(got))
    err = np.abs(got - o_ref)
    assert err.max() <= (2 ** -4 + 2 ** -9) * vmax, f"o_new: max abs err {err.max():.3e} (max|V| {vmax:.3f})"
    assert err.mean() <= 4e-3, f"o_new: mean abs err {err.mean():.3e}"
    _cmp_lse("lse_new", lse, np.transpose(lse_ref, (1, 0, 2)), "bf16")


def test_rope_zero_length_sequences_and_empty_batch(ism):
    """Zero-length sequences share their offset with the next sequence: the
    rotation pass must still find each token's own sequence (positions
    restart after every boundary).  An empty batch launches nothing."""
    segs = wl.pack([([0], [0]), ([40, 100], [0, 1]), ([0], [1]), ([0], [0]), ([1], [1]), ([130, 131], [0, 1])])
    w = wl.Workload("rope_zero_len", segs, 4, 2, 128, "bf16", 128 ** -0.5, 0.5, 84)
    cos_t, sin_t = _tables(131, 128, "random", seed=7)
    inputs, outputs = _run(ism, w, cos_t, sin_t)
    _check_all(w, cos_t, sin_t, inputs, outputs)
    empty = ism.Segments.from_numpy([0, 0], [0, 0], [], [], DEV)
    q = torch.zeros((0, 4, 128), dtype=torch.bfloat16, device=DEV)
    k = torch.zeros((0, 2, 128), dtype=torch.bfloat16, device=DEV)
    launches = ism.kernel_launches()
    o, lse, qr, kr = ism.fwd_rope(empty, q, k, k, cos_t.to(DEV), sin_t.to(DEV), 0.1)
    assert o.shape == (0, 4, 128) and ism.kernel_launches() == launches
    ism.check_status()
