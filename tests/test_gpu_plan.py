"""Plans (ism_attn_plan_build): the metadata of a batch built once and shared
by the forward and backward of several layers.  The planned calls run the
same kernels on the same metadata as the one-pass calls, so their results
are compared bit for bit; the one-pass calls themselves are checked against
the oracle elsewhere, and the first case here is checked against it too."""
import numpy as np
import pytest
import torch

from oracle import ism_oracle as orc
from paper_2408_00539_gb300 import workloads as wl

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


@pytest.fixture(scope="module")
def ism():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2408_00539_gb300 import ism as m
    m.load(build_if_missing=True)
    return m


def _segs():
    return wl.pack([([70, 150, 170, 300], [0, 1, 0, 1]), ([33, 90, 200, 517], [0, 1, 0, 1]), ([129], [0]),
                    ([1], [1]), ([0, 64, 64, 128, 256], [1, 0, 1, 0, 1])])


def _plan(ism, segs, w, q):
    return ism.Plan(segs, w.num_heads_q, w.num_heads_kv, w.head_dim, q.dtype, DEV)


def _both(ism, segs, w, tensors, plan, minimal):
    q, k, v, do = tensors
    o, lse = ism.fwd(segs, q, k, v, w.softmax_scale)
    ref = (o, lse) + ism.bwd(segs, q, k, v, o, lse, do, w.softmax_scale, minimal_workspace=minimal)
    o2, lse2 = ism.fwd(segs, q, k, v, w.softmax_scale, plan=plan)
    got = (o2, lse2) + ism.bwd(segs, q, k, v, o2, lse2, do, w.softmax_scale, minimal_workspace=minimal, plan=plan)
    ism.check_status()
    return ref, got


@pytest.mark.parametrize("hq,hkv,dtype", [(8, 2, "bf16"), (4, 4, "bf16"), (6, 2, "bf16"), (4, 2, "fp32")])
@pytest.mark.parametrize("minimal", [False, True])
def test_planned_calls_equal_one_pass_calls(ism, hq, hkv, dtype, minimal):
    """Head pairs (8/2), query-tile pairs (4/4 and 6/2: one and three query
    heads per KV head) and the CUDA-core path (fp32), both backward
    schedules: O, LSE, dQ, dK, dV identical to the one-pass calls."""
    w = wl.Workload("plan", _segs(), hq, hkv, 128, dtype, 128 ** -0.5, 0.5, 61 + hq)
    host = wl.attention_tensors(w)
    tensors = tuple(t.to(DEV) for t in host)
    segs = ism.Segments.from_workload(w.segs, DEV)
    plan = _plan(ism, segs, w, tensors[0])
    ref, got = _both(ism, segs, w, tensors, plan, minimal)
    for name, a, b in zip(("o", "lse", "dq", "dk", "dv"), ref, got):
        assert torch.equal(a, b), name
    if (hq, hkv, dtype, minimal) == (8, 2, "bf16", False):
        o_ref, _ = orc.attn_fwd(*host[:3], w.segs, w.softmax_scale)
        err = np.abs(got[0].double().cpu().numpy() - o_ref)
        assert err.max() <= 2e-2 and err.mean() <= 2e-3, (err.max(), err.mean())


def test_plan_shared_by_layers(ism):
    """One plan, three layers of different inputs (and softmax scales), each
    forward and backward in turn: every result equals the one-pass calls'."""
    w = wl.Workload("plan_layers", _segs(), 8, 2, 128, "bf16", 128 ** -0.5, 0.5, 71)
    segs = ism.Segments.from_workload(w.segs, DEV)
    plan = None
    for layer in range(3):
        tensors = tuple(t.to(DEV) for t in wl.attention_tensors(w, seed_offset=layer))
        if plan is None:
            plan = _plan(ism, segs, w, tensors[0])
        wl_scaled = wl.Workload(w.name, w.segs, w.num_heads_q, w.num_heads_kv, w.head_dim, w.dtype,
                                w.softmax_scale * (1.0 + 0.25 * layer), w.value_std, w.seed)
        ref, got = _both(ism, segs, wl_scaled, tensors, plan, False)
        for name, a, b in zip(("o", "lse", "dq", "dk", "dv"), ref, got):
            assert torch.equal(a, b), f"layer {layer} {name}"


def test_plan_for_other_segments_or_heads_rejected(ism):
    """A plan is refused, before any launch, by calls over other segments or
    other head counts."""
    w = wl.Workload("plan_a", _segs(), 8, 2, 128, "bf16", 128 ** -0.5, 0.5, 81)
    q, k, v, do = (t.to(DEV) for t in wl.attention_tensors(w))
    segs = ism.Segments.from_workload(w.segs, DEV)
    plan = _plan(ism, segs, w, q)
    o, lse = ism.fwd(segs, q, k, v, w.softmax_scale, plan=plan)
    # same token count, one segment boundary moved
    other = ism.Segments.from_workload(wl.pack([([70, 151, 170, 300], [0, 1, 0, 1]), ([33, 90, 200, 517], [0, 1, 0, 1]),
                                                ([129], [0]), ([1], [1]), ([0, 64, 64, 128, 256], [1, 0, 1, 0, 1])]),
                                       DEV)
    launches = ism.kernel_launches()
    with pytest.raises(ism.IsmError) as e:
        ism.fwd(other, q, k, v, w.softmax_scale, plan=plan)
    assert e.value.code == 1
    with pytest.raises(ism.IsmError) as e:
        ism.bwd(other, q, k, v, o, lse, do, w.softmax_scale, plan=plan)
    assert e.value.code == 1
    # other head counts (4 KV heads), same segments
    k4, v4 = k.repeat(1, 2, 1).contiguous(), v.repeat(1, 2, 1).contiguous()
    with pytest.raises(ism.IsmError) as e:
        ism.fwd(segs, q, k4, v4, w.softmax_scale, plan=plan)
    assert e.value.code == 1
    assert ism.kernel_launches() == launches
    ism.check_status()


@pytest.mark.parametrize("hq,hkv", [(8, 2), (4, 4)])
def test_planned_rope_calls_equal_one_pass_calls(ism, hq, hkv):
    """The rotary forward and backward on a plan: rotated rows, O, LSE, dQ,
    dK, dV identical to the one-pass rotary calls."""
    w = wl.Workload("plan_rope", _segs(), hq, hkv, 128, "bf16", 128 ** -0.5, 0.5, 91 + hq)
    q, k, v, do = (t.to(DEV) for t in wl.attention_tensors(w))
    segs = ism.Segments.from_workload(w.segs, DEV)
    cos_np, sin_np = wl.rope_tables(int(np.diff(w.segs.cu_seqlens).max()), 128)
    cos_t, sin_t = torch.from_numpy(cos_np).to(DEV), torch.from_numpy(sin_np).to(DEV)
    plan = _plan(ism, segs, w, q)
    o, lse, qr, kr = ism.fwd_rope(segs, q, k, v, cos_t, sin_t, w.softmax_scale)
    ref = (o, lse, qr, kr) + ism.bwd_rope(segs, qr, kr, v, o, lse, do, cos_t, sin_t, w.softmax_scale)
    o2, lse2, qr2, kr2 = ism.fwd_rope(segs, q, k, v, cos_t, sin_t, w.softmax_scale, plan=plan)
    got = (o2, lse2, qr2, kr2) + ism.bwd_rope(segs, qr2, kr2, v, o2, lse2, do, cos_t, sin_t, w.softmax_scale,
                                              plan=plan)
    ism.check_status()
    for name, a, b in zip(("o", "lse", "q_rot", "k_rot", "dq", "dk", "dv"), ref, got):
        assert torch.equal(a, b), name
