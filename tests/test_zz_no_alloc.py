"""The forward entry point that allocates nothing (for callers that cannot
allocate device memory where they run attention, e.g. during CUDA graph
capture or under a fixed start-up memory reservation).  It must give the
same results as the regular forward, call after call, while reusing one
fixed scratch array."""
import ctypes as C

import numpy as np
import pytest
import torch

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


def _noalloc_fwd(ism, segs, q, k, v, scale):
    lib = ism.load()
    s, sh = segs.struct(), ism._shape(q, k, scale)
    o = torch.empty_like(q)
    lse = torch.empty((q.shape[1], q.shape[0]), dtype=torch.float32, device=q.device)
    code = lib.ism_attn_fwd_noalloc(C.byref(s), C.byref(sh), ism._ptr(q), ism._ptr(k), ism._ptr(v), ism._ptr(o),
                                    ism._ptr(lse), ism._stream(q.device))
    assert code == 0, lib.ism_last_error().decode()
    return o, lse


def _case(segs_np, hq, hkv, seed):
    w = wl.Workload("noalloc", segs_np, hq, hkv, 128, "bf16", 128 ** -0.5, 0.5, seed)
    return w, [t.to(DEV) for t in wl.attention_tensors(w, with_dout=False)]


def test_noalloc_forward_matches_regular_forward_twice(ism):
    cases = [_case(wl.pack([([70, 150, 170, 300], [0, 1, 0, 1]), ([33, 90, 200, 517], [0, 1, 0, 1])]), 8, 2, 41),
             _case(wl.pack([([129], [0]), ([0, 64, 64, 128, 256], [1, 0, 1, 0, 1]), ([1], [1])]), 4, 4, 42)]
    for w, (q, k, v) in cases:  # two calls in a row on the shared scratch
        segs = ism.Segments.from_workload(w.segs, DEV)
        o_ref, lse_ref = ism.fwd(segs, q, k, v, w.softmax_scale)
        o, lse = _noalloc_fwd(ism, segs, q, k, v, w.softmax_scale)
        torch.cuda.synchronize()
        err = (o.float() - o_ref.float()).abs()
        assert err.max().item() <= 2e-2 and err.mean().item() <= 2e-3
        assert (lse - lse_ref).abs().max().item() <= 1e-3
    ism.check_status()


def test_noalloc_rejects_batches_beyond_its_scratch(ism):
    lib = ism.load()
    cap = lib.ism_attn_fwd_noalloc_max_workspace()
    assert cap == 4 << 20
    T = 2_000_000  # kv_end alone needs 8 MB
    segs = ism.Segments.from_numpy([0, T], [0, 1], [T], [0], DEV)
    sh = ism._Shape()
    sh.num_heads_q, sh.num_heads_kv, sh.head_dim, sh.dtype, sh.softmax_scale = 1, 1, 128, 0, 0.1
    fake = C.c_void_p(1 << 20)
    code = lib.ism_attn_fwd_noalloc(C.byref(segs.struct()), C.byref(sh), fake, fake, fake, fake, fake, None)
    assert code == 5
    assert "no-alloc scratch" in lib.ism_last_error().decode()
