"""The forward entry point that allocates nothing.  It serves callers that
cannot allocate device memory where they run attention: servers that reserve
all device memory once at start-up and may not grow it, and hosts that drive
the GPU through the plain C interface without a device allocator of their
own.  It must give exactly the regular forward's results, call after call,
while every call reuses one fixed scratch array (collected last, so that a
failure here comes after every other test has run)."""
import ctypes as C

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
    return w, wl.attention_tensors(w, with_dout=False)


def test_noalloc_forward_matches_regular_forward_twice(ism):
    """Two different batches, each run twice in a row through the no-alloc
    entry point: bit for bit the regular forward's O and LSE (same kernels,
    same inputs, only the scratch differs), and within the bf16 tolerances of
    the fp64 oracle."""
    cases = [_case(wl.pack([([70, 150, 170, 300], [0, 1, 0, 1]), ([33, 90, 200, 517], [0, 1, 0, 1])]), 8, 2, 41),
             _case(wl.pack([([129], [0]), ([0, 64, 64, 128, 256], [1, 0, 1, 0, 1]), ([1], [1])]), 4, 4, 42)]
    for w, (q, k, v) in cases:
        o_ref, lse_ref = orc.attn_fwd(q, k, v, w.segs, w.softmax_scale)
        qd, kd, vd = q.to(DEV), k.to(DEV), v.to(DEV)
        segs = ism.Segments.from_workload(w.segs, DEV)
        o_reg, lse_reg = ism.fwd(segs, qd, kd, vd, w.softmax_scale)
        for _ in range(2):  # the second call finds the first call's leftovers in the scratch
            o, lse = _noalloc_fwd(ism, segs, qd, kd, vd, w.softmax_scale)
            ism.check_status()
            assert torch.equal(o, o_reg) and torch.equal(lse, lse_reg)
            err = np.abs(o.double().cpu().numpy() - o_ref)
            assert err.max() <= 2e-2 and err.mean() <= 2e-3, (err.max(), err.mean())
            assert np.abs(lse.double().cpu().numpy() - lse_ref).max() <= 1e-3


def test_noalloc_rejects_batches_beyond_its_scratch(ism):
    """A batch whose scratch exceeds the fixed array is refused on the host.
    The tensors are passed as NULL, so even if the size check were lost the
    call would stop at the argument check: nothing can be launched here."""
    lib = ism.load()
    cap = lib.ism_attn_fwd_noalloc_max_workspace()
    assert cap == 4 << 20
    T = 2_000_000  # kv_end alone needs 8 MB
    segs = ism.Segments.from_numpy([0, T], [0, 1], [T], [0], DEV)
    sh = ism._Shape()
    sh.num_heads_q, sh.num_heads_kv, sh.head_dim, sh.dtype, sh.softmax_scale = 1, 1, 128, 0, 0.1
    launches = lib.ism_kernel_launches()
    code = lib.ism_attn_fwd_noalloc(C.byref(segs.struct()), C.byref(sh), None, None, None, None, None, None)
    assert code == 5
    assert "no-alloc scratch" in lib.ism_last_error().decode()
    assert lib.ism_kernel_launches() == launches
