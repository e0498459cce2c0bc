"""Host-side checks of the C ABI (no GPU needed): the library loads, exports
every entry point declared in include/ism.h, and rejects malformed arguments
on the host before anything is launched."""
import ctypes as C
import os
import re

import numpy as np
import pytest

from paper_2408_00539_gb300 import ism

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    with open(os.path.join(ROOT, "include", "ism.h")) as fh:
        src = fh.read()
    return sorted(set(re.findall(r"^\s*(?:const\s+)?[\w]+\*?\s+\*?(ism_\w+)\s*\(", src, flags=re.M)))


@pytest.fixture(scope="module")
def lib():
    return ism.load(build_if_missing=True)


def test_header_declares_boundary():
    names = _declared()
    for n in ("ism_build_tile_map", "ism_attn_fwd", "ism_attn_bwd", "ism_attn_prefill_append",
              "ism_check_status", "ism_status_string"):
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    for n in _declared():
        assert hasattr(lib, n), n
        assert n in ism.EXPORTS, f"binding misses {n}"


def test_status_strings(lib):
    assert lib.ism_status_string(0) == b"ISM_OK"
    assert lib.ism_status_string(4) == b"ISM_ERR_TIMEOUT"


FAKE = 1 << 20  # a non-NULL, 256-aligned stand-in for device pointers (never dereferenced on these paths)


def _gpu_visible() -> bool:
    try:
        import torch
        return torch.cuda.is_available()
    except Exception:  # noqa: BLE001 - no torch, no GPU
        return False


# The argument checks below hand made-up device addresses to the library and
# rely on host validation rejecting the call first.  They run only where no
# GPU is visible, so that a regression in a check can never launch a kernel
# on those addresses; the GPU tests cover the same entry points with real
# buffers.
host_only = pytest.mark.skipif(_gpu_visible(), reason="made-up device pointers: only where no GPU is visible")


class _Keep:
    pass


def _segs(cu_seqlens, cu_segs, seg_end, seg_type, keep):
    h = [np.asarray(cu_seqlens, np.int32), np.asarray(cu_segs, np.int32), np.asarray(seg_end, np.int32),
         np.asarray(seg_type, np.uint8)]
    keep.h = h
    s = ism._Segments()
    s.num_seqs = len(cu_seqlens) - 1
    s.num_segs = len(seg_end)
    s.cu_seqlens = s.cu_segs = s.seg_end = s.seg_type = FAKE
    s.cu_seqlens_host, s.cu_segs_host = h[0].ctypes.data, h[1].ctypes.data
    s.seg_end_host, s.seg_type_host = h[2].ctypes.data, h[3].ctypes.data
    return s


def _shape(hq=4, hkv=2, d=128, dtype=0, scale=0.1):
    sh = ism._Shape()
    sh.num_heads_q, sh.num_heads_kv, sh.head_dim, sh.dtype, sh.softmax_scale = hq, hkv, d, dtype, scale
    return sh


def _fwd(lib, s, sh, ptr=FAKE, ws=FAKE, ws_bytes=1 << 30):
    return lib.ism_attn_fwd(C.byref(s), C.byref(sh), ptr, ptr, ptr, ptr, ptr, ws, ws_bytes, None)


@pytest.mark.parametrize("segs,msg", [
    (([0, 10], [0, 2], [4, 9], [0, 1]), "segments end at 9"),            # does not cover the sequence
    (([0, 10], [0, 2], [6, 4], [0, 1]), "non-decreasing"),                # decreasing ends
    (([0, 10], [0, 2], [4, 10], [0, 3]), "QUERY/ANSWER"),                 # bad type
    (([0, 10, 5], [0, 1, 2], [10, 0], [0, 0]), "decreases"),              # cu_seqlens decreasing
    (([1, 10], [0, 1], [9], [0]), "must be 0"),                           # cu_seqlens[0] != 0
    (([0, 10], [0, 1], [10, 10], [0, 0]), "num_segs"),                    # cu_segs[B] != num_segs
])
@host_only
def test_malformed_segments_rejected(lib, segs, msg):
    keep = _Keep()
    cs, cg, se, st = segs
    s = _segs(cs, cg, se, st, keep)
    if msg == "num_segs":
        s.num_segs = 2
    r = _fwd(lib, s, _shape())
    assert r == 1, (r, lib.ism_last_error())
    assert msg in lib.ism_last_error().decode()


@host_only
def test_too_many_sequences(lib):
    keep = _Keep()
    n = 8193                                                       # one past the most one call takes
    s = _segs(list(range(n + 1)), list(range(n + 1)), [1] * n, [0] * n, keep)
    nt, nq, nk = C.c_int64(), C.c_int64(), C.c_int64()
    assert lib.ism_tile_map_size(C.byref(s), 128, 128, C.byref(nt), C.byref(nq), C.byref(nk)) == 2
    assert "num_seqs 8193" in lib.ism_last_error().decode()


@host_only
def test_shape_errors(lib):
    keep = _Keep()
    s = _segs([0, 10], [0, 2], [4, 10], [0, 1], keep)
    assert _fwd(lib, s, _shape(hq=6, hkv=4)) == 1                 # Hq % Hkv != 0
    assert _fwd(lib, s, _shape(d=96)) == 2                        # unsupported head_dim
    assert _fwd(lib, s, _shape(dtype=7)) == 2                     # unsupported dtype
    assert _fwd(lib, s, _shape(scale=0.0)) == 1
    assert _fwd(lib, s, _shape(), ptr=FAKE + 8) == 1              # misaligned tensors
    assert _fwd(lib, s, _shape(), ptr=0) == 1                     # null tensors


@host_only
def test_workspace_errors(lib):
    keep = _Keep()
    s = _segs([0, 300], [0, 2], [100, 300], [0, 1], keep)
    sh = _shape()
    need = C.c_size_t()
    assert lib.ism_attn_fwd_workspace_size(C.byref(s), C.byref(sh), C.byref(need)) == 0
    assert need.value > 300 * 4
    assert _fwd(lib, s, sh, ws_bytes=need.value - 1) == 5
    assert _fwd(lib, s, sh, ws=FAKE + 16) == 5
    bneed = C.c_size_t()
    assert lib.ism_attn_bwd_workspace_size(C.byref(s), C.byref(sh), C.byref(bneed)) == 0
    assert bneed.value >= need.value + 4 * 300 * 4      # delta for 4 heads


@host_only
def test_tile_map_size(lib):
    keep = _Keep()
    s = _segs([0, 300, 300, 557], [0, 2, 2, 3], [100, 300, 257], [0, 1, 0], keep)
    nt, nq, nk = C.c_int64(), C.c_int64(), C.c_int64()
    assert lib.ism_tile_map_size(C.byref(s), 128, 64, C.byref(nt), C.byref(nq), C.byref(nk)) == 0
    assert (nq.value, nk.value, nt.value) == (3 + 0 + 3, 5 + 0 + 5, 3 * 5 + 3 * 5)
    assert lib.ism_tile_map_size(C.byref(s), 100, 64, C.byref(nt), C.byref(nq), C.byref(nk)) == 2


@host_only
def test_append_errors(lib):
    sh = _shape()
    se = np.array([4, 8], np.int32)
    st = np.array([0, 1], np.uint8)
    ch = np.array([10, 20], np.int32)

    def call(l_new=8, cap=28, seg_end=se, seg_type=st, nseg=2, cache_host=ch):
        return lib.ism_attn_prefill_append(C.byref(sh), 2, FAKE, FAKE, FAKE, l_new, seg_end.ctypes.data,
                                           seg_type.ctypes.data, nseg, FAKE, FAKE, cap, FAKE,
                                           cache_host.ctypes.data, FAKE, None, FAKE, 1 << 30, None)
    assert call(cap=27) == 1                                      # 20 + 8 > 27: cache overflow
    assert "exceeds capacity" in lib.ism_last_error().decode()
    assert call(l_new=9) == 1                                     # segments do not cover the chunk
    assert call(seg_type=np.array([0, 2], np.uint8)) == 1
    assert call(nseg=0) == 1
    assert call(cache_host=np.array([-1, 0], np.int32)) == 1
    many_end = np.arange(1, 258, dtype=np.int32)                  # 257 segments: one past the limit
    many_type = np.zeros(257, np.uint8)
    assert call(l_new=257, cap=300, seg_end=many_end, seg_type=many_type, nseg=257) == 1
    assert "1..256 segments" in lib.ism_last_error().decode()


@host_only
def test_paged_append_errors(lib):
    sh = _shape()
    se = np.array([4, 8], np.int32)
    st = np.array([0, 1], np.uint8)
    ch = np.array([10, 20], np.int32)
    bt = np.array([[0, 1], [2, 3]], np.int32)

    def call(page_size=128, num_pages=4, table=bt, max_pages=2, cache_host=ch):
        return lib.ism_attn_prefill_append_paged(C.byref(sh), 2, FAKE, FAKE, FAKE, 8, se.ctypes.data, st.ctypes.data,
                                                 2, FAKE, FAKE, num_pages, page_size, FAKE, table.ctypes.data,
                                                 max_pages, FAKE, cache_host.ctypes.data, FAKE, None, FAKE, 1 << 30,
                                                 None)
    assert call(page_size=64) == 1 and "page_size" in lib.ism_last_error().decode()
    bad = bt.copy()
    bad[1, 0] = 4                                                 # one past the pool
    assert call(table=bad) == 1 and "outside" in lib.ism_last_error().decode()
    assert call(cache_host=np.array([10, 250], np.int32)) == 1   # 250 + 8 keys > 2 pages of 128
    assert call(max_pages=0) == 1
    assert call(num_pages=0) == 1


class _Rope(C.Structure):
    _fields_ = [("cos", C.c_void_p), ("sin", C.c_void_p), ("rows", C.c_int32)]


@host_only
def test_rope_append_errors(lib):
    se = np.array([4, 8], np.int32)
    st = np.array([0, 1], np.uint8)
    ch = np.array([10, 20], np.int32)

    def call(rope, sh=None):
        sh = _shape() if sh is None else sh
        return lib.ism_attn_prefill_append_rope(C.byref(sh), 2, FAKE, FAKE, FAKE, 8, se.ctypes.data, st.ctypes.data,
                                                2, FAKE, FAKE, 64, FAKE, ch.ctypes.data,
                                                None if rope is None else C.byref(rope), FAKE, None, FAKE, 1 << 30,
                                                None)
    assert call(None) == 1 and "rope is NULL" in lib.ism_last_error().decode()
    assert call(_Rope(FAKE, FAKE, 28), sh=_shape(dtype=1)) == 1          # bf16 only
    assert call(_Rope(FAKE + 4, FAKE, 28)) == 1                          # misaligned table
    assert call(_Rope(None, FAKE, 28)) == 1
    assert call(_Rope(FAKE, FAKE, 27)) == 1                              # positions up to 20 + 8
    assert "rope tables cover 27" in lib.ism_last_error().decode()
    need, base = C.c_size_t(), C.c_size_t()
    assert lib.ism_attn_prefill_append_rope_workspace_size(C.byref(_shape()), 2, 8, C.byref(need)) == 0
    assert lib.ism_attn_prefill_append_workspace_size(C.byref(_shape()), 2, 8, C.byref(base)) == 0
    assert need.value >= base.value + 2 * 8 * 4 * 128 * 2                # plus the rotated queries


@host_only
def test_e4m3_entry_errors(lib):
    keep = _Keep()
    s = _segs([0, 10], [0, 2], [4, 10], [0, 1], keep)
    assert _fwd(lib, s, _shape(dtype=2)) == 2                    # e4m3 only through ism_attn_fwd_e4m3

    def fwd8(sh, qd=1.0, kd=1.0, vd=1.0):
        return lib.ism_attn_fwd_e4m3(C.byref(s), C.byref(sh), FAKE, FAKE, FAKE, qd, kd, vd, FAKE, FAKE, FAKE, 1 << 30,
                                     None)
    assert fwd8(_shape(dtype=0)) == 1                            # shape must say ISM_E4M3
    assert fwd8(_shape(dtype=2), qd=0.0) == 1                    # descales positive
    assert fwd8(_shape(dtype=2), vd=float("inf")) == 1
    need = C.c_size_t()
    assert lib.ism_attn_fwd_workspace_size(C.byref(s), C.byref(_shape(dtype=2)), C.byref(need)) == 0
    assert lib.ism_attn_fwd_workspace_size(C.byref(s), C.byref(_shape(dtype=2, d=64)), C.byref(need)) == 2


def test_plan_size_host_only(lib):
    """The plan's size is a host computation: the per-token key bounds, the
    tile descriptors and work lists of both passes, growing with the tokens;
    the same for any softmax scale."""
    keep = _Keep()
    sizes = []
    for L in (100, 1000, 10000):
        s = _segs([0, L], [0, 2], [L // 2, L], [0, 1], keep)
        n = C.c_size_t()
        assert lib.ism_attn_plan_size(C.byref(s), C.byref(_shape()), C.byref(n)) == 0
        n2 = C.c_size_t()
        assert lib.ism_attn_plan_size(C.byref(s), C.byref(_shape(scale=0.7)), C.byref(n2)) == 0
        assert n.value == n2.value
        sizes.append(n.value)
    assert sizes[0] < sizes[1] < sizes[2]
    assert sizes[2] >= 4 * 10000                                   # a key bound per token at least


@host_only
def test_planned_calls_need_a_plan(lib):
    """Planned calls without a plan or its host record are refused on the
    host before anything else."""
    keep = _Keep()
    s = _segs([0, 10], [0, 2], [4, 10], [0, 1], keep)
    info = ism._PlanInfo()
    r = lib.ism_attn_fwd_planned(C.byref(s), C.byref(_shape()), None, C.byref(info), FAKE, FAKE, FAKE, FAKE, FAKE,
                                 None)
    assert r == 1 and "plan" in lib.ism_last_error().decode()
    r = lib.ism_attn_bwd_planned(C.byref(s), C.byref(_shape()), FAKE, None, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE,
                                 FAKE, FAKE, FAKE, FAKE, 1 << 30, None)
    assert r == 1 and "plan" in lib.ism_last_error().decode()
