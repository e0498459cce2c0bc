"""CPU checks of the benchmark's host logic."""
import numpy as np

import bench
from oracle import ism_oracle as orc
from paper_2408_00539_gb300 import workloads as wl


def test_visible_pair_count_matches_mask():
    rng = np.random.Generator(np.random.PCG64(5))
    segs = wl.random_dialogue_set(rng, 20, 300)
    assert bench.n_visible(segs) == int(orc.packed_mask(segs).sum())
    tiny = wl.tiny_fp32().segs
    assert bench.n_visible(tiny) == int(orc.packed_mask(tiny).sum())


def test_headline_density_close_to_half():
    w = wl.gqa_8k()
    dens = bench.n_visible(w.segs) / sum(L * L for L in np.diff(w.segs.cu_seqlens))
    assert 0.5 <= dens <= 0.56


def test_tile_pair_count_matches_tile_map():
    """The stored-dS traffic figure counts the non-empty 128 x 128 tiles."""
    rng = np.random.Generator(np.random.PCG64(6))
    for segs in (wl.random_dialogue_set(rng, 30, 700), wl.gqa_8k().segs, wl.tiny_fp32().segs):
        ref = int(orc.tile_map_packed(segs, 128, 128)["kt_end"].sum())
        assert bench.n_tile_pairs(segs) == ref


def test_session_workload_shape():
    s = wl.latency_session()
    ends, types = s.dialogue()
    assert s.capacity == 4000 and ends[-1] == s.capacity and len(ends) == 2 * s.turns
    assert types == [wl.QUERY, wl.ANSWER] * s.turns
    assert all(b - a in (s.q_len, s.a_len) for a, b in zip([0] + ends[:-1], ends))


def test_triplet_expansion_samples_and_counts():
    # one sample per non-empty answer: everything before it as one bidirectional
    # prefix, then the answer; pair counts agree with the materialised masks
    segs = wl.pack([([5, 12, 20, 33], [wl.QUERY, wl.ANSWER, wl.QUERY, wl.ANSWER]),
                    ([4, 9, 9], [wl.ANSWER, wl.QUERY, wl.ANSWER])])
    tri = wl.triplet_expansion(segs)
    got = [(tri.seq(b)[2].tolist(), tri.seq(b)[3].tolist()) for b in range(tri.num_seqs)]
    assert got == [([5, 12], [0, 1]), ([20, 33], [0, 1]), ([4], [1])]
    brute = sum(int(orc.mask_eq_fj(se, st).sum()) for _, _, se, st in (tri.seq(b) for b in range(tri.num_seqs)))
    assert bench.n_visible(tri) == brute
    # the one pass over each dialogue sees fewer pairs than its samples together
    assert bench.n_visible(segs) < bench.n_visible(tri)
