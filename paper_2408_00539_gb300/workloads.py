"""Seeded synthetic dialogue workloads for ISM attention.

This module only draws inputs: dialogue segment structures (query/answer
turn boundaries, Section 2.1 of the paper: a sample is [P, Q1, A1, ..., Qn])
and random Q/K/V/dO values.  It holds none of the attention arithmetic and
none of the mask rule, so both the CUDA path and the fp64 oracle can take
their inputs from it.

Segment format (shared by every consumer):
  * ``cu_seqlens`` int32 [B+1]  token offsets of the packed sequences
  * ``cu_segs``    int32 [B+1]  segment offsets per sequence
  * ``seg_end``    int32 [nseg] exclusive end of each segment, relative to
                                its sequence (the paper's m_{q_k}, m_{a_k})
  * ``seg_type``   uint8 [nseg] 0 = QUERY (the prompt P is part of the first
                                query segment), 1 = ANSWER

Length distributions follow the dialogue statistics used for the measured
workloads: turns drawn uniformly, query lengths log-normal with median 64
(clipped to [8, 1024]) and answer lengths log-normal with median 256 (clipped
to [16, 2048]), sigma 1.0.  A dialogue longer than the target length is
truncated; a shorter one has its final answer extended to fill it.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import List, Optional, Sequence, Tuple

import numpy as np

QUERY = 0
ANSWER = 1

Q_MEDIAN, Q_CLIP = 64.0, (8, 1024)
A_MEDIAN, A_CLIP = 256.0, (16, 2048)
LOGNORMAL_SIGMA = 1.0


@dataclass
class Segments:
    cu_seqlens: np.ndarray
    cu_segs: np.ndarray
    seg_end: np.ndarray
    seg_type: np.ndarray

    @property
    def num_seqs(self) -> int:
        return int(self.cu_seqlens.shape[0] - 1)

    @property
    def total_tokens(self) -> int:
        return int(self.cu_seqlens[-1])

    @property
    def num_segs(self) -> int:
        return int(self.seg_end.shape[0])

    def seq(self, b: int) -> Tuple[int, int, np.ndarray, np.ndarray]:
        """(start token, length, seg_end, seg_type) of sequence b."""
        t0, t1 = int(self.cu_seqlens[b]), int(self.cu_seqlens[b + 1])
        s0, s1 = int(self.cu_segs[b]), int(self.cu_segs[b + 1])
        return t0, t1 - t0, self.seg_end[s0:s1], self.seg_type[s0:s1]


def pack(dialogues: Sequence[Tuple[Sequence[int], Sequence[int]]]) -> Segments:
    """Pack per-dialogue (seg_end, seg_type) lists into the varlen format."""
    cu_seqlens = [0]
    cu_segs = [0]
    ends: List[int] = []
    types: List[int] = []
    for seg_end, seg_type in dialogues:
        assert len(seg_end) == len(seg_type) and len(seg_end) > 0
        cu_seqlens.append(cu_seqlens[-1] + int(seg_end[-1]))
        cu_segs.append(cu_segs[-1] + len(seg_end))
        ends.extend(int(e) for e in seg_end)
        types.extend(int(t) for t in seg_type)
    return Segments(
        cu_seqlens=np.asarray(cu_seqlens, dtype=np.int32),
        cu_segs=np.asarray(cu_segs, dtype=np.int32),
        seg_end=np.asarray(ends, dtype=np.int32),
        seg_type=np.asarray(types, dtype=np.uint8),
    )


def lengths_to_segments(lengths: Sequence[int], types: Sequence[int]):
    ends = np.cumsum(np.asarray(lengths, dtype=np.int64)).astype(np.int32)
    return ends.tolist(), [int(t) for t in types]


def _lognormal_len(rng: np.random.Generator, median: float, clip) -> int:
    x = rng.lognormal(mean=np.log(median), sigma=LOGNORMAL_SIGMA)
    return int(np.clip(np.round(x), clip[0], clip[1]))


def draw_dialogue(rng: np.random.Generator, length: int, turns_lo: int, turns_hi: int):
    """One dialogue of exactly ``length`` tokens as (seg_end, seg_type).

    Turns are (query, answer) pairs; the stream is truncated at ``length``
    or, when shorter, its last answer is extended to reach ``length``.
    """
    n_turns = int(rng.integers(turns_lo, turns_hi + 1))
    lens: List[int] = []
    types: List[int] = []
    total = 0
    for _ in range(n_turns):
        for kind, med, clip in ((QUERY, Q_MEDIAN, Q_CLIP), (ANSWER, A_MEDIAN, A_CLIP)):
            if total >= length:
                break
            n = min(_lognormal_len(rng, med, clip), length - total)
            lens.append(n)
            types.append(kind)
            total += n
    if total < length:
        if types[-1] == ANSWER:
            lens[-1] += length - total
        else:
            lens.append(length - total)
            types.append(ANSWER)
    return lengths_to_segments(lens, types)


@dataclass
class Workload:
    name: str
    segs: Segments
    num_heads_q: int
    num_heads_kv: int
    head_dim: int
    dtype: str  # "bf16" or "fp32"
    softmax_scale: float
    value_std: float
    seed: int
    extra: dict = field(default_factory=dict)

    @property
    def total_tokens(self) -> int:
        return self.segs.total_tokens


def tiny_fp32(seed: int = 1) -> Workload:
    """One 256-token dialogue of 3 turns, query/answer lengths
    [40,30],[30,60],[50,46]; 2 heads, head_dim 64, fp32, values N(0,1)."""
    ends, types = lengths_to_segments([40, 30, 30, 60, 50, 46], [0, 1, 0, 1, 0, 1])
    return Workload("tiny_fp32_L256_H2_D64", pack([(ends, types)]), 2, 2, 64, "fp32",
                    1.0 / np.sqrt(64.0), 1.0, seed)


def mha_4k(seed: int = 2, batch: int = 4, seqlen: int = 4096) -> Workload:
    """Batch 4 x 4096, 32 heads MHA, head_dim 128, bf16, 2-8 turns."""
    rng = np.random.Generator(np.random.PCG64(seed))
    dia = [draw_dialogue(rng, seqlen, 2, 8) for _ in range(batch)]
    return Workload(f"mha_b{batch}_s{seqlen}_h32_d128", pack(dia), 32, 32, 128, "bf16",
                    1.0 / np.sqrt(128.0), 0.5, seed)


def gqa_8k(seed: int = 3, batch: int = 2, seqlen: int = 8192) -> Workload:
    """Batch 2 x 8192, 32 query heads / 8 KV heads, head_dim 128, bf16,
    4-16 turns, softmax scale 1/sqrt(128)."""
    rng = np.random.Generator(np.random.PCG64(seed))
    dia = [draw_dialogue(rng, seqlen, 4, 16) for _ in range(batch)]
    return Workload(f"gqa_b{batch}_s{seqlen}_hq32_hkv8_d128", pack(dia), 32, 8, 128, "bf16",
                    1.0 / np.sqrt(128.0), 0.5, seed)


def packed_32k(seed: int = 4, total: int = 32768, min_len: int = 512) -> Workload:
    """One 32768-token buffer of 4-8 packed dialogues with random lengths
    (uniform cut points, at least ``min_len`` tokens each, not tile
    aligned), 2-32 turns each, 32 query heads / 8 KV heads, head_dim 128."""
    rng = np.random.Generator(np.random.PCG64(seed))
    n = int(rng.integers(4, 9))
    while True:
        cuts = np.sort(rng.choice(np.arange(1, total), size=n - 1, replace=False))
        lens = np.diff(np.concatenate([[0], cuts, [total]]))
        if lens.min() >= min_len:
            break
    dia = [draw_dialogue(rng, int(L), 2, 32) for L in lens]
    return Workload(f"packed_t{total}_n{n}_hq32_hkv8_d128", pack(dia), 32, 8, 128, "bf16",
                    1.0 / np.sqrt(128.0), 0.5, seed)


def long_dialogue(length: int, seed: int = 131, turns=(300, 400)) -> Workload:
    """One dialogue of ``length`` tokens with a few hundred turns of the
    config-2 length recipe, 32 query / 8 KV heads, head_dim 128, bf16."""
    rng = np.random.Generator(np.random.PCG64(seed))
    dia = [draw_dialogue(rng, length, turns[0], turns[1])]
    return Workload(f"long_t{length}_hq32_hkv8_d128", pack(dia), 32, 8, 128, "bf16", 1.0 / np.sqrt(128.0), 0.5, seed)


@dataclass
class AppendWorkload:
    name: str
    batch: int
    cache_len: np.ndarray      # int32 [B]
    capacity: int
    l_new: int
    new_seg_end: np.ndarray    # int32, chunk-relative
    new_seg_type: np.ndarray   # uint8
    decode_steps: int
    num_heads_q: int
    num_heads_kv: int
    head_dim: int
    softmax_scale: float
    value_std: float
    seed: int


def append_16k(seed: int = 5, batch: int = 8, cache_len: int = 16384, l_new: int = 512,
               decode_steps: int = 256) -> AppendWorkload:
    """KV cache of 16384 tokens per sequence (batch 8, 32 query / 8 KV heads,
    head_dim 128, bf16), a new 512-token query segment appended, then 256
    single-token answer (causal) decode steps against the grown cache."""
    cap = cache_len + l_new + decode_steps
    return AppendWorkload(f"append_b{batch}_c{cache_len}_n{l_new}_dec{decode_steps}", batch,
                          np.full((batch,), cache_len, dtype=np.int32), cap, l_new,
                          np.asarray([l_new], dtype=np.int32), np.asarray([QUERY], dtype=np.uint8),
                          decode_steps, 32, 8, 128, 1.0 / np.sqrt(128.0), 0.5, seed)


def triplet_expansion(segs: Segments) -> Segments:
    """The training samples a prefix-LM needs for the same dialogues: one per
    answer segment, holding everything before the answer as one bidirectional
    prefix (a QUERY segment) followed by the answer (causal).  Each sample
    re-reads the whole history that the one-pass ISM sequence shares."""
    samples = []
    for b in range(segs.num_seqs):
        _, _, se, st = segs.seq(b)
        start = 0
        for e, t in zip(se.tolist(), st.tolist()):
            if t == ANSWER and e > start:
                samples.append(([start, e], [QUERY, ANSWER]) if start > 0 else ([e], [ANSWER]))
            start = e
    return pack(samples)


@dataclass
class SessionWorkload:
    """A serving session: every dialogue of the batch alternates a query turn,
    appended in one prefill call, and an answer generated one token at a time
    (decode calls), against a KV cache that keeps the whole dialogue."""
    name: str
    batch: int
    turns: int
    q_len: int
    a_len: int
    num_heads_q: int
    num_heads_kv: int
    head_dim: int
    softmax_scale: float
    value_std: float
    seed: int

    @property
    def capacity(self) -> int:
        return self.turns * (self.q_len + self.a_len)

    def dialogue(self):
        """(seg_end, seg_type) of one whole dialogue."""
        ends, types, pos = [], [], 0
        for _ in range(self.turns):
            pos += self.q_len
            ends.append(pos)
            types.append(QUERY)
            pos += self.a_len
            ends.append(pos)
            types.append(ANSWER)
        return ends, types


def latency_session(seed: int = 6, batch: int = 40, turns: int = 20, q_len: int = 40, a_len: int = 160) -> SessionWorkload:
    """The shape of the paper's latency experiment (Section 3.6): 40 dialogues of
    20 turns, 40 query and 160 answer tokens a turn (context up to 4000 tokens),
    here for one attention layer of 32 query / 8 KV heads, head_dim 128, bf16."""
    return SessionWorkload(f"session_b{batch}_t{turns}_q{q_len}_a{a_len}", batch, turns, q_len, a_len, 32, 8, 128,
                           1.0 / np.sqrt(128.0), 0.5, seed)


def normal(rng: np.random.Generator, shape, std: float) -> np.ndarray:
    return (rng.standard_normal(size=shape, dtype=np.float32) * np.float32(std)).astype(np.float32)


def round_to(x: np.ndarray, dtype: str):
    """Return a torch CPU tensor holding ``x`` rounded to ``dtype``."""
    import torch
    t = torch.from_numpy(np.ascontiguousarray(x))
    return t.to(torch.bfloat16) if dtype == "bf16" else t.to(torch.float32)


def attention_tensors(w: Workload, with_dout: bool = True, seed_offset: int = 0):
    """Q [T,Hq,D], K,V [T,Hkv,D] (and dO [T,Hq,D]) as torch CPU tensors of
    the workload's dtype; dO is drawn from N(0,1)."""
    rng = np.random.Generator(np.random.PCG64(w.seed + 1000 * seed_offset))
    T = w.total_tokens
    q = round_to(normal(rng, (T, w.num_heads_q, w.head_dim), w.value_std), w.dtype)
    k = round_to(normal(rng, (T, w.num_heads_kv, w.head_dim), w.value_std), w.dtype)
    v = round_to(normal(rng, (T, w.num_heads_kv, w.head_dim), w.value_std), w.dtype)
    out = [q, k, v]
    if with_dout:
        out.append(round_to(normal(rng, (T, w.num_heads_q, w.head_dim), 1.0), w.dtype))
    return tuple(out)


def quantize_e4m3(x):
    """Per-tensor e4m3 (float8_e4m3fn) copy of a torch tensor: the values are
    scaled so that the largest magnitude maps to 448, the format's largest
    finite value, and rounded to nearest.  Returns (x8, descale) with
    x ~= x8.float() * descale."""
    import torch
    amax = float(x.float().abs().max())
    descale = amax / 448.0 if amax > 0 else 1.0
    return (x.float() / descale).to(torch.float8_e4m3fn), descale


def rope_tables(rows: int, head_dim: int, base: float = 10000.0):
    """Rotary-encoding tables, an input of the RoPE append: position p and
    pair k < head_dim/2 get the angle p * base**(-2k/head_dim) (the usual
    frequency schedule); returns (cos, sin) as float32 numpy arrays
    [rows, head_dim/2].  Any table of cosines and sines is a valid input."""
    half = head_dim // 2
    inv_freq = base ** (-2.0 * np.arange(half, dtype=np.float64) / head_dim)
    ang = np.arange(rows, dtype=np.float64)[:, None] * inv_freq[None, :]
    return np.cos(ang).astype(np.float32), np.sin(ang).astype(np.float32)


def random_dialogue_set(rng: np.random.Generator, n_seqs: int, max_len: int,
                        zero_len: bool = True, min_len: int = 1) -> Segments:
    """Small random segmentations for tests: any mix of QUERY/ANSWER
    segments, including zero-length segments, consecutive segments of one
    type and dialogues that start with an answer."""
    dia = []
    for _ in range(n_seqs):
        L = int(rng.integers(min_len, max_len + 1))
        cuts = sorted(int(c) for c in rng.integers(0, L + 1, size=int(rng.integers(0, 8))))
        if not zero_len:
            cuts = sorted(set(c for c in cuts if 0 < c < L))
        bounds = [0] + cuts + [L]
        ends = bounds[1:]
        types = [int(t) for t in rng.integers(0, 2, size=len(ends))]
        dia.append((ends, types))
    return pack(dia)
