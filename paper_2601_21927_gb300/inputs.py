"""Seeded synthetic inputs shared by the CUDA path, the oracle and the benchmark.

This module holds input *structure* and random numbers only -- no step of the
attention, mask or retention arithmetic.  It builds augmented dialogue layouts
S_aug = {I_sys, m_1, N^(1), ..., m_h, N^(h), Q_curr} (Sec. 3.1, Eq. 1) as
per-token role and segment arrays, packs several dialogues into one ragged
batch, and draws N(0, 1) tensors from seeded torch generators.

Roles (stored as uint8): 0 = system prompt, 1 = segment body B_i,
2 = Nexus token N_i, 3 = current query / current turn.  Segment numbers
(int32): 0 = system prompt, i = history segment m_i (1..h), h+1 = current.

The workload recipes (shapes of the five named workloads) sit here too, so
that tests and the benchmark draw exactly the same inputs.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from typing import List, Optional, Sequence, Tuple

import numpy as np
import torch

ROLE_SYS, ROLE_BODY, ROLE_NEXUS, ROLE_CURR = 0, 1, 2, 3


@dataclass
class Dialogue:
    """One augmented dialogue: lengths of I_sys, each (body, Nexus) segment, Q_curr."""
    sys_len: int
    segments: List[Tuple[int, int]]  # (body length |B_i|, Nexus count K_i)
    curr_len: int

    @property
    def length(self) -> int:
        return self.sys_len + sum(b + k for b, k in self.segments) + self.curr_len

    @property
    def recipe_retained(self) -> int:
        """|I_sys| + sum_i K_i + |Q_curr|, read off the recipe (not computed by any rule)."""
        return self.sys_len + sum(k for _, k in self.segments) + self.curr_len

    def arrays(self) -> Tuple[np.ndarray, np.ndarray]:
        role = np.empty(self.length, np.uint8)
        seg = np.empty(self.length, np.int32)
        t = 0
        role[t:t + self.sys_len] = ROLE_SYS
        seg[t:t + self.sys_len] = 0
        t += self.sys_len
        for i, (b, k) in enumerate(self.segments, start=1):
            role[t:t + b] = ROLE_BODY
            seg[t:t + b] = i
            t += b
            role[t:t + k] = ROLE_NEXUS
            seg[t:t + k] = i
            t += k
        role[t:t + self.curr_len] = ROLE_CURR
        seg[t:t + self.curr_len] = len(self.segments) + 1
        return role, seg

    def retained_arrays(self) -> Tuple[np.ndarray, np.ndarray]:
        """Role/segment arrays of the dialogue with every body left out (recipe view)."""
        d = Dialogue(self.sys_len, [(0, k) for _, k in self.segments], self.curr_len)
        return d.arrays()


@dataclass
class Batch:
    """A ragged batch of dialogues packed along one token axis."""
    dialogues: List[Dialogue]
    role: np.ndarray = field(init=False)
    seg: np.ndarray = field(init=False)
    k_start: np.ndarray = field(init=False)
    k_len: np.ndarray = field(init=False)

    def __post_init__(self):
        roles, segs, starts, lens = [], [], [], []
        t = 0
        for d in self.dialogues:
            r, s = d.arrays()
            roles.append(r)
            segs.append(s)
            starts.append(t)
            lens.append(d.length)
            t += d.length
        self.role = np.concatenate(roles) if roles else np.zeros(0, np.uint8)
        self.seg = np.concatenate(segs) if segs else np.zeros(0, np.int32)
        self.k_start = np.asarray(starts, np.int32)
        self.k_len = np.asarray(lens, np.int32)

    @property
    def total(self) -> int:
        return int(self.k_len.sum())

    @property
    def B(self) -> int:
        return len(self.dialogues)


def random_dialogue(rng: np.random.Generator, max_segments: int = 5, max_body: int = 40,
                    max_nexus: int = 6, max_sys: int = 20, max_curr: int = 30,
                    allow_empty: bool = True) -> Dialogue:
    """A small random dialogue, including degenerate pieces (K_i = 0, empty body,
    no history, empty system prompt) when allow_empty is set."""
    lo = 0 if allow_empty else 1
    h = int(rng.integers(0, max_segments + 1))
    segs = [(int(rng.integers(lo, max_body + 1)), int(rng.integers(lo, max_nexus + 1)))
            for _ in range(h)]
    return Dialogue(int(rng.integers(lo, max_sys + 1)), segs,
                    int(rng.integers(1, max_curr + 1)))


# ---------------------------------------------------------------------------
# Seeded tensors
# ---------------------------------------------------------------------------

def randn(shape: Sequence[int], seed: int, dtype=torch.bfloat16, device="cpu",
          chunk_elems: int = 1 << 28) -> torch.Tensor:
    """N(0, 1) values, drawn in float32 from a seeded generator and rounded
    (round-to-nearest-even) to ``dtype``.  Large tensors are drawn in chunks
    of the flattened tensor so the float32 temporary stays small."""
    shape = tuple(int(s) for s in shape)
    n = int(np.prod(shape)) if shape else 1
    out = torch.empty(n, dtype=dtype, device=device)
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    for s in range(0, n, chunk_elems):
        e = min(n, s + chunk_elems)
        out[s:e] = torch.randn(e - s, generator=g, device=device,
                               dtype=torch.float32).to(dtype)
    return out.view(shape)


# ---------------------------------------------------------------------------
# Workload recipes (the five named workloads)
# ---------------------------------------------------------------------------

@dataclass
class Heads:
    n_layers: int
    hq: int
    hkv: int
    d: int


def tiny_ref() -> Tuple[Batch, Heads]:
    """1 layer, 2 query / 1 KV head, D = 64; 16 system tokens, 3 history
    segments of 32 body + 4 Nexus tokens, a 24-token current query (L = 148)."""
    return Batch([Dialogue(16, [(32, 4)] * 3, 24)]), Heads(1, 2, 1, 64)


def decode_llama8b() -> Tuple[Batch, Heads]:
    """Batch 16; 256 system tokens, 8 history turns of 256 body tokens with 32
    Nexus tokens each, a 128-token current turn (L = 2688, retained 640);
    32 layers, 32 query / 8 KV heads, D = 128."""
    return Batch([Dialogue(256, [(256, 32)] * 8, 128) for _ in range(16)]), Heads(32, 32, 8, 128)


def masked_prefill() -> Tuple[Batch, Heads]:
    """Batch 8; 512 system tokens, 16 history segments of 256 body + 32 Nexus
    tokens, a 512-token current turn (L = 5632, retained 1536); 32 layers,
    32 query / 8 KV heads, D = 128."""
    return Batch([Dialogue(512, [(256, 32)] * 16, 512) for _ in range(8)]), Heads(32, 32, 8, 128)


def long_ragged(nexus_div: int, seed: int = 1, batch: int = 64,
                sys_len: int = 256) -> Tuple[Batch, Heads]:
    """Batch 64 ragged dialogues: turn count ~ U[4, 32], turn length
    ~ U[64, 1024]; the last turn is the current one; every history turn gets
    ceil(len / nexus_div) Nexus tokens (nexus_div = 2 or 5); 256 system
    tokens; 32 layers, 32 query / 8 KV heads, D = 128."""
    rng = np.random.default_rng(seed)
    dl = []
    for _ in range(batch):
        n_turns = int(rng.integers(4, 33))
        lens = rng.integers(64, 1025, size=n_turns)
        segs = [(int(x), int(math.ceil(int(x) / nexus_div))) for x in lens[:-1]]
        dl.append(Dialogue(sys_len, segs, int(lens[-1])))
    return Batch(dl), Heads(32, 32, 8, 128)


@dataclass
class MixedStep:
    """Mixed serving step: sequences 0..n_prefill-1 resume with a new current
    turn (their raw history is compacted, then the turn is prefilled over the
    retained cache); the rest decode one token over their retained cache."""
    heads: Heads
    raw_hist: List[Dialogue]      # prefill sequences: raw history, curr_len = 0
    prefill_q: List[int]          # new current-turn length of each prefill sequence
    decode_hist: List[Dialogue]   # decode sequences: retained cache (bodies already gone)
    reserve: int                  # free rows after every retained sequence


def mixed_serving(seed: int = 1, batch: int = 64, n_prefill: int = 8,
                  sys_len: int = 256, nexus_div: int = 3,
                  raw_range=(4096, 65536), turn_range=(64, 1024),
                  q_range=(256, 2048)) -> MixedStep:
    """Qwen-like heads (28 layers, 28 query / 4 KV heads, D = 128).  Raw
    histories of ~U[4k, 64k] tokens made of turns ~U[64, 1024] with
    ceil(len / 3) Nexus tokens each, so the retained cache is about a quarter
    of the raw history (1k-16k rows).  8 sequences prefill a new current turn
    ~U[256, 2048]; 56 decode one token, their current turn (~U[256, 2048]
    tokens so far) already in the retained cache."""
    rng = np.random.default_rng(seed)
    heads = Heads(28, 28, 4, 128)

    def history():
        target = int(rng.integers(raw_range[0], raw_range[1] + 1))
        segs, n = [], sys_len
        while True:
            x = int(rng.integers(turn_range[0], turn_range[1] + 1))
            k = int(math.ceil(x / nexus_div))
            if n + x + k > target and segs:
                break
            segs.append((x, k))
            n += x + k
        return segs

    raw, qs, dec = [], [], []
    for b in range(batch):
        segs = history()
        if b < n_prefill:
            raw.append(Dialogue(sys_len, segs, 0))
            qs.append(int(rng.integers(q_range[0], q_range[1] + 1)))
        else:
            cur = int(rng.integers(q_range[0], q_range[1] + 1))
            dec.append(Dialogue(sys_len, segs, cur))
    return MixedStep(heads, raw, qs, dec, reserve=max(q_range[1], 1) + 64)
