"""Seeded synthetic inputs shared by the oracle's tests and the GPU benchmark.

This module holds no arithmetic of the eviction method.  It provides:

* the counter-based generator of bf16 keys/values/queries (definition in
  ``csrc/synth_gen.h``): a host C build and a CUDA build of one source, plus a
  numpy restatement used to cross-check both;
* the trace recipes (region spans, insertion steps, budgets, region parameters)
  of the five workload configurations, shaped after the paper's agent traces
  (Sec. IV-A: ~450- and ~1,700-token episodes built from contiguous region
  spans, Sec. III-A) and the scaled serving batches.

Region ids follow the order the paper lists them in Sec. III-A.
"""
from __future__ import annotations

import ctypes
import math
import os
import subprocess
from dataclasses import dataclass, field, replace
from typing import List, Optional, Sequence

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libmdsynth.so")
SRC = [os.path.join(HERE, "csrc", "synth.cu")]
HDR = [os.path.join(HERE, "csrc", "synth_gen.h")]

REGIONS = ("system", "plan", "user", "tool_in", "tool_out", "retrieval", "scratchpad")
SYSTEM, PLAN, USER, TOOL_IN, TOOL_OUT, RETRIEVAL, SCRATCHPAD = range(7)

T_K, T_V, T_Q, T_SIGN, T_HOT = 1, 2, 3, 5, 6
NORM = np.float32(2.6429130e-05)
STRUCT_DIMS = 16
HOT_THRESHOLD = 335544

# Structured variant: per-region key offsets (multiples of 1/64), chosen so the
# logit gain kappa_q*kappa_r*16/sqrt(128) approximates ln(m_r / m_min) for the
# young-age attention masses the paper plots per region (Fig. 3): system
# 0.01355, plan 0.00118, tool_out 0.00114, retrieval 0.00061, scratchpad 0.0245.
# user and tool_in are not plotted; they take tool_out's offset.
KAPPA_STRUCT = (2.1875, 0.46875, 0.4375, 0.4375, 0.4375, 0.0, 2.625, 2.0, 1.0)

M64 = (1 << 64) - 1


# ----------------------------------------------------------------- build ----
def build(force: bool = False, verbose: bool = False) -> str:
    """Compile libmdsynth.so (host + sm_103a device code) in-tree."""
    newest = max(os.path.getmtime(p) for p in SRC + HDR)
    if not force and os.path.exists(LIB_PATH) and os.path.getmtime(LIB_PATH) >= newest:
        return LIB_PATH
    cmd = [
        "nvcc", "-O2", "-shared", "-Xcompiler", "-fPIC", "-Xcompiler", "-ffp-contract=off",
        "-gencode", "arch=compute_103a,code=sm_103a", "-lineinfo",
        "-o", LIB_PATH + ".tmp", *SRC,
    ]
    if verbose:
        print(" ".join(cmd))
    subprocess.run(cmd, check=True)
    os.replace(LIB_PATH + ".tmp", LIB_PATH)
    return LIB_PATH


_lib = None


def lib():
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            build()
        L = ctypes.CDLL(LIB_PATH)
        u64, i32, vp = ctypes.c_uint64, ctypes.c_int, ctypes.c_void_p
        L.synth_key.restype = u64
        L.synth_key.argtypes = [u64]
        L.synth_fill_kv_host.restype = None
        L.synth_fill_kv_host.argtypes = [u64, i32, vp, i32, i32, i32, i32, i32, i32, vp, vp, vp]
        L.synth_fill_q_host.restype = None
        L.synth_fill_q_host.argtypes = [u64, i32, vp, i32, i32, i32, i32, i32, i32, vp]
        L.synth_fill_kv_dev.restype = i32
        L.synth_fill_kv_dev.argtypes = [u64, i32, vp, i32, i32, i32, i32, i32, i32, vp, vp, vp, vp]
        L.synth_fill_q_dev.restype = i32
        L.synth_fill_q_dev.argtypes = [u64, i32, vp, i32, i32, i32, i32, i32, i32, vp, vp]
        L.synth_fill_step_kv_dev.restype = i32
        L.synth_fill_step_kv_dev.argtypes = [u64, i32, vp, i32, i32, i32, i32, vp, vp, vp, vp, vp]
        _lib = L
    return _lib


def _kappa_arr(structured: bool):
    if not structured:
        return None, None
    arr = (ctypes.c_float * 9)(*KAPPA_STRUCT)
    return arr, ctypes.cast(arr, ctypes.c_void_p)


# ------------------------------------------------------- host fast fills ----
def kv_host(seed: int, b: int, L: int, Hkv: int, pos0: int, n: int,
            regions: Optional[np.ndarray] = None, structured: bool = False, D: int = 128):
    """Keys and values of sequence b, positions [pos0, pos0+n): uint16 [L][Hkv][n][D]."""
    k = np.empty((L, Hkv, n, D), np.uint16)
    v = np.empty((L, Hkv, n, D), np.uint16)
    keep, kp = _kappa_arr(structured)
    reg = None
    if regions is not None:
        reg = np.ascontiguousarray(regions, dtype=np.uint8)
    lib().synth_fill_kv_host(seed, int(structured), kp, b, L, Hkv, D, pos0, n,
                             None if reg is None else reg.ctypes.data,
                             k.ctypes.data, v.ctypes.data)
    return k, v


def q_host(seed: int, B: int, L: int, Hq: int, Hkv: int, step: int,
           structured: bool = False, D: int = 128):
    """Queries of decode step `step`: uint16 [B][L][Hq][D]."""
    q = np.empty((B, L, Hq, D), np.uint16)
    keep, kp = _kappa_arr(structured)
    lib().synth_fill_q_host(seed, int(structured), kp, B, L, Hq, Hq // Hkv, D, step, q.ctypes.data)
    return q


def step_kv_host(seed: int, positions: Sequence[int], regions: Sequence[int], L: int, Hkv: int,
                 structured: bool = False, D: int = 128):
    """New token keys/values for a decode step: uint16 [B][L][Hkv][D]."""
    B = len(positions)
    k = np.empty((B, L, Hkv, D), np.uint16)
    v = np.empty((B, L, Hkv, D), np.uint16)
    for b in range(B):
        kb, vb = kv_host(seed, b, L, Hkv, int(positions[b]), 1,
                         np.array([regions[b]], np.uint8), structured, D)
        k[b] = kb[:, :, 0, :]
        v[b] = vb[:, :, 0, :]
    return k, v


# --------------------------------------------------- numpy restatement ----
def splitmix64_np(x: np.ndarray) -> np.ndarray:
    x = np.asarray(x, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = x + np.uint64(0x9E3779B97F4A7C15)
        z = (z ^ (z >> np.uint64(30))) * np.uint64(0xBF58476D1CE4E5B9)
        z = (z ^ (z >> np.uint64(27))) * np.uint64(0x94D049BB133111EB)
    return z ^ (z >> np.uint64(31))


def ctr_np(tensor, b, l, h, pos, d) -> np.ndarray:
    u = np.uint64
    return ((u(tensor) & u(0xF)) << u(60)) | ((np.asarray(b, np.uint64) & u(0xFFF)) << u(48)) | \
        ((np.asarray(l, np.uint64) & u(0xFF)) << u(40)) | ((np.asarray(h, np.uint64) & u(0x3F)) << u(34)) | \
        ((np.asarray(pos, np.uint64) & u(0x3FFFFFF)) << u(8)) | (np.asarray(d, np.uint64) & u(0xFF))


def bf16_rne_np(f: np.ndarray) -> np.ndarray:
    u = np.asarray(f, np.float32).view(np.uint32).astype(np.uint64)
    u = u + np.uint64(0x7FFF) + ((u >> np.uint64(16)) & np.uint64(1))
    return ((u >> np.uint64(16)) & np.uint64(0xFFFF)).astype(np.uint16)


def normal_f32_np(seed: int, tensor: int, b, l, h, pos, d) -> np.ndarray:
    key = splitmix64_np(np.uint64(seed & M64))
    z = splitmix64_np(ctr_np(tensor, b, l, h, pos, d) ^ key)
    m = np.uint64(0xFFFF)
    s = (z & m).astype(np.int64) + ((z >> np.uint64(16)) & m).astype(np.int64) + \
        ((z >> np.uint64(32)) & m).astype(np.int64) + ((z >> np.uint64(48)) & m).astype(np.int64)
    return (s - 131070).astype(np.float32) * NORM


def sign_np(seed: int, l, kvh, d) -> np.ndarray:
    key = splitmix64_np(np.uint64(seed & M64))
    z = splitmix64_np(ctr_np(T_SIGN, 0, l, kvh, 0, d) ^ key)
    return np.where((z & np.uint64(1)) == 1, np.float32(1.0), np.float32(-1.0))


def hot_np(seed: int, b, pos) -> np.ndarray:
    key = splitmix64_np(np.uint64(seed & M64))
    z = splitmix64_np(ctr_np(T_HOT, b, 0, 0, pos, 0) ^ key)
    return (z >> np.uint64(40)) < np.uint64(HOT_THRESHOLD)


def key_bits_np(seed, b, l, kvh, pos, d, region, structured=False) -> np.ndarray:
    v = normal_f32_np(seed, T_K, b, l, kvh, pos, d)
    if structured:
        kap = np.asarray(KAPPA_STRUCT[:7], np.float32)[np.asarray(region)]
        kap = np.where(hot_np(seed, b, pos), kap + np.float32(KAPPA_STRUCT[7]), kap).astype(np.float32)
        add = (kap * sign_np(seed, l, kvh, d)).astype(np.float32)
        v = np.where(np.asarray(d) < STRUCT_DIMS, (v + add).astype(np.float32), v)
    return bf16_rne_np(v)


def bf16_to_f64(bits: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns."""
    return (np.asarray(bits, np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32).astype(np.float64)


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    return bf16_rne_np(np.asarray(x, np.float32))


# ----------------------------------------------------------- workloads ----
DEFAULT_BASE = (1.0, 0.8, 0.7, 0.4, 0.3, 0.5, 0.2)
DEFAULT_HALF_LIFE = (160.0, 80.0, 60.0, 30.0, 25.0, 40.0, 15.0)
DEFAULT_PINNED = (1, 0, 0, 0, 0, 0, 0)
CONFIG0_SPANS = (64, 48, 48, 32, 96, 96, 64)


@dataclass
class Workload:
    """One synthetic workload: geometry, traces, policy parameters, schedule."""
    name: str
    L: int
    Hq: int
    Hkv: int
    page_size: int
    regions: List[np.ndarray]          # per sequence, uint8 per prefill token
    insert_steps: List[np.ndarray]     # per sequence, int32 per prefill token
    budget_pages: List[int]            # per sequence
    steps: int                         # decode steps
    window_k: int = 1                  # observation (md_evict) every k steps
    base: Sequence[float] = DEFAULT_BASE
    half_life: Sequence[float] = DEFAULT_HALF_LIFE
    pinned: Sequence[int] = DEFAULT_PINNED
    attn_weight: float = 1.0
    rho: float = 0.9
    gamma: float = 0.1
    tau_scale: float = 2.0
    score_mode: int = 0
    page_reduce: int = 0
    decode_region: int = SCRATCHPAD
    seed: int = 0
    structured: bool = False
    D: int = 128
    extra: dict = field(default_factory=dict)

    @property
    def B(self) -> int:
        return len(self.regions)

    @property
    def G(self) -> int:
        return self.Hq // self.Hkv

    def n0(self, b: int) -> int:
        return int(len(self.regions[b]))

    def pages0(self, b: int) -> int:
        return -(-self.n0(b) // self.page_size)

    def max_pages_per_seq(self) -> int:
        return max(self.pages0(b) for b in range(self.B)) + self.steps // self.page_size + 2

    def num_phys_pages(self) -> int:
        return sum(self.pages0(b) for b in range(self.B)) + self.B * (self.steps // self.page_size + 2)

    def describe(self) -> str:
        n = [self.n0(b) for b in range(self.B)]
        return (f"{self.name}: L={self.L} Hq={self.Hq} Hkv={self.Hkv} D={self.D} ps={self.page_size} "
                f"B={self.B} tokens/seq={min(n)}..{max(n)} budget={min(self.budget_pages)} pages "
                f"steps={self.steps} k={self.window_k} w={self.attn_weight} "
                f"{'structured' if self.structured else 'iid'} seed={self.seed}")


def largest_remainder(total: int, weights: Sequence[float], minimum: int = 0) -> List[int]:
    """Integer split of `total` proportional to weights (Hamilton's method),
    each part at least `minimum`; ties go to the lower index."""
    w = np.asarray(weights, np.float64)
    k = len(w)
    free = total - minimum * k
    quota = free * w / w.sum()
    base = np.floor(quota).astype(np.int64)
    rem = quota - base
    left = free - int(base.sum())
    order = sorted(range(k), key=lambda i: (-rem[i], i))
    for i in order[:left]:
        base[i] += 1
    return [int(x) + minimum for x in base]


def spans_to_labels(spans: Sequence[int]) -> np.ndarray:
    return np.concatenate([np.full(s, r, np.uint8) for r, s in enumerate(spans) if s > 0])


def _turn_blocks(rng: np.random.Generator, total: int, lo: int, hi: int, labels_fn):
    """512-token pinned system span, then turn blocks of U{lo..hi} tokens until
    `total` tokens (the last block truncated).  Returns labels and per-token
    insertion steps: block j of nb gets insert step -(nb - j) * 16, a turn every
    16 decode steps before the trace's end."""
    blocks = [(SYSTEM, 512)]
    used = 512
    j = 0
    while used < total:
        ln = int(rng.integers(lo, hi + 1))
        ln = min(ln, total - used)
        blocks.append((labels_fn(j), ln))
        used += ln
        j += 1
    nb = len(blocks)
    lab = np.concatenate([np.full(n, r, np.uint8) for r, n in blocks])
    ins = np.concatenate([np.full(n, -(nb - i) * 16, np.int32) for i, (_, n) in enumerate(blocks)])
    return lab, ins


def make_workload(config: int, seed: int = 0, **overrides) -> Workload:
    """The five workload configurations (0-4)."""
    rng = np.random.default_rng(np.random.SeedSequence([seed, 7919, config]))
    if config == 0:
        lab = spans_to_labels(CONFIG0_SPANS)
        w = Workload("config0: 1 layer, 12/2 heads, 448-token trace", 1, 12, 2, 16,
                     [lab], [np.zeros(len(lab), np.int32)], [14], 64, seed=seed)
    elif config == 1:
        spans = largest_remainder(1700, CONFIG0_SPANS)
        lab = spans_to_labels(spans)
        w = Workload("config1: Qwen2.5-1.5B geometry (28 layers, 12/2), 1,700-token trace", 28, 12, 2, 16,
                     [lab], [np.zeros(len(lab), np.int32)], [26], 256, seed=seed)
    elif config == 2:
        regs, ins = [], []
        for b in range(32):
            g = rng.gamma(2.0, 1.0, size=7)
            spans = largest_remainder(1700, g / g.sum(), minimum=1)
            regs.append(spans_to_labels(spans))
            off = int(rng.integers(0, 256))
            ins.append(np.full(1700, -off, np.int32))
        w = Workload("config2: Qwen2.5-3B geometry (36 layers, 16/2), B=32 x 1,700 tokens", 36, 16, 2, 16,
                     regs, ins, [26] * 32, 256, seed=seed)
    elif config == 3:
        regs, ins = [], []
        cycle = (PLAN, USER, TOOL_IN, TOOL_OUT, RETRIEVAL, SCRATCHPAD)
        for b in range(64):
            lab, st = _turn_blocks(rng, 32768, 64, 2048, lambda j: cycle[j % 6])
            regs.append(lab)
            ins.append(st)
        w = Workload("config3: Qwen2.5-3B geometry, B=64 x 32,768-token agent traces", 36, 16, 2, 16,
                     regs, ins, [204] * 64, 256, window_k=16, seed=seed)
    elif config == 4:
        regs, ins = [], []
        for b in range(16):
            draws = rng.integers(1, 7, size=4096)
            lab, st = _turn_blocks(rng, 131072, 64, 589, lambda j, dr=draws: int(dr[j]))
            regs.append(lab)
            ins.append(st)
        w = Workload("config4: Qwen2.5-3B geometry, B=16 x 131,072-token traces (stress)", 36, 16, 2, 32,
                     regs, ins, [204] * 16, 64, seed=seed)
    else:
        raise ValueError(f"unknown config {config}")
    return replace(w, **overrides) if overrides else w


def custom_workload(name: str, L: int, Hq: int, Hkv: int, page_size: int, lengths: Sequence[int],
                    budget_frac: float, steps: int, seed: int = 0, spans_seed: int = 1,
                    **kw) -> Workload:
    """A small trace family for parity tests: per sequence, seven contiguous
    region spans with seeded Dirichlet(2) proportions (each >= 1 token)."""
    rng = np.random.default_rng(np.random.SeedSequence([spans_seed, len(lengths), int(1e6 * budget_frac)]))
    regs, ins = [], []
    for n in lengths:
        g = rng.gamma(2.0, 1.0, size=7)
        regs.append(spans_to_labels(largest_remainder(int(n), g / g.sum(), minimum=1)) if n >= 7
                    else np.asarray(rng.integers(0, 7, size=n), np.uint8))
        ins.append(np.zeros(int(n), np.int32))
    pages = [-(-int(n) // page_size) for n in lengths]
    budgets = [max(1, int(math.floor(budget_frac * p))) for p in pages]
    return Workload(name, L, Hq, Hkv, page_size, regs, ins, budgets, steps, seed=seed, **kw)


def straddle_fraction(labels: np.ndarray, page_size: int) -> float:
    """Fraction of pages that hold tokens of more than one region (the
    statistic the paper reports in Sec. III-D)."""
    n = len(labels)
    pages = -(-n // page_size)
    mixed = 0
    for p in range(pages):
        seg = labels[p * page_size:(p + 1) * page_size]
        mixed += int(len(np.unique(seg)) > 1)
    return mixed / max(1, pages)
