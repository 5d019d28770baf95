"""fp64 CPU oracle of MemDecay's decode-time eviction loop.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and
``bench.py``'s cpu_baseline / reference legs may import this module.  The
product path (the CUDA library and its binding) never calls it, and it shares
no code with that path: inputs come from the ``synth`` generator module or
from the tests themselves.

It restates the paper's definitions as plainly as possible, in float64, one
sequence / layer / head at a time:

* paged KV cache with a block table per sequence and a LIFO free stack of
  physical page ids (Sec. III-D: fixed-size pages as in vLLM);
* decode attention over every cached token, softmax weights p (Sec. III-C);
* the observed attention mass Abar_i: the mass token i received, averaged over
  query heads, layers and the observation window (Sec. III-C);
* attention EWMA a_i <- rho*a_i + gamma*Abar_i (Eq. 2; the paper's gamma = 1-rho);
* decay-clock refresh t_ref <- t when Abar_i >= tau, tau = c/|K_t| (Eq. 3);
* retention score s_i = b_r exp(-lambda_r dt) + alpha a_i (Eq. 4), with
  lambda_r = ln2 / half-life (Eq. 7); or, score_mode 1, the multiplicative
  form (b_r + alpha a_i) exp(-lambda_r dt); pinned regions score +inf;
* page score S_p = mean of member scores (Eq. 5), or their max (page_reduce 1);
* Algorithm 1: when |K_t| exceeds the budget, evict non-pinned pages in
  ascending S_p, using a min-heap (the paper's own selection procedure).

Readings where the paper is silent (each one is also a line of the design
notes): budgets are counted in pages, resident pages include the partial tail
page, the tail page (the one being written) is protected, ties are broken by
ascending logical page index, when pins exceed the budget all evictable pages
go and a warning status is returned, freed physical ids are pushed in
(sequence, logical page) order, a page holding any pinned token is pinned, the
eviction and refresh decisions are taken on fp32-rounded values (the kernel's
precision), and the refresh comparison is ">=".
"""
from __future__ import annotations

import heapq
import math
from dataclasses import dataclass
from typing import Dict, List, Optional, Sequence, Tuple

import numpy as np

NUM_REGIONS = 7
MD_OK = 0
MD_WARN_OVER_BUDGET = 1


# ------------------------------------------------------------ definitions ---
def bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    """bf16 bit patterns -> exact float64 values."""
    u = np.asarray(bits, np.uint16).astype(np.uint32) << np.uint32(16)
    return u.view(np.float32).astype(np.float64)


def attention_group(q: np.ndarray, K: np.ndarray, V: np.ndarray) -> Tuple[np.ndarray, np.ndarray]:
    """Scaled dot-product decode attention of the G query heads that share one
    KV head, over all n cached tokens (Sec. III-C; decoding attends to every
    cached token, so there is no mask).

    q: [G][D], K: [n][D], V: [n][D] (float64).  Returns o [G][D] and the
    softmax weights p [G][n] (each row sums to 1)."""
    D = q.shape[1]
    s = (q @ K.T) / math.sqrt(D)              # s[h, i] = q_h . k_i / sqrt(D)
    m = s.max(axis=1, keepdims=True)
    e = np.exp(s - m)
    p = e / e.sum(axis=1, keepdims=True)
    o = p @ V
    return o, p


def observed_mass(W: np.ndarray, window_steps: int, L: int, Hq: int) -> np.ndarray:
    """Abar_i (Sec. III-C): W_i is the sum over decode steps of the window,
    layers and query heads of the softmax weight token i received; averaging
    over heads, layers and window divides by window_steps * L * Hq.  A token
    inserted inside the window contributes nothing before it exists."""
    return W / float(window_steps * L * Hq)


def ewma(a: np.ndarray, abar: np.ndarray, rho: float, gamma: float) -> np.ndarray:
    """Eq. 2: a_i <- rho a_i + (1 - rho) Abar_i; gamma generalises (1 - rho)."""
    return rho * a + gamma * abar


def refresh(t_ref: np.ndarray, abar: np.ndarray, tau: float, t: int) -> np.ndarray:
    """Eq. 3: the decay clock restarts at the observation step t when
    Abar_i >= tau.  The comparison is made on fp32-rounded values."""
    hit = np.float32(abar) >= np.float32(tau) if np.isscalar(abar) else \
        np.asarray(abar, np.float32) >= np.float32(tau)
    return np.where(hit, t, t_ref)


def decay(dt: np.ndarray, half_life: np.ndarray) -> np.ndarray:
    """exp(-lambda_r dt) with lambda_r = ln 2 / t_half (Eqs. 4 and 7), written
    as 2^(-dt / t_half) so that one half-life gives exactly 1/2.  An infinite
    half-life is lambda = 0 (no decay)."""
    dt = np.asarray(dt, np.float64)
    h = np.asarray(half_life, np.float64)
    return np.power(2.0, -(dt / h))


def token_score(base: np.ndarray, d: np.ndarray, a: np.ndarray, alpha: float, mode: int,
                n_cached: int = 1, t_ins: np.ndarray = None, noise: np.ndarray = None) -> np.ndarray:
    """Retention score of each token.
    mode 0: Eq. 4, s_i = b_r d_i + alpha a_i (the paper's additive form);
    mode 1: the multiplicative reading (b_r + alpha a_i) d_i;
    mode 2: Eq. 4 with the attention term normalised to the uniform level
            1/|K_t| (the design change of Sec. IV-D / Sec. V): b_r d_i + alpha a_i |K_t|;
    mode 3: recency (the streaming baseline of Sec. IV-C): newer tokens score
            higher, s_i = t_ins_i;
    mode 4: a uniform random draw per token and observation (the random
            baseline of Sec. IV-C)."""
    if mode == 0:
        return base * d + alpha * a
    if mode == 1:
        return (base + alpha * a) * d
    if mode == 2:
        return base * d + alpha * a * float(n_cached)
    if mode == 3:
        return np.asarray(t_ins, np.float64)
    return np.asarray(noise, np.float64)


def random_draw(seed: int, t: int, slot: np.ndarray) -> np.ndarray:
    """Uniform draws in [0, 1) for the random baseline: the SplitMix64
    finaliser (Steele, Lea, Flood 2014) of (seed, step, physical slot), top 24
    bits scaled by 2^-24 (exact in fp32)."""
    M = (1 << 64) - 1
    out = np.empty(len(slot))
    for i, sl in enumerate(np.asarray(slot, np.int64)):
        x = ((seed * 0x9E3779B97F4A7C15) ^ (int(t) << 40) ^ int(sl)) & M
        z = (x + 0x9E3779B97F4A7C15) & M
        z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & M
        z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & M
        z = z ^ (z >> 31)
        out[i] = (z >> 40) * 2.0 ** -24
    return out


def page_score(member_scores: np.ndarray, reduce_mode: int) -> float:
    """Eq. 5: S_p = (1/|p|) sum_{i in p} s_i over the page's tokens
    (reduce_mode 1: the max instead)."""
    if reduce_mode == 0:
        return float(np.sum(member_scores) / len(member_scores))
    return float(np.max(member_scores))


def select_pages_min_heap(S32: Sequence[float], evictable: Sequence[bool], n_evict: int) -> List[int]:
    """Algorithm 1: build a min-heap over the non-pinned (evictable) pages
    keyed by S_p and pop the minimum until n_evict pages are gone.  Keys are
    (S_p, logical page index): equal scores evict the older page first."""
    heap = [(float(S32[p]), p) for p in range(len(S32)) if evictable[p]]
    heapq.heapify(heap)
    out = []
    while len(out) < n_evict and heap:
        out.append(heapq.heappop(heap)[1])
    return sorted(out)


CALIB_BUCKET_WIDTH = 4      # Fig. 3: age buckets of 4 decode steps
CALIB_BUCKETS = 256         # ages 0 .. 1023 steps


def age_bucket(age: int, width: int = CALIB_BUCKET_WIDTH) -> int:
    """Age bucket of a token of age `age` (decode steps since insertion)."""
    return int(age) // width


def wls_log_linear_fit(ages: np.ndarray, mean_mass: np.ndarray, weights: np.ndarray):
    """Eq. 6: fit log Abar_r(dt) ~ log c_r - lambda_r dt by weighted least
    squares, weights = observation counts (the count-weighted fit of
    Sec. IV-B).  Normal equations of min sum w (y - a - b x)^2 with
    x = age, y = log mean mass.  Returns (lambda_hat, log c_hat)."""
    x = np.asarray(ages, np.float64)
    y = np.log(np.asarray(mean_mass, np.float64))
    w = np.asarray(weights, np.float64)
    W, Sx, Sy = w.sum(), (w * x).sum(), (w * y).sum()
    Sxx, Sxy = (w * x * x).sum(), (w * x * y).sum()
    slope = (W * Sxy - Sx * Sy) / (W * Sxx - Sx * Sx)
    intercept = (Sy - slope * Sx) / W
    return -slope, intercept


def half_life(rate: float) -> float:
    """Eq. 7: t_half = ln 2 / lambda."""
    return math.log(2.0) / rate if rate > 0 else math.inf


def calibrate(mass_sum: np.ndarray, count: np.ndarray, width: int = CALIB_BUCKET_WIDTH,
              min_count: int = 1):
    """Per region: the mean attention mass of each age bucket (bucket centre
    age width*b + width/2, as Fig. 3 plots), then the Eq. 6 fit over the
    buckets with at least min_count observations and a positive mean.
    Returns (lambda_hat[r], half_life[r]); NaN where fewer than two buckets."""
    R, NB = mass_sum.shape
    rates = np.full(R, np.nan)
    halves = np.full(R, np.nan)
    for r in range(R):
        ok = (count[r] >= max(1, min_count)) & (mass_sum[r] > 0)
        if ok.sum() < 2:
            continue
        b = np.nonzero(ok)[0]
        ages = width * b + width / 2.0
        lam, _ = wls_log_linear_fit(ages, mass_sum[r, b] / count[r, b], count[r, b])
        rates[r] = lam
        halves[r] = half_life(lam)
    return rates, halves


# ------------------------------------------------------------------ state ---
@dataclass
class OracleConfig:
    num_layers: int
    num_q_heads: int
    num_kv_heads: int
    head_dim: int
    page_size: int
    max_batch: int
    max_pages_per_seq: int
    num_phys_pages: int
    rho: float = 0.9
    gamma: float = 0.1
    tau_scale: float = 2.0
    attn_weight: float = 1.0
    score_mode: int = 0
    page_reduce: int = 0
    random_seed: int = 0
    region_aligned: bool = False


class Oracle:
    """The paged cache and the MemDecay state of a batch of sequences, with
    the same calls as the library: append_tokens, decode_step, evict."""

    def __init__(self, cfg: OracleConfig):
        self.cfg = cfg
        ps = cfg.page_size
        self.t = 0
        self.window_steps = 0
        # LIFO free stack of physical page ids; the first pop returns 0.
        self.free: List[int] = list(range(cfg.num_phys_pages - 1, -1, -1))
        self.block: List[List[int]] = [[] for _ in range(cfg.max_batch)]
        self.fill: List[List[int]] = [[] for _ in range(cfg.max_batch)]   # tokens per page
        self.tail_region = [-1] * cfg.max_batch
        self.n_tokens = [0] * cfg.max_batch
        nslots = cfg.num_phys_pages * ps
        self.region = np.zeros(nslots, np.uint8)
        self.a = np.zeros(nslots, np.float64)
        self.t_ref = np.zeros(nslots, np.int64)
        self.W = np.zeros(nslots, np.float64)
        self.abar = np.zeros(nslots, np.float64)
        self.prio = np.zeros(nslots, np.float64)
        self.page_S: List[np.ndarray] = [np.zeros(0) for _ in range(cfg.max_batch)]
        self.pool: Dict[int, Tuple[np.ndarray, np.ndarray]] = {}
        self.base = np.zeros(NUM_REGIONS)
        self.half_life = np.full(NUM_REGIONS, np.inf)
        self.pinned = np.zeros(NUM_REGIONS, bool)
        # calibration (Sec. IV-B): insertion step per slot, histogram of the
        # observed mass by (region, age bucket)
        self.t_ins = np.zeros(nslots, np.int64)
        self.calib_on = False
        self.calib_sum = np.zeros((NUM_REGIONS, CALIB_BUCKETS))
        self.calib_cnt = np.zeros((NUM_REGIONS, CALIB_BUCKETS), np.int64)

    def calib_enable(self, on: bool = True) -> None:
        """Start (and clear) or stop gathering the calibration histogram."""
        self.calib_on = bool(on)
        self.calib_sum[:] = 0.0
        self.calib_cnt[:] = 0

    # -- configuration (Table 1: base priority, decay rate, pinned flag) --
    def set_region_params(self, r: int, base: float, half_life: float, pinned: bool) -> None:
        self.base[r] = base
        self.half_life[r] = half_life
        self.pinned[r] = bool(pinned)

    # -- paging --
    def _page(self, phys: int):
        if phys not in self.pool:
            c = self.cfg
            shape = (c.num_layers, c.num_kv_heads, c.page_size, c.head_dim)
            self.pool[phys] = (np.zeros(shape, np.uint16), np.zeros(shape, np.uint16))
        return self.pool[phys]

    def _append_one(self, b: int, region: int, k: np.ndarray, v: np.ndarray, insert_step: int) -> None:
        """Append one token (Fig. 1 "append KV"): region label r(i), insertion
        step t_ins, clock t_ref = t_ins, importance a = 0.  A full (or absent)
        tail page takes a fresh physical page from the free stack; with
        region-aligned allocation (the variant Sec. III-D leaves to future
        work) a token whose region differs from the tail page's also opens a
        fresh page, so no page straddles a region boundary."""
        ps = self.cfg.page_size
        fills = self.fill[b]
        if not fills or fills[-1] == ps or (self.cfg.region_aligned and self.tail_region[b] != region):
            if len(self.block[b]) >= self.cfg.max_pages_per_seq or not self.free:
                raise RuntimeError("capacity")
            self.block[b].append(self.free.pop())
            fills.append(0)
        off = fills[-1]
        fills[-1] += 1
        self.tail_region[b] = region
        phys = self.block[b][-1]
        kp, vp = self._page(phys)
        kp[:, :, off, :] = k
        vp[:, :, off, :] = v
        slot = phys * ps + off
        self.region[slot] = region
        self.t_ref[slot] = insert_step
        self.t_ins[slot] = insert_step
        self.a[slot] = 0.0
        self.W[slot] = 0.0
        self.abar[slot] = 0.0
        self.prio[slot] = 0.0
        self.n_tokens[b] += 1

    def append_tokens(self, b: int, regions: np.ndarray, K: np.ndarray, V: np.ndarray,
                      insert_step=None) -> None:
        """Prefill: K, V are bf16 bits [L][Hkv][n][D]; regions [n]; insert_step
        an int, one int per token, or None (the current step)."""
        n = len(regions)
        if insert_step is None:
            steps = np.full(n, self.t, np.int64)
        else:
            steps = np.broadcast_to(np.asarray(insert_step, np.int64), (n,))
        if n and steps.max() > self.t:
            raise ValueError("insert_step after the current step")
        for i in range(n):
            self._append_one(b, int(regions[i]), K[:, :, i, :], V[:, :, i, :], int(steps[i]))

    def slots(self, b: int) -> np.ndarray:
        """Physical slots of sequence b's tokens in logical order."""
        ps = self.cfg.page_size
        return np.array([phys * ps + o for phys, f in zip(self.block[b], self.fill[b]) for o in range(f)],
                        np.int64)

    def page_of_token(self, b: int) -> np.ndarray:
        """Logical page index of each of sequence b's tokens (logical order)."""
        return np.repeat(np.arange(len(self.fill[b])), self.fill[b])

    def _gather(self, b: int, l: int, h: int) -> Tuple[np.ndarray, np.ndarray]:
        ks, vs = [], []
        for phys, cnt in zip(self.block[b], self.fill[b]):
            kp, vp = self.pool[phys]
            ks.append(kp[l, h, :cnt])
            vs.append(vp[l, h, :cnt])
        return bf16_bits_to_f64(np.concatenate(ks)), bf16_bits_to_f64(np.concatenate(vs))

    # -- one decode step --
    def decode_step(self, batch: int, Q: np.ndarray, K_new: np.ndarray, V_new: np.ndarray,
                    new_regions: Sequence[int]) -> np.ndarray:
        """Advance t, append each sequence's new token (t_ins = t), then attend
        over every cached token (new one included) in every layer and head,
        accumulating the attention mass of the observation window.

        Q: bf16 bits [B][L][Hq][D]; K_new, V_new: [B][L][Hkv][D].
        Returns the attention output o, float64 [B][L][Hq][D]."""
        c = self.cfg
        G = c.num_q_heads // c.num_kv_heads
        self.t += 1
        for b in range(batch):
            self._append_one(b, int(new_regions[b]), K_new[b], V_new[b], self.t)
        O = np.zeros((batch, c.num_layers, c.num_q_heads, c.head_dim))
        for b in range(batch):
            sl = self.slots(b)
            mass = np.zeros(len(sl))
            for l in range(c.num_layers):
                for h in range(c.num_kv_heads):
                    K, V = self._gather(b, l, h)
                    q = bf16_bits_to_f64(Q[b, l, h * G:(h + 1) * G])
                    o, p = attention_group(q, K, V)
                    O[b, l, h * G:(h + 1) * G] = o
                    mass += p.sum(axis=0)
            self.W[sl] += mass
        self.window_steps += 1
        return O

    # -- one observation step (Algorithm 1) --
    def observe_and_score(self, b: int, observe: bool) -> np.ndarray:
        """Algorithm 1 up to the page scores, for sequence b: EWMA (Eq. 2),
        refresh (Eq. 3), token scores (Eq. 4), page scores (Eq. 5).
        Returns S_p in float64 (pinned and protected pages +inf)."""
        c = self.cfg
        ps = c.page_size
        sl = self.slots(b)
        n = len(sl)
        reg = self.region[sl]
        if observe:
            abar = observed_mass(self.W[sl], self.window_steps, c.num_layers, c.num_q_heads)
            self.abar[sl] = abar
            self.a[sl] = ewma(self.a[sl], abar, c.rho, c.gamma)
            tau = c.tau_scale / n
            self.t_ref[sl] = refresh(self.t_ref[sl], abar, tau, self.t)
            self.W[sl] = 0.0
            if self.calib_on:
                for i, slot in enumerate(sl):
                    bkt = age_bucket(self.t - self.t_ins[slot])
                    if 0 <= bkt < CALIB_BUCKETS:
                        self.calib_sum[reg[i], bkt] += abar[i]
                        self.calib_cnt[reg[i], bkt] += 1
        d = decay(self.t - self.t_ref[sl], self.half_life[reg])
        noise = random_draw(c.random_seed, self.t, sl) if c.score_mode == 4 else None
        s = token_score(self.base[reg], d, self.a[sl], c.attn_weight, c.score_mode, n,
                        self.t_ins[sl], noise)
        pinned_tok = self.pinned[reg]
        s = np.where(pinned_tok, np.inf, s)
        self.prio[sl] = s
        P = len(self.block[b])
        S = np.zeros(P)
        bounds = np.concatenate([[0], np.cumsum(self.fill[b])])
        for j in range(P):
            lo, hi = bounds[j], bounds[j + 1]
            if pinned_tok[lo:hi].any() or j == P - 1:      # pinning / protected tail
                S[j] = np.inf
            else:
                S[j] = page_score(s[lo:hi], c.page_reduce)
        self.page_S[b] = S
        return S

    def evict(self, batch: int, budget_pages: Sequence[int]):
        """The observation step: score every sequence, then, where the number
        of resident pages exceeds the budget, evict the lowest-S_p evictable
        pages (Algorithm 1), compact the block table in order and push the
        freed physical ids on the free stack in (sequence, logical) order.

        Returns (status, n_evicted[B], evicted physical ids per sequence,
        evicted logical indices per sequence)."""
        observe = self.window_steps > 0
        status = MD_OK
        n_ev, ids, logical = [], [], []
        for b in range(batch):
            S = self.observe_and_score(b, observe)
            P = len(S)
            want = max(0, P - int(budget_pages[b]))
            S32 = np.asarray(S, np.float32)
            evictable = [bool(np.isfinite(S[j])) for j in range(P)]
            if sum(evictable) < want:
                status = MD_WARN_OVER_BUDGET
            out = select_pages_min_heap(S32, evictable, want)
            gone = set(out)
            freed = [self.block[b][j] for j in out]
            self.n_tokens[b] -= sum(self.fill[b][j] for j in out)
            self.block[b] = [self.block[b][j] for j in range(P) if j not in gone]
            self.fill[b] = [self.fill[b][j] for j in range(P) if j not in gone]
            n_ev.append(len(out))
            ids.append(freed)
            logical.append(out)
        for b in range(batch):
            self.free.extend(ids[b])
        self.window_steps = 0
        return status, n_ev, ids, logical
