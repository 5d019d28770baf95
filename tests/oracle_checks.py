"""Pins of the fp64 oracle against facts that do not come from the oracle:
closed forms, the paper's worked example (Fig. 2), invariants stated in the
paper, and brute force on tiny inputs.

Each check takes the oracle module as an argument, so that the mutation test
can run every check against an oracle with a planted mistake and show that
one of them fails.  Checks raise AssertionError."""
from __future__ import annotations

import itertools
import math
import os

import numpy as np

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
REGION_IDS = {"system": 0, "plan": 1, "user": 2, "tool_in": 3, "tool_out": 4,
              "retrieval": 5, "scratchpad": 6}


def read_golden(name):
    rows = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                rows.append(line.split())
    return rows


def f32_bits_to_bf16_bits(x):
    """bf16 (round to nearest even) bit patterns of float values."""
    u = np.asarray(x, np.float32).view(np.uint32).astype(np.uint64)
    u = u + np.uint64(0x7FFF) + ((u >> np.uint64(16)) & np.uint64(1))
    return ((u >> np.uint64(16)) & np.uint64(0xFFFF)).astype(np.uint16)


def make(om, L=1, Hq=1, Hkv=1, D=16, ps=4, B=1, phys=64, max_pages=64, **kw):
    cfg = om.OracleConfig(num_layers=L, num_q_heads=Hq, num_kv_heads=Hkv, head_dim=D,
                          page_size=ps, max_batch=B, max_pages_per_seq=max_pages,
                          num_phys_pages=phys, **kw)
    o = om.Oracle(cfg)
    for r in range(7):
        o.set_region_params(r, 0.5, 30.0, False)
    return o


def zeros_kv(L, Hkv, n, D):
    return np.zeros((L, Hkv, n, D), np.uint16), np.zeros((L, Hkv, n, D), np.uint16)


# ------------------------------------------------------------------ decay ---
def check_decay_closed_forms(om):
    """exp(-lambda dt) with lambda = ln2 / t_half (Eq. 7): exactly 1/2 after one
    half-life, 1/4 after two, 1 at age 0 and with an infinite half-life; and the
    same numbers as the paper's exp(-lambda dt) form of Eq. 4."""
    rows = read_golden("table2_half_lives.txt")
    hs = sorted({float(x) for r in rows for x in r[1:]}) + [0.5, 1.0, 3.7, 1e6]
    for h in hs:
        assert om.decay(h, h) == 0.5, h
        assert om.decay(2 * h, h) == 0.25, h
        assert om.decay(0, h) == 1.0, h
    assert om.decay(12345, np.inf) == 1.0
    rng = np.random.default_rng(1)
    dt = rng.integers(0, 500, 200)
    h = rng.uniform(1.0, 200.0, 200)
    lam = math.log(2.0) / h
    np.testing.assert_allclose(om.decay(dt, h), np.exp(-lam * dt), rtol=1e-12)


def check_fig2_trajectories(om):
    """The paper's worked example (Fig. 2): with the attention term off, a token
    of region r scores b_r exp(-lambda_r age); the tool_out curve's clock
    restarts at age 40 when the token is attended above tau.  Run through the
    whole state machine: prefill, decode steps, observation steps."""
    for name, b, lam, ref_age in read_golden("fig2_decay.txt"):
        b, lam, ref_age = float(b), float(lam), int(ref_age)
        r = REGION_IDS[name]
        D = 16
        o = make(om, D=D, ps=4, phys=64, attn_weight=0.0)
        for rr in range(7):
            o.set_region_params(rr, 0.1, 10.0, False)
        o.set_region_params(r, b, math.log(2.0) / lam, False)
        n0 = 12
        K, V = zeros_kv(1, 1, n0, D)
        K[0, 0, 0, 0] = f32_bits_to_bf16_bits(1.0)          # tracked token: key e_0
        regions = np.full(n0, 6, np.uint8)
        regions[0] = r
        o.append_tokens(0, regions, K, V, insert_step=0)
        slot0 = o.slots(0)[0]
        for t in range(1, 101):
            q = np.zeros((1, 1, 1, D), np.uint16)
            if t == ref_age:
                q[0, 0, 0, 0] = f32_bits_to_bf16_bits(64.0)    # attend to the tracked token
            kn, vn = np.zeros((1, 1, 1, D), np.uint16), np.zeros((1, 1, 1, D), np.uint16)
            o.decode_step(1, q, kn, vn, [6])
            a_before = o.a[slot0]
            o.evict(1, [10 ** 6])
            age = t if (ref_age < 0 or t < ref_age) else t - ref_age
            want = b * math.exp(-lam * age)
            got = o.prio[slot0]
            assert abs(got - want) <= 1e-12 * want, (name, t, got, want)
            if t == ref_age:
                assert o.t_ref[slot0] == t
                # a refresh resets the clock and nothing else: a follows Eq. 2
                assert o.a[slot0] == 0.9 * a_before + 0.1 * o.abar[slot0]


# ------------------------------------------------------------------- EWMA ---
def check_ewma_closed_form(om):
    """Uniform attention (all keys equal) gives every token Abar = 1/|K_t| at
    each observation; iterating Eq. 2 from a = 0 gives the closed form
    a_T = sum_j rho^(T-j) (1-rho) / |K_j|."""
    L, Hq, Hkv, D, n0, T = 2, 4, 2, 16, 10, 12
    rho = 0.9
    o = make(om, L=L, Hq=Hq, Hkv=Hkv, D=D, ps=4, phys=64, rho=rho, gamma=1 - rho)
    K, V = zeros_kv(L, Hkv, n0, D)
    rng = np.random.default_rng(3)
    V[...] = f32_bits_to_bf16_bits(rng.standard_normal(V.shape))
    o.append_tokens(0, np.full(n0, 2, np.uint8), K, V, insert_step=0)
    slot0 = o.slots(0)[0]
    for t in range(1, T + 1):
        q = f32_bits_to_bf16_bits(rng.standard_normal((1, L, Hq, D)))
        kn = np.zeros((1, L, Hkv, D), np.uint16)
        o.decode_step(1, q, kn, kn.copy(), [6])
        o.evict(1, [10 ** 6])
    want = sum(rho ** (T - j) * (1 - rho) / (n0 + j) for j in range(1, T + 1))
    assert abs(o.a[slot0] - want) <= 1e-13 * want, (o.a[slot0], want)


# -------------------------------------------------------------- attention ---
def check_attention_closed_form(om):
    """Orthogonal keys and queries: s_{h,i} = x_h y_i [h == i] / sqrt(D), so
    p_{h,h} = e^s / (e^s + n - 1) and p_{h,i} = 1 / (e^s + n - 1) otherwise;
    one-hot values make o_h read back p_h.  A single cached token gives o = v
    exactly; identical keys give p = 1/n exactly."""
    G, n, D = 3, 4, 16
    x = np.array([1.5, -2.0, 3.0])
    y = np.array([2.0, 1.0, 0.5, 7.0])
    q = np.zeros((G, D))
    K = np.zeros((n, D))
    V = np.zeros((n, D))
    for h in range(G):
        q[h, h] = x[h]
    for i in range(n):
        K[i, i] = y[i]
        V[i, 8 + i] = 1.0
    o, p = om.attention_group(q, K, V)
    for h in range(G):
        s = x[h] * y[h] / math.sqrt(D)
        z = math.exp(s) + n - 1
        for i in range(n):
            want = (math.exp(s) if i == h else 1.0) / z
            assert abs(p[h, i] - want) < 1e-14, (h, i, p[h, i], want)
            assert abs(o[h, 8 + i] - want) < 1e-14
    rng = np.random.default_rng(5)
    v1 = rng.standard_normal((1, D))
    o1, p1 = om.attention_group(rng.standard_normal((2, D)), rng.standard_normal((1, D)), v1)
    assert np.array_equal(o1, np.repeat(v1, 2, axis=0)) and np.all(p1 == 1.0)
    Kc = np.repeat(rng.standard_normal((1, D)), 7, axis=0)
    _, pc = om.attention_group(rng.standard_normal((3, D)), Kc, rng.standard_normal((7, D)))
    assert np.all(pc == 1.0 / 7)


def check_mass_sums_to_one(om):
    """Each head's softmax sums to 1, so the observed mass Abar (averaged over
    query heads and layers, window of one step) sums to 1 over a sequence's
    tokens (Sec. III-C)."""
    L, Hq, Hkv, D, ps = 3, 6, 2, 16, 4
    rng = np.random.default_rng(7)
    o = make(om, L=L, Hq=Hq, Hkv=Hkv, D=D, ps=ps, B=2, phys=64)
    for b, n in enumerate((9, 14)):
        K = f32_bits_to_bf16_bits(rng.standard_normal((L, Hkv, n, D)))
        V = f32_bits_to_bf16_bits(rng.standard_normal((L, Hkv, n, D)))
        o.append_tokens(b, rng.integers(1, 7, n).astype(np.uint8), K, V, 0)
    q = f32_bits_to_bf16_bits(rng.standard_normal((2, L, Hq, D)))
    kn = f32_bits_to_bf16_bits(rng.standard_normal((2, L, Hkv, D)))
    o.decode_step(2, q, kn, kn.copy(), [6, 6])
    o.evict(2, [10 ** 6, 10 ** 6])
    for b in range(2):
        tot = o.abar[o.slots(b)].sum()
        assert abs(tot - 1.0) < 1e-12, (b, tot)


def check_gqa_mapping(om):
    """Query head h reads KV head h // G (G = Hq / Hkv): with uniform keys on KV
    head 0 and one strongly matching key on KV head 1, heads 0..G-1 return the
    mean of KV head 0's values and heads G..2G-1 the softmax-weighted values of
    KV head 1 in closed form."""
    L, Hq, Hkv, D, n = 1, 4, 2, 16, 5
    o = make(om, L=L, Hq=Hq, Hkv=Hkv, D=D, ps=8, phys=16)
    rng = np.random.default_rng(11)
    K, V = zeros_kv(L, Hkv, n, D)
    K[0, 1, 2, 0] = f32_bits_to_bf16_bits(4.0)
    V[...] = f32_bits_to_bf16_bits(rng.standard_normal(V.shape))
    o.append_tokens(0, np.full(n, 2, np.uint8), K, V, 0)
    q = np.zeros((1, L, Hq, D), np.uint16)
    q[0, 0, :, 0] = f32_bits_to_bf16_bits(4.0)
    kn = np.zeros((1, L, Hkv, D), np.uint16)
    vn = np.zeros((1, L, Hkv, D), np.uint16)
    out = o.decode_step(1, q, kn, vn, [6])
    Vf = om.bf16_bits_to_f64(V[0])
    Vall0 = np.vstack([Vf[0], np.zeros((1, D))])
    Vall1 = np.vstack([Vf[1], np.zeros((1, D))])
    e = math.exp(16.0 / math.sqrt(D))
    p1 = np.full(n + 1, 1.0 / (e + n))
    p1[2] = e / (e + n)
    for h in range(2):
        np.testing.assert_allclose(out[0, 0, h], Vall0.mean(axis=0), atol=1e-14)
    for h in range(2, 4):
        np.testing.assert_allclose(out[0, 0, h], p1 @ Vall1, atol=1e-13)


# --------------------------------------------------------- refresh / tau ---
def check_refresh_threshold(om):
    """tau = c / |K_t| with |K_t| counting the token appended at this step, and
    the refresh condition Abar >= tau (Eq. 3): with identical keys every token
    gets exactly Abar = 1/|K_t|, so c = 1 refreshes every clock, c = 2 none and
    c = 1 + 1e-6 none.  A refreshed token scores b + alpha a (dt = 0)."""
    for c, expect in ((1.0, True), (2.0, False), (1.0 + 1e-6, False)):
        o = make(om, L=1, Hq=2, Hkv=1, D=16, ps=4, phys=32, tau_scale=c, attn_weight=0.75)
        n0 = 9
        K, V = zeros_kv(1, 1, n0, 16)
        o.append_tokens(0, np.full(n0, 3, np.uint8), K, V, insert_step=-5)
        rng = np.random.default_rng(2)
        q = f32_bits_to_bf16_bits(rng.standard_normal((1, 1, 2, 16)))
        o.decode_step(1, q, np.zeros((1, 1, 1, 16), np.uint16), np.zeros((1, 1, 1, 16), np.uint16), [3])
        o.evict(1, [10 ** 6])
        sl = o.slots(0)
        assert np.all(o.abar[sl] == 1.0 / (n0 + 1))
        refreshed = o.t_ref[sl[:n0]] == 1
        assert bool(refreshed.all()) == expect and bool(refreshed.any()) == expect, c
        if expect:
            a = o.a[sl[0]]
            assert abs(a - 0.1 / (n0 + 1)) < 1e-16
            assert o.prio[sl[0]] == 0.5 + 0.75 * a


# ------------------------------------------------------------ page scores ---
def check_page_scores(om):
    """Hand-computed example (Eq. 5 and the pinning rule): page size 4, one
    step after insertion, half-life 1 step (decay exactly 1/2), attention term
    off.  plan b = 0.75 -> s = 0.375; user b = 0.25 -> s = 0.125.
    page 0 [plan x4] = 0.375; page 1 [plan x2, user x2] = 0.25 (max 0.375);
    page 2 holds a pinned system token -> +inf; page 3 is the tail -> +inf."""
    for mode, want1 in ((0, 0.25), (1, 0.375)):
        o = make(om, L=1, Hq=1, Hkv=1, D=16, ps=4, phys=32, attn_weight=0.0, page_reduce=mode)
        o.set_region_params(1, 0.75, 1.0, False)
        o.set_region_params(2, 0.25, 1.0, False)
        o.set_region_params(0, 1.0, 100.0, True)
        regions = np.array([1, 1, 1, 1, 1, 1, 2, 2, 2, 0, 2, 2, 2], np.uint8)
        K, V = zeros_kv(1, 1, 13, 16)
        o.append_tokens(0, regions, K, V, 0)
        z = np.zeros((1, 1, 1, 16), np.uint16)
        o.decode_step(1, z, z, z, [6])
        o.evict(1, [10 ** 6])
        S = o.page_S[0]
        assert S[0] == 0.375 and S[1] == want1, (mode, S)
        assert np.isinf(S[2]) and np.isinf(S[3])
        assert np.isinf(o.prio[o.slots(0)[9]])


# -------------------------------------------------------------- selection ---
def check_selection_bruteforce(om):
    """Greedy min-heap eviction (Algorithm 1) reaches the optimum of the
    page-level budget objective (Eq. 1 with equal page sizes, Sec. III-D):
    compared against exhaustive search over page subsets, up to ties."""
    rng = np.random.default_rng(13)
    for trial in range(300):
        P = int(rng.integers(1, 13))
        S = rng.choice([0.1, 0.2, 0.25, 0.3, 0.7, 0.9], size=P) if trial % 2 else rng.uniform(0, 1, P)
        S = np.asarray(S, np.float32)
        ev = rng.uniform(size=P) < 0.75
        budget = int(rng.integers(0, P + 1))
        want = max(0, P - budget)
        got = om.select_pages_min_heap(S, ev, want)
        cand = [p for p in range(P) if ev[p]]
        k = min(want, len(cand))
        assert len(got) == k and all(ev[p] for p in got) and len(set(got)) == k
        best = min((sum(float(S[p]) for p in c) for c in itertools.combinations(cand, k)), default=0.0)
        assert abs(sum(float(S[p]) for p in got) - best) < 1e-9, (S, ev, budget, got)
        if got:
            top = max(float(S[p]) for p in got)
            assert all(float(S[p]) >= top for p in cand if p not in got)


def check_token_level_objective(om):
    """With one token per page, Eq. 1 says keeping the B highest-scoring tokens
    after forcing the pinned set is optimal; exhaustive search over token
    subsets agrees with the oracle's eviction (the tail, the token being
    written, is kept as well)."""
    rng = np.random.default_rng(17)
    for trial in range(20):
        n0 = int(rng.integers(3, 10))
        o = make(om, L=1, Hq=2, Hkv=1, D=16, ps=1, phys=64, max_pages=64)
        for r in range(7):
            o.set_region_params(r, float(rng.uniform(0.1, 1)), float(rng.uniform(2, 40)), r == 0)
        regions = rng.integers(0, 7, n0).astype(np.uint8)
        K = f32_bits_to_bf16_bits(rng.standard_normal((1, 1, n0, 16)))
        o.append_tokens(0, regions, K, K.copy(), insert_step=-int(rng.integers(0, 30)))
        q = f32_bits_to_bf16_bits(rng.standard_normal((1, 1, 2, 16)))
        kn = f32_bits_to_bf16_bits(rng.standard_normal((1, 1, 1, 16)))
        o.decode_step(1, q, kn, kn.copy(), [int(rng.integers(1, 7))])
        before = list(o.block[0])
        n = len(before)
        budget = int(rng.integers(1, n + 1))
        o.evict(1, [budget])
        s_obs = o.prio[before]                  # one token per page: slot = physical id
        kept = [p for p in range(n) if before[p] in o.block[0]]
        forced = [p for p in range(n) if np.isinf(s_obs[p]) or p == n - 1]
        free = [p for p in range(n) if p not in forced]
        room = max(0, budget - len(forced))
        best = max((sum(s_obs[list(c)]) for c in itertools.combinations(free, min(room, len(free)))),
                   default=0.0)
        got = sum(s_obs[p] for p in kept if p not in forced)
        assert abs(got - best) < 1e-12 and all(p in kept for p in forced)


def check_compaction_and_conservation(om):
    """After evictions the kept pages keep their relative order, every physical
    id is either in exactly one block table or on the free stack (conservation),
    and the freed ids sit on top of the stack in (sequence, logical page) order."""
    rng = np.random.default_rng(19)
    B, L, D, ps = 3, 1, 16, 4
    o = make(om, L=L, Hq=2, Hkv=1, D=D, ps=ps, B=B, phys=40, max_pages=20)
    for r in range(7):
        o.set_region_params(r, float(rng.uniform(0.1, 1)), float(rng.uniform(2, 40)), r == 0)
    for b in range(B):
        n = int(rng.integers(20, 40))
        K = f32_bits_to_bf16_bits(rng.standard_normal((L, 1, n, D)))
        o.append_tokens(b, rng.integers(1, 7, n).astype(np.uint8), K, K.copy(), 0)
    for step in range(12):
        q = f32_bits_to_bf16_bits(rng.standard_normal((B, L, 2, D)))
        kn = f32_bits_to_bf16_bits(rng.standard_normal((B, L, 1, D)))
        o.decode_step(B, q, kn, kn.copy(), [6] * B)
        before = [list(r) for r in o.block[:B]]
        top_before = len(o.free)
        st, n_ev, ids, logical = o.evict(B, [4 + step % 3] * B)
        for b in range(B):
            assert o.block[b] == [p for j, p in enumerate(before[b]) if j not in logical[b]]
            assert ids[b] == [before[b][j] for j in logical[b]]
        assert o.free[top_before:] == [p for b in range(B) for p in ids[b]]
        allids = sorted(o.free + [p for b in range(B) for p in o.block[b]])
        assert allids == list(range(40))


def check_over_budget_and_no_observation(om):
    """Pins beyond the budget: every evictable page goes, pinned pages stay and
    the warning status comes back.  A second observation with no decode step
    in between changes neither a nor the clocks."""
    o = make(om, L=1, Hq=2, Hkv=1, D=16, ps=4, phys=32)
    o.set_region_params(0, 1.0, 100.0, True)
    regions = np.array([0] * 8 + [3] * 8 + [0] * 4, np.uint8)    # pages S S x x S | tail
    K, V = zeros_kv(1, 1, len(regions), 16)
    o.append_tokens(0, regions, K, V, 0)
    zq = np.zeros((1, 1, 2, 16), np.uint16)
    zkv = np.zeros((1, 1, 1, 16), np.uint16)
    o.decode_step(1, zq, zkv, zkv, [3])
    st, n_ev, ids, logical = o.evict(1, [2])
    assert st == om.MD_WARN_OVER_BUDGET and logical[0] == [2, 3], (st, logical)
    a0, t0 = o.a.copy(), o.t_ref.copy()
    st2, n2, _, _ = o.evict(1, [100])
    assert n2 == [0] and np.array_equal(a0, o.a) and np.array_equal(t0, o.t_ref)


def check_bf16_widening(om):
    bits = np.array([0x3F80, 0xC000, 0x3F81, 0x0000, 0x8000, 0x7F7F], np.uint16)
    got = om.bf16_bits_to_f64(bits)
    want = [1.0, -2.0, 1.0078125, 0.0, -0.0, 3.3895313892515355e38]
    assert list(got) == want


# ------------------------------------------------------------ calibration ---
def check_calibration_fit(om):
    """Eq. 6-7: on exactly exponential bucket means the count-weighted fit
    returns the true rate and half-life; with noise it agrees with numpy's
    least-squares routine (an independent implementation: SVD-based lstsq on
    the sqrt-weighted system)."""
    ages = np.arange(0, 160, 4) + 2.0
    for lam in (0.002, 0.0217, 0.0495):     # half-lives ~347, 32, 14 steps (Table 2 range)
        mean = 0.013 * np.exp(-lam * ages)
        cnt = np.arange(len(ages), 0, -1) * 7
        got, logc = om.wls_log_linear_fit(ages, mean, cnt)
        assert abs(got - lam) < 1e-12 and abs(logc - math.log(0.013)) < 1e-10
        assert abs(om.half_life(got) - math.log(2) / lam) < 1e-8
    rng = np.random.default_rng(23)
    mean = 0.01 * np.exp(-0.03 * ages) * np.exp(rng.normal(0, 0.2, len(ages)))
    cnt = rng.integers(1, 500, len(ages))
    lam, logc = om.wls_log_linear_fit(ages, mean, cnt)
    sw = np.sqrt(cnt)
    A = np.stack([np.ones_like(ages), ages], axis=1) * sw[:, None]
    coef = np.linalg.lstsq(A, np.log(mean) * sw, rcond=None)[0]
    assert abs(lam + coef[1]) < 1e-12 and abs(logc - coef[0]) < 1e-12
    # calibrate(): bucket centres width*b + width/2, regions with < 2 buckets -> NaN
    S = np.zeros((7, 8))
    C = np.zeros((7, 8), np.int64)
    C[2, :5] = 10
    S[2, :5] = 10 * 0.02 * np.exp(-0.05 * (4 * np.arange(5) + 2))
    C[3, 1] = 4
    S[3, 1] = 0.1
    rates, halves = om.calibrate(S, C)
    assert abs(rates[2] - 0.05) < 1e-12 and np.isnan(rates[3]) and np.isnan(rates[0])


def check_calibration_histogram(om):
    """The histogram gathers Abar by (region, age // 4): with identical keys
    every token gets Abar = 1/|K_t| exactly, so each bucket's sum is its
    count / |K_t|, with ages counted from the insertion steps."""
    o = make(om, L=1, Hq=2, Hkv=1, D=16, ps=4, phys=32)
    regions = np.array([1] * 5 + [4] * 6, np.uint8)
    steps = np.array([-9, -9, -9, -1, -1, -5, -5, -5, -5, -30, -30])
    K, V = zeros_kv(1, 1, len(regions), 16)
    o.append_tokens(0, regions, K, V, steps)
    o.calib_enable(True)
    zq = np.zeros((1, 1, 2, 16), np.uint16)
    zkv = np.zeros((1, 1, 1, 16), np.uint16)
    o.decode_step(1, zq, zkv, zkv, [6])           # t = 1: ages 10,10,10,2,2 | 6 x4, 31, 31 | new 0
    o.evict(1, [100])
    n = 12
    want = {(1, 2): 3, (1, 0): 2, (4, 1): 4, (4, 7): 2, (6, 0): 1}
    for (r, b), c in want.items():
        assert o.calib_cnt[r, b] == c, (r, b, o.calib_cnt[r, b])
        assert abs(o.calib_sum[r, b] - c / n) < 1e-15
    assert o.calib_cnt.sum() == n


# --------------------------------------------------------- policy variants ---
def check_policy_variants(om):
    """Mode 2 (attention term relative to the uniform level 1/|K_t|): under
    uniform attention a_1 = gamma/|K_t|, so alpha a |K_t| = alpha gamma for any
    |K_t|.  Mode 3 (recency) evicts the oldest evictable pages first, as a
    streaming window does.  Mode 4 draws are uniform in [0, 1): their mean and
    spread over many draws match U(0,1), and they are reproducible."""
    for n0 in (9, 30):
        o = make(om, L=1, Hq=2, Hkv=1, D=16, ps=4, phys=32, score_mode=2, attn_weight=3.0)
        K, V = zeros_kv(1, 1, n0, 16)
        o.append_tokens(0, np.full(n0, 2, np.uint8), K, V, 0)
        z = np.zeros((1, 1, 2, 16), np.uint16)
        zk = np.zeros((1, 1, 1, 16), np.uint16)
        o.decode_step(1, z, zk, zk, [2])
        o.evict(1, [100])
        s0 = o.prio[o.slots(0)[0]]
        assert abs(s0 - (0.5 * 2 ** (-1 / 30) + 3.0 * 0.1)) < 1e-12, (n0, s0)
    o = make(om, L=1, Hq=2, Hkv=1, D=16, ps=4, phys=32, score_mode=3)
    K, V = zeros_kv(1, 1, 24, 16)
    o.append_tokens(0, np.full(24, 3, np.uint8), K, V, np.repeat(np.arange(-6, 0), 4))
    z = np.zeros((1, 1, 2, 16), np.uint16)
    zk = np.zeros((1, 1, 1, 16), np.uint16)
    o.decode_step(1, z, zk, zk, [3])
    st, n, ids, logical = o.evict(1, [4])
    assert logical[0] == [0, 1, 2], logical
    u = om.random_draw(5, 3, np.arange(20000))
    assert 0.0 <= u.min() and u.max() < 1.0 and abs(u.mean() - 0.5) < 0.01 and abs(u.var() - 1 / 12) < 0.003
    assert np.array_equal(u, om.random_draw(5, 3, np.arange(20000)))
    assert not np.array_equal(u, om.random_draw(5, 4, np.arange(20000)))


# -------------------------------------------------- region-aligned pages ---
def check_region_aligned_pages(om):
    """Region-aligned allocation (Sec. III-D: a fresh page at each region
    boundary) leaves no page straddling a boundary; pages keep their partial
    fill, eviction removes exactly their tokens, and on page-aligned spans it
    makes the same layout as the default allocator."""
    regions = np.array([0] * 5 + [1] * 7 + [2] * 3 + [1] * 9, np.uint8)
    for aligned in (False, True):
        o = make(om, L=1, Hq=2, Hkv=1, D=16, ps=4, phys=32, region_aligned=aligned)
        K, V = zeros_kv(1, 1, len(regions), 16)
        o.append_tokens(0, regions, K, V, 0)
        sl = o.slots(0)
        pages = o.page_of_token(0)
        straddle = sum(len(set(regions[pages == p])) > 1 for p in range(len(o.block[0])))
        if aligned:
            assert o.fill[0] == [4, 1, 4, 3, 3, 4, 4, 1] and straddle == 0
        else:
            assert o.fill[0] == [4] * 6 and straddle == 2
        assert len(sl) == len(regions) and o.n_tokens[0] == len(regions)
        assert np.array_equal(o.region[sl], regions)
    # eviction removes the evicted pages' tokens, whatever their fill
    o = make(om, L=1, Hq=2, Hkv=1, D=16, ps=4, phys=32, region_aligned=True)
    for r in range(7):
        o.set_region_params(r, 0.1 * (r + 1), 30.0, False)
    K, V = zeros_kv(1, 1, len(regions), 16)
    o.append_tokens(0, regions, K, V, 0)
    z = np.zeros((1, 1, 2, 16), np.uint16)
    zk = np.zeros((1, 1, 1, 16), np.uint16)
    o.decode_step(1, z, zk, zk, [1])           # region 1 joins the last region-1 page
    st, n, ids, logical = o.evict(1, [6])
    assert o.fill[0][-1] == 2 and logical[0] == [0, 1]
    assert o.n_tokens[0] == len(regions) + 1 - 5
    # page-aligned spans: identical layout with or without alignment
    r2 = np.array([3] * 8 + [5] * 4 + [6] * 12, np.uint8)
    outs = []
    for aligned in (False, True):
        o = make(om, L=1, Hq=2, Hkv=1, D=16, ps=4, phys=32, region_aligned=aligned)
        o.append_tokens(0, r2, *zeros_kv(1, 1, len(r2), 16), 0)
        outs.append((list(o.block[0]), list(o.fill[0]), list(o.slots(0))))
    assert outs[0] == outs[1]


ALL_CHECKS = [
    check_decay_closed_forms, check_fig2_trajectories, check_ewma_closed_form,
    check_attention_closed_form, check_mass_sums_to_one, check_gqa_mapping,
    check_refresh_threshold, check_page_scores, check_selection_bruteforce,
    check_token_level_objective, check_compaction_and_conservation,
    check_over_budget_and_no_observation, check_bf16_widening,
    check_calibration_fit, check_calibration_histogram, check_policy_variants,
    check_region_aligned_pages,
]
