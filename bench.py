"""Benchmark of the MemDecay decode-time eviction loop on GB300.

One step = one pass of the whole hot path over one batch: md_decode_step
(append + stage-1 paged GQA attention with per-token attention mass) and
md_evict (stages 2-4: retention priorities, page priorities, budgeted radix
selection and compaction).  Metric: cached tokens scored + evicted per second
per decode step (sum over sequences of |K_t| / step time).

Default workload: the largest single-GPU configuration, config 4 (Qwen2.5-3B
attention geometry, 16 sequences x 131,072 tokens, pages of 32, budget 5%,
w = 1), at its full-trace step: the first decode step after the prefill,
attending over the whole trace (77 GB of K/V) and evicting down to budget.
The device state is restored (untimed) before every timed step, so every
step does that full work; `--phase steady` times continuing steps instead.
Each timed step is bracketed by CUDA events on the launching stream and holds
no other event; the per-kernel times behind the roofline come from a second
pass over the same steps with the library's event pairs.  Where a step's K/V
would fit in L2 (configs 0 and 1), a 1 GiB write flushes it before each
step, outside the brackets.

`--impl reference` times the fp64 CPU oracle on the host cores on a bounded
sample of the same workload (the paper ships no code; the oracle is the
reference implementation of its equations).
"""
from __future__ import annotations

import argparse
import copy
import ctypes
import hashlib
import json
import os
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "cached tokens scored+evicted per second per decode step"
UNIT = "tokens/s"
SPEC_HBM_GBS = 8000.0
FALLBACK_HBM_GBS = 6800.0
L2_BYTES = 129 * 10**6          # GB300 L2
# written between timed steps when a step's K/V would fit in L2; larger than L2
# and long enough (about 0.16 ms) that the host has enqueued the next step before
# the GPU reaches it, so a latency-bound step's time is the GPU's, not the host's
FLUSH_BYTES = 2**30


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="native", choices=["native", "reference"])
    ap.add_argument("--config", type=int, default=4)
    ap.add_argument("--w", type=float, default=1.0, help="attention weight (config 4 sweeps 0/0.5/1/4)")
    ap.add_argument("--phase", default="full", choices=["full", "steady"])
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--max-tokens", type=int, default=0,
                    help="truncate every trace to this many tokens (small profiling cases)")
    ap.add_argument("--layerwise", action="store_true",
                    help="decode through md_decode_layer, one call per layer")
    ap.add_argument("--aligned", action="store_true",
                    help="region-aligned page allocation (a fresh page at each region boundary)")
    ap.add_argument("--structured", action="store_true",
                    help="keys and queries with region structure and hot tokens (refreshes fire)")
    ap.add_argument("--calib", action="store_true",
                    help="gather the calibration histogram (Eqs. 6-7) during observation steps")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-clocks", action="store_true")
    return ap.parse_args()


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return FALLBACK_HBM_GBS, "fallback"


def source_hash():
    h = hashlib.sha256()
    with open(os.path.join(ROOT, "paper_2607_10582_gb300", "csrc", "md_attn.cu"), "rb") as f:
        h.update(f.read())
    return h.hexdigest()[:16]


def ncu_traffic_per_token():
    """DRAM bytes per cached token per layer of the attention kernel, from the
    committed ncu summary, if it was taken on the current kernel source."""
    p = os.path.join(ROOT, "profiles", "attn_mass_kernel_traffic.txt")
    if not os.path.exists(p):
        return None
    vals = {}
    with open(p) as f:
        for line in f:
            if ":" in line and not line.startswith("#"):
                k, v = line.split(":", 1)
                vals[k.strip()] = v.strip()
    if vals.get("kernel_source_sha256_16") != source_hash():
        return None
    try:
        return float(vals["dram_bytes_per_token_layer"])
    except (KeyError, ValueError):
        return None


class ClockSampler:
    """nvidia-smi samples during the timed region (the GPU's clocks and
    throttle reasons are read, never set)."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "25"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except OSError:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append((time.perf_counter(), line.strip()))

    @staticmethod
    def _summary(lines):
        sm, mx, reasons = [], 0.0, set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for _, ln in lines:
            parts = [x.strip() for x in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx = max(mx, float(parts[2]))
            except ValueError:
                continue
            for name, val in zip(names, parts[5:9]):
                if val.lower() == "active":
                    reasons.add(name)
        if not sm:
            return None
        return {"sm_mhz": float(np.median(sm)), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}

    def stop(self, t0: float, t1: float):
        """Summary of the samples that arrived while the timed region ran
        (t0..t1 on time.perf_counter, plus 50 ms for the last one).  If the
        region was shorter than the sampling interval, the samples around it
        are used and the result says so."""
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        return self.summarise(t0, t1)

    def summarise(self, t0: float, t1: float):
        inside = [x for x in self.lines if t0 <= x[0] <= t1 + 0.05]
        res = self._summary(inside)
        if res is not None:
            res["window"] = "timed region"
            return res
        res = self._summary(self.lines)
        if res is not None:
            res["window"] = "around the timed region (shorter than the 25 ms sampling interval)"
        return res


# --------------------------------------------------------------- native ----
def run_native(args, rank, world, local_rank):
    import torch
    import paper_2607_10582_gb300 as md
    from paper_2607_10582_gb300 import build as mdbuild
    import synth

    mdbuild.build()
    synth.build()
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    stream = torch.cuda.current_stream(dev)
    w = make_workload(args, args.seed + rank)
    B, L, Hq, Hkv, ps, D = w.B, w.L, w.Hq, w.Hkv, w.page_size, w.D
    P_max, P_phys = w.max_pages_per_seq(), w.num_phys_pages()
    if args.aligned:   # each region span can leave one partly filled page
        spans = [int(np.count_nonzero(np.diff(w.regions[b].astype(np.int16)))) + 1 for b in range(B)]
        P_max += max(spans)
        P_phys += sum(spans)
    cache = md.Cache(L, Hq, Hkv, ps, B, P_max, P_phys,
                     rho=w.rho, gamma=w.gamma, tau_scale=w.tau_scale, attn_weight=w.attn_weight,
                     score_mode=w.score_mode, page_reduce=w.page_reduce, keep_token_prio=0,
                     region_aligned_pages=int(args.aligned))
    for r in range(7):
        cache.set_region_params(r, w.base[r], w.half_life[r], bool(w.pinned[r]))
    lib = synth.lib()
    kap = (ctypes.c_float * 9)(*synth.KAPPA_STRUCT) if w.structured else None
    nmax = max(w.n0(b) for b in range(B))
    kbuf = torch.empty(L * Hkv * nmax * D, dtype=torch.int16, device=dev)
    vbuf = torch.empty_like(kbuf)
    for b in range(B):
        n = w.n0(b)
        reg_d = torch.from_numpy(w.regions[b]).to(dev)
        assert lib.synth_fill_kv_dev(w.seed, int(w.structured), kap, b, L, Hkv, D, 0, n, reg_d.data_ptr(),
                                     kbuf.data_ptr(), vbuf.data_ptr(), stream.cuda_stream) == 0
        cache.append_tokens(b, w.regions[b], kbuf.data_ptr(), vbuf.data_ptr(), w.insert_steps[b])
    del kbuf, vbuf
    torch.cuda.synchronize()

    # per-step inputs, resident in HBM
    q = torch.empty((B, L, Hq, D), dtype=torch.int16, device=dev)
    kn = torch.empty((B, L, Hkv, D), dtype=torch.int16, device=dev)
    vn = torch.empty_like(kn)
    out = torch.empty_like(q)
    pos_d = torch.tensor([w.n0(b) for b in range(B)], dtype=torch.int32, device=dev)
    # the per-step host arguments as arrays, as a serving loop keeps them
    regs = np.full(B, w.decode_region, np.uint8)
    reg_d = torch.from_numpy(regs).to(dev)
    assert lib.synth_fill_q_dev(w.seed, int(w.structured), kap, B, L, Hq, Hq // Hkv, D, 1, q.data_ptr(),
                                stream.cuda_stream) == 0
    assert lib.synth_fill_step_kv_dev(w.seed, int(w.structured), kap, B, L, Hkv, D, pos_d.data_ptr(),
                                      reg_d.data_ptr(), kn.data_ptr(), vn.data_ptr(), stream.cuda_stream) == 0
    torch.cuda.synchronize()
    budgets = np.asarray(w.budget_pages, np.int32)

    # tensors a step reads from the host in the end-to-end measurement
    step_inputs = [q, kn, vn]
    step_output = out
    if args.layerwise:
        # a model hands each layer its own contiguous [B][heads][D] tensors
        q_lm = q.permute(1, 0, 2, 3).contiguous()
        kn_lm = kn.permute(1, 0, 2, 3).contiguous()
        vn_lm = vn.permute(1, 0, 2, 3).contiguous()
        out_lm = torch.empty((L, B, Hq, D), dtype=torch.int16, device=dev)
        q_l, kn_l, vn_l, out_l = list(q_lm), list(kn_lm), list(vn_lm), list(out_lm)
        step_inputs = [q_lm, kn_lm, vn_lm]
        step_output = out_lm

    def one_step():
        """One decode step (and the observation when the window is full);
        returns the pages evicted per sequence, or None."""
        if args.layerwise:
            for l in range(L):
                cache.decode_layer(l, B, q_l[l], kn_l[l], vn_l[l], regs, out_l[l])
        else:
            cache.decode_step(B, q, kn, vn, regs, out)
        # observation every window_k steps (k = 1 for configs 0-2 and 4)
        if cache.query(md.MD_QUERY_WINDOW) >= w.window_k:
            return cache.evict(budgets)[1]
        return None

    if args.phase == "steady":
        one_step()
        if cache.query(md.MD_QUERY_WINDOW) > 0:
            cache.evict(budgets)
        torch.cuda.synchronize()
    if args.calib:
        cache.calib_enable(True)
    saved = cache.save_state()
    tokens_saved = [cache.query(md.MD_QUERY_TOKENS, b) for b in range(B)]
    window_saved = cache.query(md.MD_QUERY_WINDOW)
    restore = args.phase == "full"
    # a step whose K/V could stay in L2 gets the L2 flushed before it (untimed)
    flush_buf = torch.empty(FLUSH_BYTES // 4, dtype=torch.int32, device=dev) if needs_flush(w) else None

    def before_step():
        if restore:
            cache.load_state(saved)
        if flush_buf is not None:
            flush_buf.fill_(1)

    for _ in range(args.warmup):
        before_step()
        one_step()
    torch.cuda.synchronize()
    assert cache.sync() == md.MD_OK

    def run_steps(profile: bool):
        """K steps, each bracketed by CUDA events on the launching stream
        (restore and flush happen outside the brackets).  With `profile` the
        library also records an event pair around each of its kernels."""
        starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
        ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
        tok_per_step = []
        # cached tokens per sequence, tracked on the host so that the loop adds
        # no per-sequence calls of its own: a step appends one token per
        # sequence, an eviction removes whole pages (partly filled ones only
        # with region-aligned pages, where the count is read back instead)
        tokens0 = tokens_saved if restore else [cache.query(md.MD_QUERY_TOKENS, b) for b in range(B)]
        tokens = list(tokens0)
        torch.cuda.synchronize()
        cache.profile_enable(profile)
        wall0 = time.perf_counter()
        for i in range(args.steps):
            before_step()
            if restore:
                tokens = list(tokens0)
            tok_per_step.append(sum(tokens) + B)
            starts[i].record(stream)
            n_ev = one_step()
            ends[i].record(stream)
            if args.aligned and n_ev is not None:
                tokens = [cache.query(md.MD_QUERY_TOKENS, b) for b in range(B)]
            else:
                tokens = [n + 1 - (int(n_ev[b]) * ps if n_ev is not None else 0) for b, n in enumerate(tokens)]
        torch.cuda.synchronize()
        wall = time.perf_counter() - wall0
        # the host-side count agrees with the library's
        assert tokens == [cache.query(md.MD_QUERY_TOKENS, b) for b in range(B)], "token bookkeeping"
        prof = cache.profile_read() if profile else None
        cache.profile_enable(False)
        assert cache.sync() == md.MD_OK
        return [a.elapsed_time(b) for a, b in zip(starts, ends)], tok_per_step, prof, wall0, wall

    # ---- timed region: K steps, no event inside a step ----
    clocks = ClockSampler(local_rank) if not args.no_clocks else None
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    if clocks:
        clocks.start()
        time.sleep(0.3)
    step_ms, tok_per_step, _, wall0, wall = run_steps(False)
    if world > 1:
        torch.distributed.barrier()
    clk = clocks.stop(wall0, wall0 + wall) if clocks else None
    total_ms = float(sum(step_ms))

    # ---- per-kernel times: the same K steps again with the library's event
    # pairs around every kernel (an event between two kernels keeps them
    # from overlapping, so these runs are not the timed ones) ----
    _, prof_tokens, prof, _, _ = run_steps(True)
    launches = sum(n for _, n in prof.values())
    attn_ms, attn_n = prof["attention"]

    # ---- end to end through the C ABI with host buffers ----
    e2e = None
    if not args.no_e2e:
        hosts = [t.cpu().pin_memory() for t in step_inputs]
        outh = torch.empty(step_output.shape, dtype=step_output.dtype).pin_memory()
        def e2e_steps():
            e_ms = []
            # decode steps since the last observation, tracked on the host as a
            # caller would (the library's count is checked afterwards)
            window = cache.query(md.MD_QUERY_WINDOW)
            for i in range(args.warmup + args.steps):
                before_step()
                if restore:
                    window = window_saved
                torch.cuda.synchronize()
                t0 = time.perf_counter()
                if args.layerwise:
                    # the per-layer entry takes device tensors: copy in, run, copy out
                    for d_t, h_t in zip(step_inputs, hosts):
                        d_t.copy_(h_t, non_blocking=True)
                    one_step()
                    outh.copy_(step_output, non_blocking=True)
                else:
                    # the host-buffer entry point moves inputs and output itself
                    cache.decode_step_host(B, hosts[0], hosts[1], hosts[2], regs, outh)
                    window += 1
                    if window >= w.window_k:
                        cache.evict(budgets)
                        window = 0
                torch.cuda.synchronize()
                if i >= args.warmup:
                    e_ms.append((time.perf_counter() - t0) * 1e3)
            if not args.layerwise:
                assert window == cache.query(md.MD_QUERY_WINDOW), "window bookkeeping"
            return float(np.mean(e_ms))

        e_main = e2e_steps()
        e_copies = None
        if not args.layerwise:
            cache.debug_set(md.MD_DEBUG_ZERO_COPY, 0)
            e_copies = e2e_steps()
            cache.debug_set(md.MD_DEBUG_ZERO_COPY, 1)
        h2d = sum(h_t.numel() for h_t in hosts) * 2 + B
        d2h = outh.numel() * 2
        e2e = {"ms_per_step": e_main, "ms_per_step_copies": e_copies, "tokens_per_step": tok_per_step[0],
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h}
    return dict(w=w, step_ms=step_ms, total_ms=total_ms, wall_s=wall, tokens=tok_per_step,
                prof=prof, prof_tokens=prof_tokens, launches=launches, attn_ms=attn_ms, attn_n=attn_n,
                clocks=clk, e2e=e2e, kv_bytes_per_token=L * Hkv * 2 * D * 2)


# ------------------------------------------------------------ reference ----
def oracle_sample(w, layers: int, seq: int = 0):
    """Build the oracle for one sequence of workload w, keeping `layers` of its
    L layers (the attention work is linear in L), prefilled (untimed)."""
    import oracle.memdecay_oracle as om
    import synth
    n = w.n0(seq)
    cfg = om.OracleConfig(layers, w.Hq, w.Hkv, w.D, w.page_size, 1, w.max_pages_per_seq(),
                          w.pages0(seq) + w.steps // w.page_size + 2, rho=w.rho, gamma=w.gamma,
                          tau_scale=w.tau_scale, attn_weight=w.attn_weight, score_mode=w.score_mode,
                          page_reduce=w.page_reduce)
    o = om.Oracle(cfg)
    for r in range(7):
        o.set_region_params(r, w.base[r], w.half_life[r], bool(w.pinned[r]))
    k, v = synth.kv_host(w.seed, seq, layers, w.Hkv, 0, n, w.regions[seq], w.structured)
    o.append_tokens(0, w.regions[seq], k, v, w.insert_steps[seq])
    return o


def oracle_step_inputs(w, layers: int, seq: int, t: int):
    """Queries and the new token's K/V of decode step t for one sequence."""
    import synth
    q = synth.q_host(w.seed, w.B, layers, w.Hq, w.Hkv, t, w.structured)[seq:seq + 1]
    kn, vn = synth.step_kv_host(w.seed, [w.n0(seq) + t - 1], [w.decode_region], layers, w.Hkv, w.structured)
    return q, kn, vn


def make_workload(args, seed):
    import synth
    over = {"attn_weight": args.w} if args.config == 4 else {}
    if args.structured:
        over["structured"] = True
    w = synth.make_workload(args.config, seed=seed, **over)
    if args.max_tokens:
        n = args.max_tokens
        w.regions = [r[:n].copy() for r in w.regions]
        w.insert_steps = [s[:n].copy() for s in w.insert_steps]
        w.name += f" (traces truncated to {n} tokens)"
    return w


def _oracle_worker(task):
    """One host process: the oracle on one sampled sequence (`layers` of its
    L layers).  Full-trace phase: prefilled once, then `reps` timed steps,
    each on a fresh copy of the prefilled state.  Steady phase: the first
    observation window (the full-trace step and the eviction to budget) runs
    untimed, then `reps` windows of window_k decode steps and their
    observation are timed.  Returns per step (decode seconds, evict seconds):
    a window's times divided by its decode steps."""
    args_d, seq, layers, reps = task
    a = argparse.Namespace(**args_d)
    w = make_workload(a, a.seed)
    o0 = oracle_sample(w, layers, seq)
    out = []
    if a.phase == "steady":
        o, t = o0, 0

        def window():
            nonlocal t
            dec, tok = 0.0, 0
            for _ in range(w.window_k):
                t += 1
                q, kn, vn = oracle_step_inputs(w, layers, seq, t)
                t0 = time.perf_counter()
                o.decode_step(1, q, kn, vn, [w.decode_region])
                dec += time.perf_counter() - t0
                tok += o.n_tokens[0]
            t0 = time.perf_counter()
            o.evict(1, [w.budget_pages[seq]])
            return dec, time.perf_counter() - t0, tok

        window()
        for _ in range(reps):
            dec, ev, tok = window()
            out.append((dec / w.window_k, ev / w.window_k, tok / w.window_k))
        return out
    q, kn, vn = oracle_step_inputs(w, layers, seq, 1)
    for _ in range(reps):
        o = copy.deepcopy(o0)
        t0 = time.perf_counter()
        o.decode_step(1, q, kn, vn, [w.decode_region])
        t1 = time.perf_counter()
        o.evict(1, [w.budget_pages[seq]])
        t2 = time.perf_counter()
        out.append((t1 - t0, t2 - t1, w.n0(seq) + 1))
    return out


ORACLE_SAMPLE_LAYERS = 8       # layers of the oracle's sample on a long full trace
ORACLE_ALL_LAYERS_TOKENS = 8192   # traces up to this long run every layer


def parallel_oracle(args, reps: int):
    """Time the fp64 oracle on the host cores: one process per core (numpy
    single-threaded in each), each on its own sequence of the workload.  The
    whole workload's step time is ceil(B / P) times the slowest process's
    step.  On the full-trace step of a long trace the oracle attends over
    ORACLE_SAMPLE_LAYERS layers and its decode time is scaled to all L layers
    (the attention work is linear in L); otherwise every layer runs.  Returns
    (seconds per step for each rep as measured on the sample, seconds per step
    scaled to the workload for each rep, processes, a description)."""
    import multiprocessing as mp
    w = make_workload(args, args.seed)
    long_full = args.phase == "full" and w.n0(0) > ORACLE_ALL_LAYERS_TOKENS
    layers = min(ORACLE_SAMPLE_LAYERS, w.L) if long_full else w.L
    try:
        ncpu = len(os.sched_getaffinity(0))
    except AttributeError:
        ncpu = os.cpu_count() or 1
    P = max(1, min(ncpu, w.B))
    for var in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        os.environ[var] = "1"
    args_d = dict(vars(args))
    tasks = [(args_d, b, layers, reps) for b in range(P)]
    ctx = mp.get_context("spawn")
    with ctx.Pool(P) as pool:
        res = pool.map(_oracle_worker, tasks)
    rounds = -(-w.B // P)
    measured, scaled = [], []
    for r in range(reps):
        measured.append(max(d + e for (d, e, _) in (res[p][r] for p in range(P))))
        scaled.append(rounds * max(d * (w.L / layers) + e for (d, e, _) in (res[p][r] for p in range(P))))
    # cached tokens per step of the whole batch: the measured sequences' mean
    # per sequence (exact in the full-trace phase, where every sequence of a
    # config holds the same trace length)
    tokens_step = w.B * float(np.mean([x[2] for p in range(P) for x in res[p]]))
    what = ("the full-trace step (prefill untimed, the state copied before each step)" if args.phase == "full"
            else f"steady steps: the first observation window (full trace, eviction to budget) untimed, then "
                 f"windows of {w.window_k} decode step(s) and their observation, per decode step")
    scale = []
    if layers < w.L:
        scale.append(f"decode time x{w.L / layers:g} ({layers} of {w.L} layers measured)")
    if rounds > 1:
        scale.append(f"x{rounds} rounds ({P} of {w.B} sequences measured)")
    sample = (f"sequences 0..{P - 1} of {w.B}, one per process on {P} host cores (single-threaded numpy), "
              f"{w.n0(0)}-token traces, {what}; " +
              ("measured on the whole workload" if not scale else "scaled to the workload: " + "; ".join(scale)))
    info = {"processes": P, "layers_measured": layers, "layers": w.L, "rounds": rounds, "sample": sample,
            "scaled": bool(scale), "tokens_per_step": tokens_step}
    return measured, scaled, info


def run_reference(args):
    w = make_workload(args, args.seed)
    measured, scaled, info = parallel_oracle(args, args.warmup + args.steps)
    sec = float(np.mean(scaled[args.warmup:]))
    value = info["tokens_per_step"] / sec
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": sec * 1e3, "higher_is_better": True,
            "ms_per_step_kind": ("scaled to the workload from a measured sample (see cpu_baseline.sample)"
                                 if info["scaled"] else "measured"),
            "measured_sample_ms_per_step": float(np.mean(measured[args.warmup:])) * 1e3,
            "scaled_from_layers": info["layers_measured"] if info["layers_measured"] < info["layers"] else None,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": workload_config(w, args),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": info["processes"], "kind": "oracle",
                             "sample": info["sample"]},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def needs_flush(w) -> bool:
    """Whether a step's K/V (the initial trace) is small enough to stay in L2
    between steps, so that the L2 must be flushed before each timed step."""
    tokens = sum(w.n0(b) + 1 for b in range(w.B))
    return tokens * w.L * w.Hkv * 2 * w.D * 2 < 2 * L2_BYTES


def workload_config(w, args):
    return {"workload": w.name, "batch": w.B, "tokens_per_seq": w.n0(0), "layers": w.L,
            "q_heads": w.Hq, "kv_heads": w.Hkv, "head_dim": w.D, "page_size": w.page_size,
            "budget_pages": w.budget_pages[0], "attn_weight": w.attn_weight, "window_k": w.window_k,
            "score_mode": "paper additive (Eq. 4)" if w.score_mode == 0 else "multiplicative",
            "phase": "full-trace step (state restored before each step)" if args.phase == "full"
            else "steady state",
            "l2": ("L2 flushed before every timed step (1 GiB write, untimed): a step's K/V fits in L2"
                   if needs_flush(w) else "no flush: inputs larger than L2 (K/V read per step >> 129 MB)"),
            "parallelism": "replicas" if args.gpus > 1 else "1 GPU", "seed": args.seed,
            "entry": "md_decode_layer x L + md_evict" if args.layerwise else "md_decode_step + md_evict",
            "calibration_histogram": bool(args.calib),
            "page_allocation": "region-aligned" if args.aligned else "contiguous",
            "values": ("structured: per-region key offsets along one direction, 2% hot keys (Fig. 3 mass ratios)"
                       if w.structured else "iid N(0,1)")}


def combine_over_ranks(total_ms: float, tokens_total: float, device):
    """Whole-job numbers of a replicated run: the timed region is the slowest
    rank's, the work is the sum over ranks."""
    import torch
    t = torch.tensor([total_ms], dtype=torch.float64, device=device)
    n = torch.tensor([tokens_total], dtype=torch.float64, device=device)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    torch.distributed.all_reduce(n, op=torch.distributed.ReduceOp.SUM)
    return float(t.item()), float(n.item())


# ------------------------------------------------------------------ main ----
def main():
    args = parse()
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        if rank == 0:
            run_reference(args)
        return
    import torch
    if world > 1:
        torch.cuda.set_device(local_rank)
        torch.distributed.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
    r = run_native(args, rank, world, local_rank)
    w = r["w"]
    total_ms = r["total_ms"]
    tokens = float(np.mean(r["tokens"]))
    if world > 1:
        total_ms, all_tokens = combine_over_ranks(total_ms, tokens * args.steps, "cuda")
    else:
        all_tokens = tokens * args.steps
    if rank != 0:
        torch.distributed.destroy_process_group()
        return
    ms_per_step = total_ms / args.steps
    value = all_tokens / (total_ms / 1e3)
    peak, peak_kind = peaks()
    # dominant kernel: stage-1 attention.  Algorithmic bytes per launch = the
    # K and V rows of every cached token in every layer, plus Q and O; the
    # kernel's time comes from the profiled pass over the same K steps.
    qo_bytes = 2 * w.B * w.L * w.Hq * w.D * 2
    attn_bytes = tokens * r["kv_bytes_per_token"] + qo_bytes
    prof_tokens = float(np.mean(r["prof_tokens"]))
    launches_per_step = max(1, r["attn_n"] // args.steps)     # L with --layerwise, else 1
    attn_avg_s = r["attn_ms"] / max(1, r["attn_n"]) / 1e3
    bytes_per_launch = (prof_tokens * r["kv_bytes_per_token"] + qo_bytes) / launches_per_step
    achieved = bytes_per_launch / attn_avg_s / 1e9
    tpt = ncu_traffic_per_token()
    traffic = None if tpt is None else tpt * prof_tokens * w.L / launches_per_step
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": workload_config(w, args),
        "roofline": {"bound": "hbm", "kernel": "attn_mass_kernel (stage 1)", "achieved": achieved,
                     "peak": peak, "unit": "GB/s", "frac": achieved / peak, "peak_kind": f"{peak_kind} copy",
                     "traffic": traffic, "algorithmic_bytes": bytes_per_launch,
                     "launches_per_step": launches_per_step,
                     "frac_of_8TBps_spec": achieved / SPEC_HBM_GBS,
                     "timing": "kernel time from the library's CUDA events around each launch, in a second "
                               "pass over the same K steps right after the timed region (events between "
                               "kernels would add gaps to the timed steps)"},
        "step_hbm_fraction": {"algorithmic_GBps": attn_bytes / (ms_per_step / 1e3) / 1e9,
                              "frac_measured": attn_bytes / (ms_per_step / 1e3) / 1e9 / peak,
                              "frac_of_8TBps_spec": attn_bytes / (ms_per_step / 1e3) / 1e9 / SPEC_HBM_GBS},
        "stage_ms_per_step": {k: v[0] / args.steps for k, v in r["prof"].items()},
        "stage_timing": "profiled pass (see roofline.timing); stage times include the gaps the events add",
        "gpu_launches": r["launches"],
        "clocks": r["clocks"],
        "wall_s_timed": r["wall_s"],
    }
    if r["e2e"]:
        e = r["e2e"]
        line["e2e"] = {"value": e["tokens_per_step"] * world / (e["ms_per_step"] / 1e3), "unit": UNIT,
                       "ms_per_step": e["ms_per_step"], "h2d_bytes_per_step": e["h2d_bytes_per_step"],
                       "d2h_bytes_per_step": e["d2h_bytes_per_step"],
                       "entry": ("pinned-host copies + md_decode_layer x L + md_evict" if args.layerwise
                                 else "md_decode_step_host + md_evict: the step's inputs start and its output "
                                      "ends in pinned host memory; the query rows are copied in (cudaMemcpyAsync), "
                                      "the append kernel reads the new K/V and the attention kernel writes the "
                                      "output in place over the host link (NVLink-C2C)")}
        if e.get("ms_per_step_copies") is not None:
            line["e2e"]["copy_path"] = {
                "value": e["tokens_per_step"] * world / (e["ms_per_step_copies"] / 1e3), "unit": UNIT,
                "ms_per_step": e["ms_per_step_copies"],
                "entry": "md_decode_step_host with MD_DEBUG_ZERO_COPY = 0: cudaMemcpyAsync of the inputs "
                         "into the workspace and of the output back, inside the call"}
    if not args.no_cpu_baseline and world == 1:
        measured, scaled, info = parallel_oracle(args, 3)
        line["cpu_baseline"] = {"value": info["tokens_per_step"] / min(scaled), "unit": UNIT,
                                "cores": info["processes"],
                                "kind": "oracle", "sample": info["sample"],
                                "ms_per_step": min(scaled) * 1e3,
                                "ms_per_step_kind": "scaled from the measured sample" if info["scaled"]
                                else "measured",
                                "measured_sample_ms_per_step": min(measured) * 1e3,
                                "scaled_from_layers": info["layers_measured"]
                                if info["layers_measured"] < info["layers"] else None}
    print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
