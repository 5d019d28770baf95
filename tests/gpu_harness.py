"""Lockstep parity harness: the CUDA path (through the C ABI binding) and the
fp64 oracle run the same seeded workload side by side and are compared after
every call.

Tolerances (stated here, used by every GPU parity test):
* attention output O: max abs error <= 2e-2 (bf16 K/V/Q and output);
* Abar, a and token / page priorities: max relative error <= 1e-4
  (relative to the oracle value, plus an absolute floor of 1e-30 for values
  that underflow fp32);
* eviction decisions: bit-exact block tables and free stacks, except where the
  oracle's page scores place two candidates within 1e-5 (relative) of the
  selection boundary; the refresh decision likewise where
  |Abar - tau| <= 1e-5 tau.
Where floating point allowed the GPU another valid choice, the harness checks
that the choice is valid and writes the oracle's choice back into the GPU's
state (never the other way round: no oracle input comes from the GPU)."""
from __future__ import annotations

import math

import numpy as np
import torch

import oracle.memdecay_oracle as om
import paper_2607_10582_gb300 as md
import synth

TOL_O_ABS = 2e-2
TOL_REL = 1e-4
TOL_FLOOR = 1e-30
TIE_REL = 1e-5


class TieStats:
    """How often the tie band decided anything.

    Per observation and sequence with an eviction: the relative gap between
    the selection boundary (the largest oracle page score S among the evicted
    pages) and the smallest score among the kept evictable pages.  A gap
    within TIE_REL means the oracle's own decision sat inside the band, where
    the GPU could take another valid choice.  For every choice the GPU took
    differently (an adoption), the distance of the swapped pages from the
    boundary, relative to it: the largest such distance is the narrowest band
    under which the run would still have passed.  Refresh decisions likewise,
    relative to tau."""

    def __init__(self):
        self.decisions = 0          # (observation, sequence) pairs that evicted pages
        self.pages_evicted = 0
        self.inside_band = 0        # of those, boundary gap <= TIE_REL
        self.gap_le = {1e-6: 0, 1e-7: 0, 0.0: 0}
        self.band_pages = 0         # evictable pages within TIE_REL of the boundary (all decisions)
        self.evict_adoptions = 0
        self.evict_adopt_max_dist = 0.0
        self.tokens_observed = 0
        self.refresh_in_band = 0    # tokens with |Abar - tau| <= TIE_REL tau
        self.refresh_adoptions = 0  # of those, decided differently by the GPU
        self.refresh_adopt_max_dist = 0.0

    def evict(self, S, want, got, page_flip):
        S = np.asarray(S, np.float64)
        if not want:
            return
        self.decisions += 1
        self.pages_evicted += len(want)
        boundary = max(S[j] for j in want)
        chosen = set(want)
        kept = [S[j] for j in range(len(S)) if j not in chosen and np.isfinite(S[j])]
        gap = (min(kept) - boundary) / (abs(boundary) + TOL_FLOOR) if kept else np.inf
        gap = abs(gap)
        fin = np.isfinite(S)
        self.band_pages += int(np.count_nonzero(fin & (np.abs(S - boundary) <= TIE_REL * abs(boundary))))
        if gap <= TIE_REL:
            self.inside_band += 1
        for x in self.gap_le:
            if gap <= x:
                self.gap_le[x] += 1
        if got is not None and sorted(got) != sorted(want):
            self.evict_adoptions += 1
            for j in set(got) ^ chosen:
                if not page_flip[j]:
                    d = abs(S[j] - boundary) / (abs(boundary) + TOL_FLOOR)
                    self.evict_adopt_max_dist = max(self.evict_adopt_max_dist, d)

    def refresh(self, abar, tau, mism):
        abar = np.asarray(abar, np.float64)
        self.tokens_observed += len(abar)
        self.refresh_in_band += int(np.count_nonzero(np.abs(abar - tau) <= TIE_REL * tau))
        if mism.any():
            self.refresh_adoptions += int(mism.sum())
            d = float(np.max(np.abs(abar[mism] - tau))) / tau
            self.refresh_adopt_max_dist = max(self.refresh_adopt_max_dist, d)

    def merge(self, other: "TieStats"):
        for k, v in vars(other).items():
            if k == "gap_le":
                for x, n in v.items():
                    self.gap_le[x] += n
            elif k.endswith("max_dist"):
                setattr(self, k, max(getattr(self, k), v))
            else:
                setattr(self, k, getattr(self, k) + v)

    def summary(self) -> dict:
        d = {k: v for k, v in vars(self).items() if k != "gap_le"}
        d.update({f"gap_le_{x:g}": n for x, n in self.gap_le.items()})
        return d


def to_dev(a: np.ndarray) -> torch.Tensor:
    """uint16 bf16 bits -> int16 device tensor (same bits)."""
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).cuda()


def rel_err(g, o):
    g = np.asarray(g, np.float64)
    o = np.asarray(o, np.float64)
    fin = np.isfinite(o)
    if not np.array_equal(np.isinf(g), np.isinf(o)):
        return np.inf
    if not fin.any():
        return 0.0
    return float(np.max(np.abs(g[fin] - o[fin]) / (np.abs(o[fin]) + TOL_FLOOR)))


class Lockstep:
    def __init__(self, w: synth.Workload, *, check_every=1, phys_slack=2, layerwise=False, calib=False,
                 p_max=None, host_buffers=False):
        self.w = w
        self.layerwise = layerwise
        self.host_buffers = host_buffers   # decode through md_decode_step_host with pinned buffers
        B = w.B
        self.P_max = w.max_pages_per_seq() if p_max is None else p_max
        self.P_phys = w.num_phys_pages() + phys_slack
        kw = dict(rho=w.rho, gamma=w.gamma, tau_scale=w.tau_scale, attn_weight=w.attn_weight,
                  score_mode=w.score_mode, page_reduce=w.page_reduce,
                  random_seed=w.extra.get("random_seed", 0))
        aligned = bool(w.extra.get("region_aligned", False))
        if aligned:    # a fresh page per region span can take up to one extra page per span
            self.P_max += w.extra.get("extra_pages", 64)
            self.P_phys += B * w.extra.get("extra_pages", 64)
        self.gpu = md.Cache(w.L, w.Hq, w.Hkv, w.page_size, B, self.P_max, self.P_phys,
                            region_aligned_pages=int(aligned), **kw)
        self.orc = om.Oracle(om.OracleConfig(w.L, w.Hq, w.Hkv, w.D, w.page_size, B, self.P_max,
                                             self.P_phys, region_aligned=aligned, **kw))
        for r in range(7):
            self.gpu.set_region_params(r, w.base[r], w.half_life[r], bool(w.pinned[r]))
            self.orc.set_region_params(r, w.base[r], w.half_life[r], bool(w.pinned[r]))
        if calib:
            self.gpu.calib_enable(True)
            self.orc.calib_enable(True)
        self.pos = [0] * B
        self.step_no = 0
        self.resyncs = {"evict": 0, "refresh": 0}
        self.max_err = {"O": 0.0, "ahat": 0.0, "a": 0.0, "prio": 0.0, "page": 0.0}
        self.ties = TieStats()

    # ------------------------------------------------------------ feeding --
    def prefill(self):
        w = self.w
        for b in range(w.B):
            n = w.n0(b)
            k, v = synth.kv_host(w.seed, b, w.L, w.Hkv, 0, n, w.regions[b], w.structured)
            self.gpu.append_tokens(b, w.regions[b], to_dev(k), to_dev(v), w.insert_steps[b])
            self.orc.append_tokens(b, w.regions[b], k, v, w.insert_steps[b])
            self.pos[b] = n
        torch.cuda.synchronize()

    def decode(self, regions=None, entry=None):
        """One decode step on both sides.  entry: "device" (md_decode_step),
        "host" (md_decode_step_host with pinned buffers) or "layers"
        (md_decode_layer per layer); default from the constructor."""
        w = self.w
        entry = entry or ("host" if self.host_buffers else "layers" if self.layerwise else "device")
        B = w.B
        t = self.orc.t + 1
        regions = [w.decode_region] * B if regions is None else list(regions)
        q = synth.q_host(w.seed, B, w.L, w.Hq, w.Hkv, t, w.structured)
        kn, vn = synth.step_kv_host(w.seed, self.pos, regions, w.L, w.Hkv, w.structured)
        out = torch.empty((B, w.L, w.Hq, w.D), dtype=torch.int16, device="cuda")
        if entry == "host":
            pin = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).pin_memory()
            out = torch.empty((B, w.L, w.Hq, w.D), dtype=torch.int16).pin_memory()
            self.gpu.decode_step_host(B, pin(q), pin(kn), pin(vn), regions, out)
            assert self.gpu.sync() == md.MD_OK
        elif entry == "layers":
            qd, knd, vnd = to_dev(q), to_dev(kn), to_dev(vn)
            for l in range(w.L):
                o_l = torch.empty((B, w.Hq, w.D), dtype=torch.int16, device="cuda")
                self.gpu.decode_layer(l, B, qd[:, l].contiguous(), knd[:, l].contiguous(),
                                      vnd[:, l].contiguous(), regions, o_l)
                out[:, l] = o_l
        else:
            self.gpu.decode_step(B, to_dev(q), to_dev(kn), to_dev(vn), regions, out)
        O = self.orc.decode_step(B, q, kn, vn, regions)
        for b in range(B):
            self.pos[b] += 1
        torch.cuda.synchronize()
        g = synth.bf16_to_f64(out.cpu().numpy().view(np.uint16))
        err = float(np.max(np.abs(g - O)))
        self.max_err["O"] = max(self.max_err["O"], err)
        assert err <= TOL_O_ABS, f"attention output error {err} at step {t}"
        self.step_no += 1
        return err

    # ------------------------------------------------------- observation --
    def observe(self, budgets=None):
        w = self.w
        B = w.B
        budgets = list(w.budget_pages) if budgets is None else list(budgets)
        g = self.gpu
        o = self.orc
        pre_block = [list(o.block[b]) for b in range(B)]
        pre_fill = [list(o.fill[b]) for b in range(B)]
        pre_slots = [o.slots(b) for b in range(B)]
        pre_pages = [o.page_of_token(b) for b in range(B)]
        observed = o.window_steps > 0
        ev = torch.full((B, self.P_max), -7, dtype=torch.int32, device="cuda")
        st_g, n_g = g.evict(budgets, ev)
        st_o, n_o, ids_o, logical_o = o.evict(B, budgets)
        assert st_g == st_o, (st_g, st_o)
        assert list(n_g) == list(n_o), (list(n_g), list(n_o))
        torch.cuda.synchronize()
        assert g.sync() == md.MD_OK
        ahat = g.get_state(md.MD_STATE_AHAT).cpu().numpy()
        a = g.get_state(md.MD_STATE_A).cpu().numpy()
        tref = g.get_state(md.MD_STATE_T_REF).cpu().numpy()
        prio = g.get_state(md.MD_STATE_TOKEN_PRIO).cpu().numpy()
        pscore = g.get_state(md.MD_STATE_PAGE_SCORE).cpu().numpy()
        bt = g.get_state(md.MD_STATE_BLOCK_TABLE).cpu().numpy()
        free = g.get_state(md.MD_STATE_FREE).cpu().numpy()
        evd = ev.cpu().numpy()
        ps = w.page_size
        fix_tref = False
        fix_blocks = False
        for b in range(B):
            # the slots observed this step are those of the pre-eviction block table
            sl = pre_slots[b]
            n_pre = len(sl)
            if observed:
                e = rel_err(ahat[sl], o.abar[sl])
                self.max_err["ahat"] = max(self.max_err["ahat"], e)
                assert e <= TOL_REL, f"Abar rel err {e} (seq {b})"
                e = rel_err(a[sl], o.a[sl])
                self.max_err["a"] = max(self.max_err["a"], e)
                assert e <= TOL_REL, f"a rel err {e} (seq {b})"
            # refresh decisions: exact unless within the tie band of tau
            tau = w.tau_scale / n_pre
            mism = tref[sl] != o.t_ref[sl]
            if observed:
                self.ties.refresh(o.abar[sl], tau, mism)
            flipped = np.zeros(n_pre, bool)
            if mism.any():
                amb = np.abs(o.abar[sl] - tau) <= TIE_REL * tau
                assert np.all(amb[mism]), f"refresh decision differs away from the tie band (seq {b})"
                flipped = mism
                fix_tref = True
                self.resyncs["refresh"] += int(mism.sum())
            ok_tok = ~flipped
            e = rel_err(prio[sl][ok_tok], o.prio[sl][ok_tok])
            self.max_err["prio"] = max(self.max_err["prio"], e)
            assert e <= TOL_REL, f"token priority rel err {e} (seq {b})"
            # page scores
            P_pre = len(pre_block[b])
            S_o = o.page_S[b]
            S_g = pscore[b, :P_pre].astype(np.float64)
            page_flip = np.zeros(P_pre, bool)
            page_flip[pre_pages[b][np.nonzero(flipped)[0]]] = True
            e = rel_err(S_g[~page_flip], S_o[~page_flip])
            self.max_err["page"] = max(self.max_err["page"], e)
            assert e <= TOL_REL, f"page score rel err {e} (seq {b})"
            # eviction decisions
            got = sorted(int(j) for j in np.nonzero(~np.isin(pre_block[b], bt[b, :P_pre - n_o[b]]))[0]) \
                if n_o[b] else []
            want = logical_o[b]
            # the evicted physical ids the call reports: the pages it evicted,
            # in logical order, then -1
            assert list(evd[b, n_o[b]:]) == [-1] * (self.P_max - n_o[b]), f"evicted ids padding (seq {b})"
            self.ties.evict(S_o, want, got, page_flip)
            if got != want:
                self._check_valid_choice(b, S_o, page_flip, got, want)
                assert list(evd[b, :n_o[b]]) == [pre_block[b][j] for j in got], f"evicted ids (seq {b})"
                fix_blocks = True
                self.resyncs["evict"] += 1
            else:
                assert list(bt[b, :len(o.block[b])]) == o.block[b], f"block table differs (seq {b})"
                assert list(evd[b, :n_o[b]]) == list(ids_o[b]), f"evicted ids (seq {b})"
        top = len(o.free)
        if not fix_blocks:
            assert list(free[:top]) == o.free, "free stack differs"
        if fix_blocks:
            self._push_blocks(bt, free)
        if fix_tref:
            t_fix = torch.from_numpy(o.t_ref.astype(np.int32)).cuda()
            g.set_state(md.MD_STATE_T_REF, t_fix)
        torch.cuda.synchronize()
        return n_o

    def _check_valid_choice(self, b, S_o, page_flip, got, want):
        """The GPU's evicted set is valid: same size, and it differs from the
        oracle's only among pages whose scores are within the tie band of the
        selection boundary (or whose score a tie-band refresh changed)."""
        assert len(got) == len(want)
        S = np.asarray(S_o, np.float64)
        boundary = max(S[j] for j in want)
        band = TIE_REL * abs(boundary) + TOL_FLOOR
        for j in set(got) ^ set(want):
            assert page_flip[j] or abs(S[j] - boundary) <= band, \
                f"seq {b}: page {j} (S={S[j]}) chosen differently, boundary {boundary}"

    def _push_blocks(self, bt, free):
        o = self.orc
        B = self.w.B
        bt = bt.copy()
        fill = self.gpu.get_state(md.MD_STATE_PAGE_FILL).cpu().numpy()
        ntok = self.gpu.get_state(md.MD_STATE_SEQ_TOKENS).cpu().numpy()
        for b in range(B):
            bt[b, :] = -1
            bt[b, :len(o.block[b])] = o.block[b]
            fill[b, :] = 0
            fill[b, :len(o.fill[b])] = o.fill[b]
            ntok[b] = o.n_tokens[b]
        free = free.copy()
        free[:len(o.free)] = o.free
        self.gpu.set_state(md.MD_STATE_BLOCK_TABLE, torch.from_numpy(bt).cuda())
        self.gpu.set_state(md.MD_STATE_FREE, torch.from_numpy(free).cuda())
        self.gpu.set_state(md.MD_STATE_PAGE_FILL, torch.from_numpy(fill).cuda())
        self.gpu.set_state(md.MD_STATE_SEQ_TOKENS, torch.from_numpy(ntok).cuda())

    def check_calibration(self):
        """Histogram counts bit-exact, mass sums within the Abar tolerance (plus
        the 2^-33 fixed-point rounding per observation), Eq. 6 rates close."""
        gs, gc = self.gpu.calib_read()
        o = self.orc
        assert np.array_equal(gc, o.calib_cnt), "calibration counts differ"
        tol = TOL_REL * np.abs(o.calib_sum) + gc * 2.0 ** -32 + TOL_FLOOR
        assert np.all(np.abs(gs - o.calib_sum) <= tol), "calibration sums differ"
        rate, _ = md.md_calib_fit(gs, gc)
        orate, _ = om.calibrate(o.calib_sum, o.calib_cnt)
        assert np.array_equal(np.isnan(rate), np.isnan(orate))
        ok = ~np.isnan(orate)
        assert np.all(np.abs(rate[ok] - orate[ok]) <= 1e-3 * np.abs(orate[ok]) + 1e-6), (rate, orate)
        return gc.sum()

    def check_layout(self):
        """Block tables and free stack bit-exact against the oracle."""
        bt = self.gpu.get_state(md.MD_STATE_BLOCK_TABLE).cpu().numpy()
        free = self.gpu.get_state(md.MD_STATE_FREE).cpu().numpy()
        o = self.orc
        fill = self.gpu.get_state(md.MD_STATE_PAGE_FILL).cpu().numpy()
        ntok = self.gpu.get_state(md.MD_STATE_SEQ_TOKENS).cpu().numpy()
        for b in range(self.w.B):
            assert list(bt[b, :len(o.block[b])]) == o.block[b]
            assert list(fill[b, :len(o.fill[b])]) == o.fill[b]
            assert self.gpu.query(md.MD_QUERY_TOKENS, b) == o.n_tokens[b] == ntok[b]
        assert self.gpu.query(md.MD_QUERY_FREE_TOP) == len(o.free)
        assert list(free[:len(o.free)]) == o.free

    def run(self, steps=None, check_layout_every=8):
        w = self.w
        steps = w.steps if steps is None else steps
        self.prefill()
        self.check_layout()
        for s in range(steps):
            self.decode()
            if (s + 1) % w.window_k == 0:
                self.observe()
            if (s + 1) % check_layout_every == 0:
                self.check_layout()
        return self
