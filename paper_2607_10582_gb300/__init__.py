"""GB300 (sm_103a) MemDecay decode-time eviction loop.

Python binding of ``include/memdecay.h``: the same calls, argument
marshalling only.  Every step of the path runs in the CUDA kernels of
``libmemdecay.so``; there is no CPU or PyTorch fallback, and importing the
binding fails loudly when the library has not been built.  PyTorch provides
device memory (the workspace, input and output tensors) and streams.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libmemdecay.so")

MD_OK = 0
MD_WARN_OVER_BUDGET = 1
MD_ERR_INVALID_ARG = -1
MD_ERR_CAPACITY = -2
MD_ERR_WORKSPACE = -3
MD_ERR_CUDA = -4
MD_ERR_DEVICE_TIMEOUT = -5
MD_ERR_STATE = -6
STATUS_NAMES = {0: "MD_OK", 1: "MD_WARN_OVER_BUDGET", -1: "MD_ERR_INVALID_ARG", -2: "MD_ERR_CAPACITY",
                -3: "MD_ERR_WORKSPACE", -4: "MD_ERR_CUDA", -5: "MD_ERR_DEVICE_TIMEOUT",
                -6: "MD_ERR_STATE"}

(MD_REGION_SYSTEM, MD_REGION_PLAN, MD_REGION_USER, MD_REGION_TOOL_IN, MD_REGION_TOOL_OUT,
 MD_REGION_RETRIEVAL, MD_REGION_SCRATCHPAD) = range(7)
MD_NUM_REGIONS = 7
MD_MAX_BATCH = 256
MD_HEAD_DIM = 128
MD_MAX_GROUP = 8
MD_MAX_CHUNKS = 64
MD_MAX_CHUNK_TOKENS = 4096

(MD_STATE_BLOCK_TABLE, MD_STATE_PAGE_SCORE, MD_STATE_TOKEN_PRIO, MD_STATE_A, MD_STATE_T_REF,
 MD_STATE_AHAT, MD_STATE_FREE, MD_STATE_REGION, MD_STATE_WINDOW, MD_STATE_MASS, MD_STATE_POOL,
 MD_STATE_T_INS, MD_STATE_PAGE_FILL, MD_STATE_SEQ_TOKENS, MD_STATE_CALIB) = range(15)
MD_CALIB_BUCKETS = 256
MD_CALIB_BUCKET_WIDTH = 4
(MD_QUERY_TOKENS, MD_QUERY_PAGES, MD_QUERY_FREE_TOP, MD_QUERY_STEP, MD_QUERY_WINDOW,
 MD_QUERY_PINNED_PAGES) = range(6)
(MD_DEBUG_SPIN_LIMIT_NS, MD_DEBUG_EXTRA_ARRIVALS, MD_DEBUG_GRID_LIMIT, MD_DEBUG_UNIT_OVERHEAD,
 MD_DEBUG_FORCE_CHUNKS, MD_DEBUG_COMBINE_OVERHEAD, MD_DEBUG_ZERO_COPY) = range(7)
STAGES = ("append", "attention", "fold", "score", "select")


class md_config(ctypes.Structure):
    _fields_ = [
        ("num_layers", ctypes.c_int), ("num_q_heads", ctypes.c_int), ("num_kv_heads", ctypes.c_int),
        ("head_dim", ctypes.c_int), ("page_size", ctypes.c_int),
        ("max_batch", ctypes.c_int), ("max_pages_per_seq", ctypes.c_int), ("num_phys_pages", ctypes.c_int),
        ("rho", ctypes.c_float), ("gamma", ctypes.c_float), ("tau_scale", ctypes.c_float),
        ("attn_weight", ctypes.c_float),
        ("score_mode", ctypes.c_int), ("page_reduce", ctypes.c_int), ("keep_token_prio", ctypes.c_int),
        ("workspace", ctypes.c_void_p), ("workspace_bytes", ctypes.c_size_t),
        ("stream", ctypes.c_void_p),
        ("random_seed", ctypes.c_uint64),
        ("region_aligned_pages", ctypes.c_int),
    ]


# name -> (restype, argtypes); the names and order of include/memdecay.h
_c = ctypes
_P = _c.c_void_p
SIGNATURES = {
    "md_workspace_size": (_c.c_size_t, [_c.POINTER(md_config)]),
    "md_create": (_c.c_int, [_c.POINTER(md_config), _c.POINTER(_P)]),
    "md_set_region_params": (_c.c_int, [_P, _c.c_int, _c.c_float, _c.c_float, _c.c_int]),
    "md_append_tokens": (_c.c_int, [_P, _c.c_int, _c.c_int, _P, _P, _P, _P]),
    "md_decode_step": (_c.c_int, [_P, _c.c_int, _P, _P, _P, _P, _P]),
    "md_decode_step_host": (_c.c_int, [_P, _c.c_int, _P, _P, _P, _P, _P]),
    "md_decode_layer": (_c.c_int, [_P, _c.c_int, _c.c_int, _P, _P, _P, _P, _P]),
    "md_evict": (_c.c_int, [_P, _c.c_int, _P, _P, _P]),
    "md_sync": (_c.c_int, [_P]),
    "md_destroy": (_c.c_int, [_P]),
    "md_get_state": (_c.c_int, [_P, _c.c_int, _P, _c.c_size_t]),
    "md_set_state": (_c.c_int, [_P, _c.c_int, _P, _c.c_size_t]),
    "md_query": (_c.c_int, [_P, _c.c_int, _c.c_int, _c.POINTER(_c.c_int64)]),
    "md_state_bytes": (_c.c_int, [_P, _c.POINTER(_c.c_size_t), _c.POINTER(_c.c_size_t)]),
    "md_save_state": (_c.c_int, [_P, _P, _P]),
    "md_load_state": (_c.c_int, [_P, _P, _P]),
    "md_profile_enable": (_c.c_int, [_P, _c.c_int]),
    "md_profile_read": (_c.c_int, [_P, _P, _P, _c.c_int]),
    "md_debug_set": (_c.c_int, [_P, _c.c_int, _c.c_int64]),
    "md_calib_enable": (_c.c_int, [_P, _c.c_int]),
    "md_calib_read": (_c.c_int, [_P, _P, _P]),
    "md_calib_fit": (_c.c_int, [_P, _P, _c.c_int, _c.c_int, _c.c_int64, _P, _P]),
    "md_last_error": (_c.c_char_p, [_P]),
    "md_attend_mass_noalloc": (_c.c_int, [_P, _P, _P, _P, _P, _P, _c.c_int, _c.c_int, _c.c_int, _c.c_int,
                                          _c.c_int, _c.c_int, _c.c_int, _P]),
}

_lib = None


def lib():
    """The loaded libmemdecay.so.  Raises if it has not been built: there is
    no fallback implementation."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with "
                               f"`python -m paper_2607_10582_gb300.build`")
        L = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in SIGNATURES.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


class MemDecayError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {msg}")
        self.status = status


def _ptr(x) -> Optional[int]:
    """Device pointer of a torch tensor (or an int / None)."""
    if x is None:
        return None
    if isinstance(x, int):
        return x
    return x.data_ptr()


def _hptr(x) -> int:
    """Address of a contiguous host buffer: a CPU torch tensor (pinned for
    full copy speed) or a numpy array."""
    if isinstance(x, np.ndarray):
        if not x.flags["C_CONTIGUOUS"]:
            raise ValueError("host buffer must be contiguous")
        return x.ctypes.data
    if x.is_cuda or not x.is_contiguous():
        raise ValueError("host buffer must be a contiguous CPU tensor")
    return x.data_ptr()


def _host(arr, dtype):
    a = np.ascontiguousarray(np.asarray(arr, dtype=dtype))
    return a, a.ctypes.data


def md_workspace_size(cfg: md_config) -> int:
    return int(lib().md_workspace_size(ctypes.byref(cfg)))


def md_calib_fit(mass_sum: np.ndarray, count: np.ndarray, bucket_width: int = MD_CALIB_BUCKET_WIDTH,
                 min_count: int = 1):
    """Eq. 6-7 fit of a calibration histogram: (rate[7], half_life[7])."""
    s = np.ascontiguousarray(mass_sum, np.float64)
    n = np.ascontiguousarray(count, np.int64)
    rate = np.zeros(MD_NUM_REGIONS)
    half = np.zeros(MD_NUM_REGIONS)
    st = lib().md_calib_fit(s.ctypes.data, n.ctypes.data, s.shape[1], bucket_width, min_count,
                            rate.ctypes.data, half.ctypes.data)
    if st != MD_OK:
        raise MemDecayError(st, "md_calib_fit")
    return rate, half


class Cache:
    """One md_ctx with the workspace it lives in (a torch uint8 tensor on the
    current CUDA device).  Methods map one to one onto the C calls."""

    def __init__(self, num_layers: int, num_q_heads: int, num_kv_heads: int, page_size: int,
                 max_batch: int, max_pages_per_seq: int, num_phys_pages: int, *,
                 rho: float = 0.9, gamma: float = 0.1, tau_scale: float = 2.0,
                 attn_weight: float = 1.0, score_mode: int = 0, page_reduce: int = 0,
                 keep_token_prio: int = 1, random_seed: int = 0, region_aligned_pages: int = 0,
                 stream=None, device=None):
        import torch
        self.torch = torch
        self.device = torch.device(device) if device is not None else torch.device("cuda", torch.cuda.current_device())
        self.stream = stream if stream is not None else torch.cuda.current_stream(self.device)
        c = md_config(num_layers, num_q_heads, num_kv_heads, MD_HEAD_DIM, page_size,
                      max_batch, max_pages_per_seq, num_phys_pages,
                      rho, gamma, tau_scale, attn_weight, score_mode, page_reduce, keep_token_prio,
                      None, 0, ctypes.c_void_p(self.stream.cuda_stream), random_seed,
                      int(region_aligned_pages))
        need = md_workspace_size(c)
        if need == 0:
            raise MemDecayError(MD_ERR_INVALID_ARG, "invalid configuration")
        self.workspace = torch.empty(need + 1024, dtype=torch.uint8, device=self.device)
        base = self.workspace.data_ptr()
        aligned = (base + 1023) // 1024 * 1024
        c.workspace = aligned
        c.workspace_bytes = need
        self.cfg = c
        self.L, self.Hq, self.Hkv, self.ps = num_layers, num_q_heads, num_kv_heads, page_size
        self.max_batch, self.P_max, self.P_phys = max_batch, max_pages_per_seq, num_phys_pages
        h = ctypes.c_void_p()
        self._check(lib().md_create(ctypes.byref(c), ctypes.byref(h)), None)
        self.h = h

    # -- plumbing --
    def _check(self, st: int, h=0, ok=(MD_OK,)):
        if st in ok:
            return st
        msg = ""
        if h is not None:
            hh = self.h if h == 0 else h
            msg = lib().md_last_error(hh).decode()
        raise MemDecayError(st, msg)

    def close(self):
        if getattr(self, "h", None):
            lib().md_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # -- calls --
    def set_region_params(self, region: int, base: float, half_life: float, pinned: bool):
        return self._check(lib().md_set_region_params(self.h, region, base, half_life, int(pinned)))

    def append_tokens(self, seq: int, regions, k, v, insert_steps=None):
        regs, rp = _host(regions, np.uint8)
        sp = None
        if insert_steps is not None:
            steps, sp = _host(insert_steps, np.int32)
        return self._check(lib().md_append_tokens(self.h, seq, len(regs), rp, sp, _ptr(k), _ptr(v)))

    def decode_step(self, batch: int, q, k_new, v_new, new_regions, out):
        regs, rp = _host(new_regions, np.uint8)
        return self._check(lib().md_decode_step(self.h, batch, _ptr(q), _ptr(k_new), _ptr(v_new), rp, _ptr(out)))

    def decode_step_host(self, batch: int, q, k_new, v_new, new_regions, out):
        """md_decode_step_host: q, k_new, v_new and out are host buffers (CPU
        tensors or numpy arrays, bf16 bits); out is written once the stream
        gets there (sync() or a stream synchronisation)."""
        regs, rp = _host(new_regions, np.uint8)
        return self._check(lib().md_decode_step_host(self.h, batch, _hptr(q), _hptr(k_new), _hptr(v_new), rp,
                                                     _hptr(out)))

    def decode_layer(self, layer: int, batch: int, q, k_new, v_new, new_regions, out):
        regs, rp = _host(new_regions, np.uint8)
        return self._check(lib().md_decode_layer(self.h, layer, batch, _ptr(q), _ptr(k_new), _ptr(v_new), rp,
                                                 _ptr(out)))

    def evict(self, budgets: Sequence[int], evicted_ids=None):
        bud, bp = _host(budgets, np.int32)
        n_ev = np.zeros(len(bud), np.int32)
        st = lib().md_evict(self.h, len(bud), bp, n_ev.ctypes.data, _ptr(evicted_ids))
        self._check(st, 0, ok=(MD_OK, MD_WARN_OVER_BUDGET))
        return st, n_ev

    def sync(self):
        return lib().md_sync(self.h)

    def query(self, what: int, seq: int = 0) -> int:
        v = ctypes.c_int64()
        self._check(lib().md_query(self.h, what, seq, ctypes.byref(v)))
        return int(v.value)

    def state_spec(self, what: int):
        slots = self.P_phys * self.ps
        t = self.torch
        return {
            MD_STATE_BLOCK_TABLE: ((self.max_batch, self.P_max), t.int32),
            MD_STATE_PAGE_SCORE: ((self.max_batch, self.P_max), t.float32),
            MD_STATE_TOKEN_PRIO: ((slots,), t.float32),
            MD_STATE_A: ((slots,), t.float32),
            MD_STATE_T_REF: ((slots,), t.int32),
            MD_STATE_AHAT: ((slots,), t.float32),
            MD_STATE_FREE: ((self.P_phys,), t.int32),
            MD_STATE_REGION: ((slots,), t.uint8),
            MD_STATE_WINDOW: ((slots,), t.float32),
            MD_STATE_MASS: ((slots,), t.int64),
            MD_STATE_POOL: ((self.L, self.P_phys, self.Hkv, 2, self.ps, MD_HEAD_DIM), t.int16),
            MD_STATE_T_INS: ((slots,), t.int32),
            MD_STATE_PAGE_FILL: ((self.max_batch, self.P_max), t.uint8),
            MD_STATE_SEQ_TOKENS: ((self.max_batch,), t.int32),
            MD_STATE_CALIB: ((8 * MD_CALIB_BUCKETS * 12,), t.uint8),
        }[what]

    def get_state(self, what: int):
        shape, dt = self.state_spec(what)
        out = self.torch.empty(shape, dtype=dt, device=self.device)
        self._check(lib().md_get_state(self.h, what, out.data_ptr(), out.numel() * out.element_size()))
        return out

    def set_state(self, what: int, src):
        self._check(lib().md_set_state(self.h, what, src.data_ptr(), src.numel() * src.element_size()))

    def state_bytes(self):
        d, h = ctypes.c_size_t(), ctypes.c_size_t()
        self._check(lib().md_state_bytes(self.h, ctypes.byref(d), ctypes.byref(h)))
        return d.value, h.value

    def save_state(self):
        d, h = self.state_bytes()
        dev = self.torch.empty(d, dtype=self.torch.uint8, device=self.device)
        host = np.zeros(h, np.uint8)
        self._check(lib().md_save_state(self.h, dev.data_ptr(), host.ctypes.data))
        return dev, host

    def load_state(self, saved):
        dev, host = saved
        self._check(lib().md_load_state(self.h, dev.data_ptr(), host.ctypes.data))

    def profile_enable(self, on: bool = True):
        self._check(lib().md_profile_enable(self.h, int(on)))

    def profile_read(self):
        ms = np.zeros(5, np.float64)
        n = np.zeros(5, np.int64)
        self._check(lib().md_profile_read(self.h, ms.ctypes.data, n.ctypes.data, 5))
        return {STAGES[i]: (float(ms[i]), int(n[i])) for i in range(5)}

    def calib_enable(self, on: bool = True):
        self._check(lib().md_calib_enable(self.h, int(on)))

    def calib_read(self):
        """(mass_sum [7][256], count [7][256]) of the calibration histogram."""
        s = np.zeros((MD_NUM_REGIONS, MD_CALIB_BUCKETS), np.float64)
        n = np.zeros((MD_NUM_REGIONS, MD_CALIB_BUCKETS), np.int64)
        self._check(lib().md_calib_read(self.h, s.ctypes.data, n.ctypes.data))
        return s, n

    def debug_set(self, key: int, value: int):
        self._check(lib().md_debug_set(self.h, key, value))
