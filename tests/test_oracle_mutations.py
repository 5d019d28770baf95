"""Planted mistakes in the oracle (on the CPU) must each fail at least one pin:
evidence that the pins constrain every step of the oracle.  Each mutant is a
plausible slip: a dropped term or factor, a wrong sign, a transposed operand,
a wrong axis or divisor, a strict comparison, a max-heap for a min-heap."""
import math

import numpy as np
import pytest

import oracle.memdecay_oracle as om
from tests import oracle_checks as oc


def _attn_no_scale(q, K, V):
    s = q @ K.T
    e = np.exp(s - s.max(axis=1, keepdims=True))
    p = e / e.sum(axis=1, keepdims=True)
    return p @ V, p


def _attn_wrong_axis(q, K, V):
    s = (q @ K.T) / math.sqrt(q.shape[1])
    e = np.exp(s - s.max())
    p = e / e.sum(axis=0, keepdims=True)
    return p @ V, p


def _attn_transposed_values(q, K, V):
    s = (q @ K.T) / math.sqrt(q.shape[1])
    e = np.exp(s - s.max(axis=1, keepdims=True))
    p = e / e.sum(axis=1, keepdims=True)
    n, D = V.shape
    Vt = V.T[:n, :] if D >= n else V
    return p @ np.resize(Vt, V.shape), p


MUTANTS = {
    "decay_without_ln2": ("decay", lambda dt, h: np.exp(-np.asarray(dt, float) / np.asarray(h, float))),
    "decay_wrong_sign": ("decay", lambda dt, h: np.power(2.0, np.asarray(dt, float) / np.asarray(h, float))),
    "ewma_swapped_weights": ("ewma", lambda a, abar, rho, gamma: gamma * a + rho * abar),
    "ewma_dropped_memory": ("ewma", lambda a, abar, rho, gamma: gamma * abar),
    "refresh_strict": ("refresh", lambda t_ref, abar, tau, t:
                       np.where(np.asarray(abar, np.float32) > np.float32(tau), t, t_ref)),
    "refresh_never": ("refresh", lambda t_ref, abar, tau, t: t_ref),
    "score_dropped_attention": ("token_score", lambda base, d, a, alpha, mode, *r: base * d),
    "score_dropped_decay": ("token_score", lambda base, d, a, alpha, mode, *r: base + alpha * a),
    "normalised_term_unscaled": ("token_score", lambda base, d, a, alpha, mode, n=1, ti=None, nz=None,
                                 f=om.token_score: f(base, d, a, alpha, 0 if mode == 2 else mode, n, ti, nz)),
    "recency_reversed": ("token_score", lambda base, d, a, alpha, mode, n=1, ti=None, nz=None,
                         f=om.token_score: -np.asarray(ti, float) if mode == 3 else f(base, d, a, alpha, mode, n, ti, nz)),
    "page_sum_not_mean": ("page_score", lambda s, mode: float(np.sum(s))),
    "page_min_not_mean": ("page_score", lambda s, mode: float(np.min(s))),
    "mass_wrong_divisor": ("observed_mass", lambda W, k, L, Hq: W / float(k * L)),
    "attention_no_scale": ("attention_group", _attn_no_scale),
    "attention_wrong_axis": ("attention_group", _attn_wrong_axis),
    "attention_transposed_values": ("attention_group", _attn_transposed_values),
    "select_max_heap": ("select_pages_min_heap", lambda S, ev, k: sorted(
        sorted([p for p in range(len(S)) if ev[p]], key=lambda p: (-float(S[p]), p))[:k])),
    "fit_unweighted": ("wls_log_linear_fit", lambda x, y, w, f=om.wls_log_linear_fit: f(x, y, np.ones_like(np.asarray(w, float)))),
    "fit_wrong_sign": ("wls_log_linear_fit", lambda x, y, w, f=om.wls_log_linear_fit: (-f(x, y, w)[0], f(x, y, w)[1])),
    "bucket_width_8": ("age_bucket", lambda age, width=4: int(age) // 8),
    "half_life_without_ln2": ("half_life", lambda rate: 1.0 / rate if rate > 0 else math.inf),
    "select_ignores_pins": ("select_pages_min_heap", lambda S, ev, k: sorted(
        sorted(range(len(S)), key=lambda p: (float(S[p]), p))[:k])),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutant_is_caught(name, monkeypatch):
    attr, fn = MUTANTS[name]
    monkeypatch.setattr(om, attr, fn)
    caught = []
    for check in oc.ALL_CHECKS:
        try:
            check(om)
        except AssertionError:
            caught.append(check.__name__)
        except Exception:   # a crash is not counted as a pin catching the mistake
            pass
    assert caught, f"no pin catches mutant {name}"
