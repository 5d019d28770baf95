"""The C-ABI library loads and exports every symbol include/memdecay.h
declares; host-only calls behave (no GPU needed)."""
import ctypes
import os
import re

import pytest

import paper_2607_10582_gb300 as md
from paper_2607_10582_gb300 import build as mdbuild

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_functions():
    names = []
    for fn in sorted(os.listdir(os.path.join(ROOT, "include"))):
        if not fn.endswith(".h"):
            continue
        text = open(os.path.join(ROOT, "include", fn)).read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        names += re.findall(r"^[A-Za-z_][\w \*]*?\b(md_\w+)\s*\(", text, flags=re.M)
    return sorted(set(names))


@pytest.fixture(scope="module")
def lib():
    mdbuild.build()
    return md.lib()


def test_exports_every_declared_symbol(lib):
    names = declared_functions()
    assert len(names) >= 18, names
    for n in names:
        assert hasattr(lib, n), n
    assert set(names) == set(md.SIGNATURES), set(names) ^ set(md.SIGNATURES)


def _cfg(**kw):
    c = dict(num_layers=2, num_q_heads=16, num_kv_heads=2, head_dim=128, page_size=16,
             max_batch=4, max_pages_per_seq=64, num_phys_pages=256, rho=0.9, gamma=0.1,
             tau_scale=2.0, attn_weight=1.0, score_mode=0, page_reduce=0, keep_token_prio=1,
             workspace=None, workspace_bytes=0, stream=None, random_seed=0, region_aligned_pages=0)
    c.update(kw)
    return md.md_config(*[c[f] for f, _ in md.md_config._fields_])


def test_workspace_size_is_host_arithmetic(lib):
    n = md.md_workspace_size(_cfg())
    pool = 2 * 256 * 2 * 2 * 16 * 128 * 2
    assert n > pool
    assert md.md_workspace_size(_cfg(num_phys_pages=512)) - n >= pool
    for bad in (dict(head_dim=64), dict(page_size=8), dict(num_q_heads=18),
                dict(num_q_heads=32), dict(max_batch=0), dict(max_batch=257), dict(rho=1.5),
                dict(score_mode=5), dict(max_pages_per_seq=1 << 20), dict(num_layers=0)):
        assert md.md_workspace_size(_cfg(**bad)) == 0, bad


def test_step_mass_headroom_bounds_layers_times_query_heads(lib):
    """A decode step's mass per token is a u64 with 48 fraction bits, and a
    token receives at most 1 from each query head of each layer, so the
    product of layers and query heads must stay below 2^16."""
    assert md.md_workspace_size(_cfg(num_layers=255, num_q_heads=256, num_kv_heads=32)) > 0
    assert md.md_workspace_size(_cfg(num_layers=255, num_q_heads=264, num_kv_heads=33)) == 0


def test_create_rejects_bad_arguments_before_cuda(lib):
    h = ctypes.c_void_p()
    assert lib.md_create(None, ctypes.byref(h)) == md.MD_ERR_INVALID_ARG
    assert lib.md_create(ctypes.byref(_cfg(page_size=12)), ctypes.byref(h)) == md.MD_ERR_INVALID_ARG
    # no workspace / misaligned / too small
    assert lib.md_create(ctypes.byref(_cfg()), ctypes.byref(h)) == md.MD_ERR_WORKSPACE
    c = _cfg(workspace=1024 + 16, workspace_bytes=1 << 40)
    assert lib.md_create(ctypes.byref(c), ctypes.byref(h)) == md.MD_ERR_WORKSPACE
    c = _cfg(workspace=1 << 20, workspace_bytes=100)
    assert lib.md_create(ctypes.byref(c), ctypes.byref(h)) == md.MD_ERR_WORKSPACE
    assert lib.md_evict(None, 1, None, None, None) == md.MD_ERR_INVALID_ARG
    assert lib.md_last_error(None) == b"null handle"


def test_binding_fails_loudly_without_library(monkeypatch, tmp_path):
    monkeypatch.setattr(md, "_lib", None)
    monkeypatch.setattr(md, "LIB_PATH", str(tmp_path / "missing.so"))
    with pytest.raises(RuntimeError):
        md.lib()
