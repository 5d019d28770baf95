"""md_attend_mass_noalloc: stage 1 for callers that cannot allocate device
memory (a serving engine that owns the allocator, code that must not
allocate once it is running, a fixed memory budget).  It uses a fixed
scratch array inside the library instead of a workspace.  Its output must
match the workspace path (md_decode_step's attention output, and its step
mass per token: the sum of the rows over layers and KV heads)
within the parity tolerances, on two calls in a row (the second call finds
the first call's leftovers in the shared array)."""
import ctypes

import numpy as np
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu
if not torch.cuda.is_available():  # pragma: no cover
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

import paper_2607_10582_gb300 as md  # noqa: E402
import synth  # noqa: E402
from paper_2607_10582_gb300 import build as mdbuild  # noqa: E402
from tests.gpu_harness import TOL_FLOOR, TOL_O_ABS, TOL_REL, to_dev  # noqa: E402

mdbuild.build()
synth.build()


@pytest.mark.parametrize("L,Hq,ps,lengths", [
    (2, 16, 16, [900, 2500]),
    (2, 12, 32, [3000, 70, 1500]),
    # many items and long sequences: the split that fills the grid (3 chunks
    # per item) does not fit the fixed array, so the call takes 4; the
    # 40-token sequence gets fewer chunks than the others
    (16, 16, 16, [3000] * 7 + [40] + [3000] * 8),
    # a serving batch shaped like the 3B geometry at budget: one chunk per
    # item, no partials
    (36, 16, 16, [420 + 9 * i for i in range(32)]),
])
def test_noalloc_matches_workspace_path_twice(L, Hq, ps, lengths):
    w = synth.custom_workload("noalloc", L=L, Hq=Hq, Hkv=2, page_size=ps, lengths=lengths,
                              budget_frac=0.5, steps=4, seed=21, structured=True)
    B, L, Hkv, D = w.B, w.L, w.Hkv, 128
    c = md.Cache(L, Hq, Hkv, ps, B, w.max_pages_per_seq(), w.num_phys_pages())
    for r in range(7):
        c.set_region_params(r, w.base[r], w.half_life[r], bool(w.pinned[r]))
    for b in range(B):
        k, v = synth.kv_host(w.seed, b, L, Hkv, 0, w.n0(b), w.regions[b], True)
        c.append_tokens(b, w.regions[b], to_dev(k), to_dev(v))
    q = to_dev(synth.q_host(w.seed, B, L, Hq, Hkv, 1, True))
    kn, vn = synth.step_kv_host(w.seed, [w.n0(b) for b in range(B)], [6] * B, L, Hkv, True)
    out_ref = torch.empty((B, L, Hq, D), dtype=torch.int16, device="cuda")
    c.decode_step(B, q, to_dev(kn), to_dev(vn), [6] * B, out_ref)
    mass_ref = c.get_state(md.MD_STATE_MASS)
    pool = c.get_state(md.MD_STATE_POOL)
    bt = c.get_state(md.MD_STATE_BLOCK_TABLE)
    n_tok = np.array([c.query(md.MD_QUERY_TOKENS, b) for b in range(B)], np.int32)
    torch.cuda.synchronize()

    bt_h = bt.cpu().numpy()
    slots = np.concatenate([[bt_h[b, i // ps] * ps + i % ps for i in range(n_tok[b])] for b in range(B)])
    ref_o = synth.bf16_to_f64(out_ref.cpu().numpy().view(np.uint16))
    # the workspace path keeps the step's mass per token, summed over layers
    # and query heads, in fixed point (2^48 = 1.0)
    ref_m = mass_ref.cpu().numpy()[slots].astype(np.float64) * 2.0 ** -48
    stream = torch.cuda.current_stream().cuda_stream
    for call in range(2):
        out = torch.zeros_like(out_ref)
        mass = torch.zeros((L * Hkv, c.P_phys * ps), dtype=torch.float32, device="cuda")
        st = md.lib().md_attend_mass_noalloc(pool.data_ptr(), bt.data_ptr(), n_tok.ctypes.data, q.data_ptr(),
                                             out.data_ptr(), mass.data_ptr(), B, L, Hq, Hkv, ps,
                                             c.P_max, c.P_phys, stream)
        assert st == md.MD_OK, (call, st)
        torch.cuda.synchronize()
        got_o = synth.bf16_to_f64(out.cpu().numpy().view(np.uint16))
        assert np.max(np.abs(got_o - ref_o)) <= TOL_O_ABS, call
        got_m = mass.cpu().numpy()[:, slots].astype(np.float64).sum(axis=0)
        rel = np.max(np.abs(got_m - ref_m) / (np.abs(ref_m) + TOL_FLOOR))
        assert rel <= TOL_REL, (call, rel)
    c.close()


def test_noalloc_rejects_work_beyond_its_fixed_scratch():
    """Too many (sequence, layer, KV head) items for the fixed array: a clear
    capacity error before anything is launched."""
    dummy = torch.zeros(64, dtype=torch.int32, device="cuda")
    n_tok = np.full(256, 4096, np.int32)
    p = dummy.data_ptr()
    st = md.lib().md_attend_mass_noalloc(p, p, n_tok.ctypes.data, p, p, p, 256, 36, 16, 2, 16, 4096, 64, None)
    assert st == md.MD_ERR_CAPACITY
    # the 3B geometry's full trace, 32 x 1,700 tokens: two chunks per item
    # would need about 37 MiB of scores and partials
    n_tok2 = np.full(32, 1700, np.int32)
    st = md.lib().md_attend_mass_noalloc(p, p, n_tok2.ctypes.data, p, p, p, 32, 36, 16, 2, 16, 107, 64, None)
    assert st == md.MD_ERR_CAPACITY
    st = md.lib().md_attend_mass_noalloc(p, p, n_tok.ctypes.data, p, p, p, 1, 2, 16, 2, 24, 4096, 64, None)
    assert st == md.MD_ERR_INVALID_ARG
    torch.cuda.synchronize()
