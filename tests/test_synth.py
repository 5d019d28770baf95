"""The seeded input generator and the workload recipes (no GPU)."""
import numpy as np
import pytest

import synth


def test_host_generator_matches_numpy_restatement():
    regions = (np.arange(37) * 5 % 7).astype(np.uint8)
    for structured in (False, True):
        k, v = synth.kv_host(123, 5, 3, 2, 1000, 37, regions=regions, structured=structured)
        L, H, n, D = k.shape
        l, h, i, d = np.meshgrid(np.arange(L), np.arange(H), np.arange(n), np.arange(D), indexing="ij")
        kr = synth.key_bits_np(123, 5, l, h, 1000 + i, d, regions[i], structured=structured)
        vr = synth.bf16_rne_np(synth.normal_f32_np(123, synth.T_V, 5, l, h, 1000 + i, d))
        assert np.array_equal(k, kr) and np.array_equal(v, vr)
    q = synth.q_host(9, 3, 2, 8, 2, 17, structured=True)
    b, l, h, d = np.meshgrid(np.arange(3), np.arange(2), np.arange(8), np.arange(128), indexing="ij")
    qv = synth.normal_f32_np(9, synth.T_Q, b, l, h, 17, d)
    add = (np.float32(synth.KAPPA_STRUCT[8]) * synth.sign_np(9, l, h // 4, d)).astype(np.float32)
    qv = np.where(d < synth.STRUCT_DIMS, (qv + add).astype(np.float32), qv)
    assert np.array_equal(q, synth.bf16_rne_np(qv))


def test_generator_moments_and_independence():
    k, v = synth.kv_host(0, 0, 4, 2, 0, 2048)
    x = synth.bf16_to_f64(k).ravel()
    y = synth.bf16_to_f64(v).ravel()
    assert abs(x.mean()) < 0.01 and abs(x.std() - 1) < 0.01
    assert abs(np.corrcoef(x, y)[0, 1]) < 0.01
    k2, _ = synth.kv_host(1, 0, 4, 2, 0, 2048)
    assert not np.array_equal(k, k2)


def test_bf16_round_to_nearest_even():
    f = np.array([1.0, 1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, 1.0 + 2 ** -9, -2.5, 3.0e38], np.float32)
    bits = synth.bf16_rne_np(f)
    # 1+2^-8 is a tie between 1 and 1+2^-7: even mantissa wins (1.0);
    # 1+3*2^-8 ties between 1+2^-7 and 1+2^-6: even is 1+2^-6.
    assert list(bits[:4]) == [0x3F80, 0x3F80, 0x3F82, 0x3F80]
    assert synth.bf16_to_f64(bits)[4] == -2.5


def test_recipes():
    w0 = synth.make_workload(0)
    assert w0.n0(0) == 448 and w0.pages0(0) == 28 and w0.budget_pages == [14]
    assert synth.straddle_fraction(w0.regions[0], 16) == 0.0
    w1 = synth.make_workload(1)
    spans = np.bincount(w1.regions[0], minlength=7)
    assert list(spans) == [243, 182, 182, 122, 364, 364, 243]
    assert w1.pages0(0) == 107 and w1.budget_pages == [26] and w1.L == 28
    w2 = synth.make_workload(2)
    assert w2.B == 32 and all(w2.n0(b) == 1700 for b in range(32))
    for b in range(32):
        lab = w2.regions[b]
        assert np.all(np.diff(lab.astype(int)) >= 0)          # seven contiguous spans in order
        assert len(np.unique(lab)) == 7
        assert -255 <= int(w2.insert_steps[b][0]) <= 0
    w3 = synth.make_workload(3)
    assert w3.B == 64 and w3.window_k == 16 and w3.page_size == 16
    for b in (0, 63):
        lab = w3.regions[b]
        assert len(lab) == 32768 and np.all(lab[:512] == 0) and not np.any(lab[512:] == 0)
        assert np.all(np.diff(w3.insert_steps[b]) >= 0) and w3.insert_steps[b][-1] == -16
    w4 = synth.make_workload(4)
    assert w4.B == 16 and w4.page_size == 32 and w4.pages0(0) == 4096 and w4.budget_pages[0] == 204
    lab = w4.regions[3]
    assert len(lab) == 131072 and np.all(lab[:512] == 0) and not np.any(lab[512:] == 0)


def test_largest_remainder():
    assert synth.largest_remainder(10, [1, 1, 1]) == [4, 3, 3]
    parts = synth.largest_remainder(1700, [0.001, 5, 5, 5, 5, 5, 5], minimum=1)
    assert sum(parts) == 1700 and min(parts) >= 1
