"""The library's host-side Eq. 6-7 fit (md_calib_fit) against the oracle's
calibrate() on the same histograms (two independent implementations of the
count-weighted log-linear fit; no GPU needed)."""
import numpy as np

import oracle.memdecay_oracle as om
import paper_2607_10582_gb300 as md
from paper_2607_10582_gb300 import build as mdbuild


def test_library_fit_matches_oracle_fit():
    mdbuild.build()
    rng = np.random.default_rng(31)
    for trial in range(20):
        NB = 256
        cnt = rng.integers(0, 50, size=(7, NB)).astype(np.int64)
        cnt[:, rng.integers(5, NB):] = 0
        lam = rng.uniform(0.001, 0.08, size=7)
        ages = 4 * np.arange(NB) + 2.0
        mean = 0.01 * np.exp(-lam[:, None] * ages[None, :]) * np.exp(rng.normal(0, 0.3, (7, NB)))
        S = mean * cnt
        if trial == 3:
            cnt[4] = 0
            S[4] = 0
            cnt[5, 1] = 3
        rate, half = md.md_calib_fit(S, cnt)
        orate, ohalf = om.calibrate(S, cnt)
        assert np.array_equal(np.isnan(rate), np.isnan(orate))
        ok = ~np.isnan(orate)
        np.testing.assert_allclose(rate[ok], orate[ok], rtol=1e-9, atol=1e-14)
        np.testing.assert_allclose(half[ok], ohalf[ok], rtol=1e-9)
    # exact exponential: the library recovers the rate too
    S = np.zeros((7, 256))
    C = np.zeros((7, 256), np.int64)
    C[1, :40] = 9
    S[1, :40] = 9 * 0.02 * np.exp(-0.0433 * (4 * np.arange(40) + 2))
    rate, half = md.md_calib_fit(S, C)
    assert abs(rate[1] - 0.0433) < 1e-12 and abs(half[1] - np.log(2) / 0.0433) < 1e-9
