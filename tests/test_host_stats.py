"""Host-side statistics of the library (no GPU): wdc_correlations, which the
Fig. 3a diagnostic uses, against scipy and against the oracle's own numpy
implementation (the two share no code)."""
import numpy as np
import pytest

from oracle import diagnostics as odg
from paper_2608_01845_gb300 import wdc


@pytest.mark.parametrize("n", [3, 22, 500])
def test_correlations_match_scipy_and_the_oracle(n):
    from scipy import stats
    g = np.random.default_rng(n)
    x = g.standard_normal(n)
    y = 0.6 * x + 0.8 * g.standard_normal(n)
    pe, sp = wdc.correlations(x, y)
    assert pe == pytest.approx(stats.pearsonr(x, y)[0], abs=1e-12)
    assert sp == pytest.approx(stats.spearmanr(x, y)[0], abs=1e-12)
    po, so = odg.correlations(x, y)
    assert pe == pytest.approx(po, abs=1e-12) and sp == pytest.approx(so, abs=1e-12)


def test_correlations_special_cases():
    x = np.arange(10.0)
    assert wdc.correlations(x, 3 * x + 1) == pytest.approx((1.0, 1.0))
    assert wdc.correlations(x, -x) == pytest.approx((-1.0, -1.0))
    # a monotone but non-linear relation: Spearman 1, Pearson below 1
    pe, sp = wdc.correlations(x, np.exp(x))
    assert sp == pytest.approx(1.0) and pe < 0.9
    # ties take average ranks (scipy's convention)
    from scipy import stats
    a = np.array([1.0, 2.0, 2.0, 3.0, 5.0, 5.0, 5.0])
    b = np.array([2.0, 1.0, 4.0, 3.0, 7.0, 6.0, 6.0])
    assert wdc.correlations(a, b)[1] == pytest.approx(stats.spearmanr(a, b)[0], abs=1e-12)
    assert np.isnan(wdc.correlations(np.ones(5), x[:5])[0])
    with pytest.raises(wdc.WdcError):
        wdc.correlations([1.0], [2.0])
