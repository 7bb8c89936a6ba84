"""The band-z tolerance's condition term (tests/harness.py): perturbing every
g value of a window by a relative error of at most u (fp32 roundoff) moves
the fp64 band-z score by no more than 2u * kappa(t), on well-spread windows
and on windows whose values nearly coincide (where kappa is huge)."""
import numpy as np

from oracle import epikv_oracle as O

from .harness import U32, bandz_condition_g


def _score_at(g_a, g_b, t, w):
    za = [[O.window_zscore(np.asarray(g[max(1, t - w + 1):t + 1]))] for g in g_a]
    zb = [[O.window_zscore(np.asarray(g[max(1, t - w + 1):t + 1]))] for g in g_b]
    return float(O.epiphany_score(za, zb)[0])


def test_rounding_of_g_stays_inside_the_condition_bound():
    rng = np.random.default_rng(5)
    T, w = 40, 16
    for trial in range(30):
        n_a, n_b = int(rng.integers(1, 4)), int(rng.integers(1, 4))
        spread = [10 ** float(rng.uniform(-6, 0)) for _ in range(n_a + n_b)]   # sigma / g from 1e-6 to 1
        gs = [np.concatenate([[np.nan], 16.0 * (1.0 + s * rng.standard_normal(T - 1))]) for s in spread]
        g_a, g_b = gs[:n_a], gs[n_a:]
        kappa = bandz_condition_g(g_a, g_b, w)
        for t in range(2, T):
            s0 = _score_at(g_a, g_b, t, w)
            for _ in range(3):
                pa = [g * (1.0 + U32 * rng.uniform(-1, 1, T)) for g in g_a]
                pb = [g * (1.0 + U32 * rng.uniform(-1, 1, T)) for g in g_b]
                assert abs(_score_at(pa, pb, t, w) - s0) <= 2.0 * U32 * kappa[t] + 1e-12
    assert kappa.max() > 1e5      # the ill-conditioned windows were reached
