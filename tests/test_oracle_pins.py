"""Pins of the fp64 oracle to facts the paper and the mathematics fix.

None of these re-types the oracle's formula: each checks a closed form, an
invariant, a special case, brute force on a tiny input or a hand-worked
example (tests/golden/).  A dropped term, a wrong sign or index, a transposed
operand or a sample-vs-population std slip fails at least one of them.
"""
import itertools
import math
import os

import numpy as np
import pytest

from oracle import epikv_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ---------------------------------------------------------------- Eq. 1 (g)
def test_g_identical_rows_is_zero():
    h = np.random.default_rng(0).normal(size=64)
    assert O.hidden_change(h, h) == 0.0


@pytest.mark.parametrize("a", [1.0, -2.5, 1e-3, 7.0])
def test_g_one_hot_change_is_abs_amplitude(a):
    h0 = np.random.default_rng(1).normal(size=33)
    h1 = h0.copy()
    h1[17] += a
    assert O.hidden_change(h0, h1) == pytest.approx(abs(a), rel=1e-12)


def test_g_pythagorean_triple():
    h0 = np.zeros(8)
    h1 = np.zeros(8)
    h1[2], h1[5] = 3.0, -4.0
    assert O.hidden_change(h0, h1) == 5.0


def test_g_is_norm_of_difference_not_of_state():
    rng = np.random.default_rng(2)
    h0, h1 = rng.normal(size=(2, 40))
    off = 100.0 + rng.normal(size=40)          # large per-channel offset
    g = O.hidden_change(h0, h1)
    assert O.hidden_change(h0 + off, h1 + off) == pytest.approx(g, rel=1e-12)
    assert abs(g - np.linalg.norm(h1 + off)) > 100.0


def test_g_homogeneous_and_symmetric():
    rng = np.random.default_rng(3)
    h0, h1 = rng.normal(size=(2, 50))
    g = O.hidden_change(h0, h1)
    assert O.hidden_change(-3.0 * h0, -3.0 * h1) == pytest.approx(3.0 * g, rel=1e-12)
    assert O.hidden_change(h1, h0) == pytest.approx(g, rel=1e-15)


def test_g_trace_uses_previous_position():
    e = np.eye(4)[1]
    rows = np.stack([0 * e, 0 * e, e, e, 3 * e])
    g = O.hidden_change_trace(rows)
    assert np.isnan(g[0])
    np.testing.assert_array_equal(g[1:], [0.0, 1.0, 0.0, 2.0])


# ---------------------------------------------------------------- Eq. 3 (z)
def test_z_constant_signal_is_exactly_zero():
    g = np.full(300, 90.5)
    g[0] = np.nan
    assert np.all(O.rolling_zscore(g, 64) == 0.0)


@pytest.mark.parametrize("w", [64, 16])
@pytest.mark.parametrize("slope", [0.37, -2.0])
def test_z_linear_drift_closed_form_population_std(w, slope):
    # a full window of equally spaced values: z = sign(b) sqrt(3 (w-1)/(w+1))
    # with the population std; the sample std would give a different constant
    t = np.arange(400, dtype=np.float64)
    g = 5.0 + slope * t
    z = O.rolling_zscore(g, w, eps=1e-300)
    want = math.copysign(math.sqrt(3.0 * (w - 1) / (w + 1)), slope)
    np.testing.assert_allclose(z[w + 1:], want, rtol=1e-10)
    if w == 64:
        assert abs(want) == pytest.approx(1.7051957, abs=1e-7)
        sample = abs(want) * math.sqrt((w - 1) / w)
        assert abs(abs(z[200]) - sample) > 1e-2


def test_z_two_value_window_is_plus_minus_one():
    g = np.array([np.nan, 2.0, 5.0, 1.0])
    z = O.rolling_zscore(g, 64, eps=1e-300)
    assert z[0] == 0.0 and z[1] == 0.0      # no predecessor / single value
    assert z[2] == pytest.approx(1.0, rel=1e-15)
    # three values 2, 5, 1: mean 8/3, population std sqrt(26)/3
    assert z[3] == pytest.approx((1.0 - 8.0 / 3.0) / (math.sqrt(26.0) / 3.0), rel=1e-12)


def test_z_window_length_and_inclusion_of_t():
    w, p = 64, 200
    g = np.zeros(400)
    g[p] = 1.0
    z = O.rolling_zscore(g, w, eps=1e-300)
    # the spike as newest value: z = sqrt(w - 1)
    assert z[p] == pytest.approx(math.sqrt(w - 1), rel=1e-12)
    # the spike as oldest value (t = p + w - 1): z = -(1/w)/sqrt((1/w)(1 - 1/w))
    assert z[p + w - 1] == pytest.approx(-1.0 / math.sqrt(w - 1), rel=1e-12)
    # one step later the spike has left the window
    assert z[p + w] == 0.0
    assert z[p - 1] == 0.0


def test_z_ignores_position_zero_and_warms_up_on_available_count():
    g = np.array([1e9, 1.0, 2.0, 3.0, 4.0])
    z = O.rolling_zscore(g, 64, eps=1e-300)
    g2 = g.copy()
    g2[0] = -7.0
    np.testing.assert_array_equal(z, O.rolling_zscore(g2, 64, eps=1e-300))
    # t = 4 uses 1..4: mean 2.5, population std sqrt(1.25)
    assert z[4] == pytest.approx(1.5 / math.sqrt(1.25), rel=1e-12)


def test_z_affine_invariance():
    rng = np.random.default_rng(4)
    g = rng.gamma(4.0, 2.0, size=300)
    z = O.rolling_zscore(g, 64, eps=1e-300)
    np.testing.assert_allclose(O.rolling_zscore(3.5 * g + 11.0, 64, eps=1e-300), z, rtol=1e-9, atol=1e-9)


def test_z_causal():
    rng = np.random.default_rng(5)
    g = rng.normal(10, 1, size=200)
    z = O.rolling_zscore(g, 64)
    g2 = g.copy()
    g2[120:] = rng.normal(50, 9, size=80)
    np.testing.assert_array_equal(O.rolling_zscore(g2, 64)[:120], z[:120])


# ------------------------------------------------------- band combination
def test_band_swap_negates_and_singletons_reduce_to_difference():
    rng = np.random.default_rng(6)
    za, zb, zc = rng.normal(size=(3, 50))
    s = O.epiphany_score([za], [zb])
    np.testing.assert_array_equal(s, za - zb)
    np.testing.assert_array_equal(O.epiphany_score([zb], [za]), -s)
    # band means, not sums: a duplicated layer leaves the band mean unchanged
    np.testing.assert_allclose(O.epiphany_score([za, za], [zb, zc, zb, zc]),
                               za - 0.5 * (zb + zc), rtol=1e-12, atol=1e-12)


def test_bandz_scores_are_causal_and_zero_on_constant_change():
    rng = np.random.default_rng(7)
    T, D = 120, 16
    ra = [rng.normal(size=(T, D)) for _ in range(2)]
    rb = [rng.normal(size=(T, D)) for _ in range(3)]
    s = O.bandz_scores(ra, rb, w=8)
    ra2 = [r.copy() for r in ra]
    ra2[1][80:] += 5.0 * rng.normal(size=(T - 80, D))
    s2 = O.bandz_scores(ra2, rb, w=8)
    np.testing.assert_array_equal(s2[:80], s[:80])
    assert np.any(s2[80:] != s[80:])
    # a walk with constant step length gives g constant, so z = 0 and s = 0
    steps = np.zeros((T, D))
    steps[:, 0] = np.arange(T)
    assert np.all(O.bandz_scores([steps], [steps * 2.0], w=8) == 0.0)


# ---------------------------------------------------------------- Lag-KV
def _golden_lag():
    K, V, u, s = {}, {}, {}, {}
    with open(os.path.join(GOLDEN, "lagkv_hand_example.txt")) as f:
        for line in f:
            line = line.split("#")[0].split()
            if not line:
                continue
            tag, pos, vals = line[0], int(line[1]), [float(x) for x in line[2:]]
            {"K": K, "V": V, "u": u, "s": s}[tag][pos] = vals if tag in "KV" else vals[0]
    n = len(K)
    Kr = np.array([K[i] for i in range(n)]).reshape(n, 1, 1, 2)
    Vr = np.array([V[i] for i in range(n)]).reshape(n, 1, 1, 2)
    return Kr, Vr, np.array([u[i] for i in range(n)]), np.array([s[i] for i in range(n)])


def test_lagkv_hand_example_exact():
    K, V, u, s = _golden_lag()
    np.testing.assert_allclose(O.lag_variance_trace(K, V, lag=2, eps=1e-300), u, rtol=1e-15, atol=0)
    np.testing.assert_allclose(O.lagkv_scores(K, V, lag=2, eps=0.0, w=64), s, rtol=1e-14, atol=0)
    # with the default eps the values move by O(eps) only
    np.testing.assert_allclose(O.lagkv_scores(K, V, lag=2, w=64), s, rtol=1e-5, atol=1e-7)


def test_lagkv_uses_previous_chunk_only():
    rng = np.random.default_rng(8)
    T, lag = 64, 16
    K = rng.normal(size=(T, 2, 2, 8))
    V = rng.normal(size=(T, 2, 2, 8))
    u = O.lag_variance_trace(K, V, lag)
    assert np.all(u[:lag] == 0.0)
    t = 40                                   # chunk 2, previous chunk = 16..31
    for p in (t + 1, 47, 10, 33):            # same chunk, chunk 0, earlier in chunk 2
        K2 = K.copy()
        K2[p] *= 9.0
        assert O.lag_variance_trace(K2, V, lag)[t] == u[t]
    K3 = K.copy()
    K3[20, 0, 0, 3] = 50.0                   # inside the previous chunk: range changes
    assert O.lag_variance_trace(K3, V, lag)[t] != u[t]


def test_lagkv_per_channel_affine_invariance():
    rng = np.random.default_rng(9)
    T, lag = 48, 8
    K = rng.normal(size=(T, 2, 3, 8))
    V = rng.normal(size=(T, 2, 3, 8))
    a = rng.uniform(0.5, 3.0, size=(2, 3, 8))
    b = rng.normal(size=(2, 3, 8)) * 10
    u0 = O.lag_variance_trace(K, V, lag, eps=1e-300)
    u1 = O.lag_variance_trace(a * K + b, V * 2.0 - 1.0, lag, eps=1e-300)
    np.testing.assert_allclose(u1, u0, rtol=1e-10, atol=1e-13)


def test_lagkv_constant_previous_chunk_and_head_mean():
    lag = 2
    K = np.zeros((4, 1, 1, 4))
    V = np.zeros((4, 1, 1, 4))
    K[2] = 0.0                               # equals the constant previous range
    assert O.lag_variance_trace(K, V, lag)[2] == 0.0
    rng = np.random.default_rng(10)
    K = rng.normal(size=(40, 1, 1, 8))
    V = rng.normal(size=(40, 1, 1, 8))
    u1 = O.lag_variance_trace(K, V, 8)
    # a second identical head leaves the (layer, head) mean unchanged
    u2 = O.lag_variance_trace(np.concatenate([K, K], 2), np.concatenate([V, V], 2), 8)
    np.testing.assert_allclose(u2, u1, rtol=1e-14)
    # a head with zero normalised variance halves it
    Z = np.zeros_like(K)
    u3 = O.lag_variance_trace(np.concatenate([K, Z], 2), np.concatenate([V, Z], 2), 8)
    np.testing.assert_allclose(u3, 0.5 * u1, rtol=1e-14)


def test_rolling_mean_window():
    u = np.zeros(300)
    u[100] = 64.0
    s = O.rolling_mean(u, 64)
    assert s[99] == 0.0 and s[100] == 1.0 and s[163] == 1.0 and s[164] == 0.0
    u[10] = 11.0                             # warm-up: mean over the t + 1 available values
    assert O.rolling_mean(u, 64)[10] == 1.0
    np.testing.assert_allclose(O.rolling_mean(np.arange(3.0), 64), [0.0, 0.5, 1.0])


# ------------------------------------------------------ selection (App. D)
def _better(s, i, j):
    """True if slot i outranks slot j: higher score, NaN lowest, lower slot on ties."""
    a, b = s[i], s[j]
    if math.isnan(a) or math.isnan(b):
        return (not math.isnan(a)) or (math.isnan(b) and i < j)
    return a > b or (a == b and i < j)


def _brute_kept(s, K, P, cap):
    n = len(s)
    if n <= K:
        return list(range(n))
    P = min(P, n)
    R = min(min(cap, K // 4), max(0, K - P))
    M = max(0, K - P - R)
    cand = list(range(P, n - R))
    valid = []
    for S in itertools.combinations(cand, M):          # every M-subset
        rest = [j for j in cand if j not in S]
        if all(_better(s, i, j) for i in S for j in rest):
            valid.append(S)
    assert len(valid) == 1
    return sorted(set(range(P)) | set(range(n - R, n)) | set(valid[0]))


def test_select_equals_brute_force_on_tiny_inputs():
    rng = np.random.default_rng(11)
    for trial in range(300):
        n = int(rng.integers(1, 11))
        K = int(rng.integers(1, 10))
        P = int(rng.integers(0, 4))
        cap = int(rng.integers(0, 4))
        s = rng.integers(-2, 3, size=n).astype(np.float64)   # many ties
        if trial % 5 == 0:
            s[rng.integers(0, n)] = np.nan
        if trial % 7 == 0:
            s[s == 0] = -0.0
        assert O.select_kept(s, K, P, cap) == _brute_kept(list(s), K, P, cap)


def test_select_budget_protection_and_recency():
    rng = np.random.default_rng(12)
    s = rng.normal(size=700)
    kept = O.select_kept(s, 512, prefill=0)
    assert len(kept) == 512 and kept == sorted(kept)
    assert kept[-128:] == list(range(700 - 128, 700))        # R = min(128, 512/4)
    kept = O.select_kept(s, 100, prefill=7)
    assert len(kept) == 100
    assert kept[:7] == list(range(7)) and kept[-25:] == list(range(675, 700))  # R = 25
    assert O.select_kept(s[:90], 100) == list(range(90))
    # prefill larger than the budget is kept whole (R7)
    assert O.select_kept(s[:50], 10, prefill=20) == list(range(20))


def test_select_ties_nan_and_signed_zero():
    s = np.array([1.0, 0.0, -0.0, 0.0, np.nan, 2.0, -0.0, 5.0, 5.0, 5.0])
    # K = 6, R = 1 -> slot 9 always kept, M = 5 of slots 0..8
    assert O.select_kept(s, 6, 0, 128) == [0, 1, 5, 7, 8, 9]
    assert O.select_kept(s, 8, 0, 128) == [0, 1, 2, 3, 5, 7, 8, 9]


def test_compaction_preserves_order_and_bytes():
    rng = np.random.default_rng(13)
    rows = rng.integers(0, 2 ** 16, size=(300, 4, 2, 8), dtype=np.uint16)
    kept = O.select_kept(rng.normal(size=300), 200)
    assert all(k >= i for i, k in enumerate(kept))
    out = O.compact(rows, kept)
    assert out.shape == (200, 4, 2, 8)
    for i, k in enumerate(kept):
        assert out[i].tobytes() == rows[k].tobytes()


def test_simulate_decode_keeps_structure():
    rng = np.random.default_rng(14)
    L = 1000
    s = rng.normal(size=L)
    events, final = O.simulate_decode(s, L, 16, 256, 256 + 15, prefill=10)
    assert len(events) > 0
    for before, after in events:
        assert len(after) == 256
        assert after[:10] == list(range(10))
        assert after[-64:] == before[-64:]                   # R = min(128, 64)
        assert after == sorted(after)
    assert len(final) <= 256 + 15



# ------------------------------------- chunk-level selection (Sec. 5 future work)
def _golden_chunk_cases():
    pos = score = None
    cases = []
    with open(os.path.join(GOLDEN, "chunk_select_hand_example.txt")) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            head, *rest = line.split()
            if head == "pos":
                pos = [int(x) for x in rest]
            elif head == "score":
                score = [float(x) for x in rest]
            elif head == "case":
                K, P, cap, C = (int(x) for x in rest[:4])
                cases.append((K, P, cap, C, [int(x) for x in rest[5:]]))
    return pos, score, cases


def test_chunked_select_hand_example():
    pos, score, cases = _golden_chunk_cases()
    assert len(cases) == 3
    for K, P, cap, C, kept in cases:
        assert O.select_kept_chunked(score, pos, K, P, cap, C) == kept


def test_chunked_select_with_unit_chunks_is_the_token_rule():
    rng = np.random.default_rng(21)
    for trial in range(200):
        n = int(rng.integers(1, 60))
        s = rng.integers(-3, 4, size=n).astype(np.float64)
        if trial % 3 == 0:
            s[rng.integers(0, n, size=3)] = np.nan
        if trial % 4 == 0:
            s[s == 0] = -0.0
        pos = np.cumsum(rng.integers(1, 4, size=n)) - 1
        K, P, cap = int(rng.integers(1, 40)), int(rng.integers(0, 6)), int(rng.integers(0, 10))
        assert O.select_kept_chunked(s, pos, K, P, cap, 1) == O.select_kept(s, K, P, cap)


def _brute_chunked(s, pos, K, P, cap, C):
    """Every M-subset of the candidates is tried; the kept one is the unique
    subset whose every member outranks every other candidate when a slot is
    valued by its chunk's exact (rational) mean, NaN lowest, lower slot on
    ties -- whole chunks in rank order, the boundary chunk's lowest slots."""
    from fractions import Fraction
    n = len(s)
    if n <= K:
        return list(range(n))
    P = min(P, n)
    R = min(min(cap, K // 4), max(0, K - P))
    M = max(0, K - P - R)
    cand = list(range(P, n - R))
    val = {}
    for i in cand:
        mates = [j for j in cand if pos[j] // C == pos[i] // C]
        if any(math.isnan(s[j]) for j in mates):
            val[i] = None
        else:
            val[i] = sum(Fraction(s[j]) for j in mates) / len(mates)

    def better(i, j):
        a, b = val[i], val[j]
        if a is None or b is None:
            return (a is not None) or (b is None and i < j)
        return a > b or (a == b and i < j)

    valid = [S for S in itertools.combinations(cand, M)
             if all(better(i, j) for i in S for j in cand if j not in S)]
    assert len(valid) == 1
    return sorted(set(range(P)) | set(range(n - R, n)) | set(valid[0]))


def test_chunk_mean_is_the_float64_mean_not_a_float32_one():
    """R18's chunk score is the members' mean itself: two chunks whose means
    differ by 2^-32 (indistinguishable once rounded to float32, where the
    earlier chunk would win the tie) rank by the exact difference, and the
    mean of members whose float32 running sum loses the small one keeps it."""
    # slots 0, 1 -> chunk 0 (mean 2); slots 2, 3 -> chunk 1 (mean 2 + 2^-32); slots 4.. recency
    s = [1.0, 3.0, 2.0 + 2.0 ** -30, 2.0 - 2.0 ** -31, 0.0, 0.0]
    pos = [0, 1, 2, 3, 4, 5]
    # K = 4: R = 1 (one recency slot), M = 3 -> chunk 1 whole, then chunk 0's lowest slot
    assert O.select_kept_chunked(s, pos, 4, 0, 1, 2) == [0, 2, 3, 5]
    assert np.float32(s[2]) == np.float32(s[3]) == np.float32(2.0)   # a float32 mean would tie at 2
    assert O.chunk_mean([1e8, 1.0, -1e8]) == pytest.approx(1.0 / 3.0, rel=1e-15)   # float32: 0 / 3
    assert math.isnan(O.chunk_mean([1.0, float("nan")]))


def test_chunked_select_equals_brute_force_on_tiny_inputs():
    rng = np.random.default_rng(22)
    for trial in range(300):
        n = int(rng.integers(1, 12))
        K = int(rng.integers(1, 10))
        P = int(rng.integers(0, 3))
        cap = int(rng.integers(0, 4))
        C = int(rng.integers(2, 5))
        pos = list(np.cumsum(rng.integers(1, 4, size=n)) - 1)
        s = (rng.integers(-4, 5, size=n) / 2.0).astype(np.float64)   # exact halves, many ties
        if trial % 6 == 0:
            s[rng.integers(0, n)] = np.nan
        assert O.select_kept_chunked(s, pos, K, P, cap, C) == _brute_chunked(list(s), pos, K, P, cap, C)


def test_chunked_select_structure_on_decode_histories():
    """Along a decode with evictions every 16 tokens: K kept, prefill and the
    recency window kept, every candidate chunk kept whole or dropped whole
    except one, whose kept members are its lowest slots, and no dropped chunk
    outranks a kept one."""
    rng = np.random.default_rng(23)
    for C in (2, 5, 16):
        L, K, P = 900, 160, 6
        s = rng.normal(size=L)
        events, final = O.simulate_decode(s, L, 16, K, K + 15, prefill=P, select_chunk=C)
        assert len(events) > 10
        for before, after in events:
            n = len(before)
            R = min(128, K // 4)
            assert len(after) == K and after == sorted(after)
            assert after[:P] == list(range(P)) and after[-R:] == before[-R:]
            kept = set(after)
            chunks = {}
            for p in before[P:n - R]:
                chunks.setdefault(p // C, []).append(p)
            partial = 0
            kept_means, dropped_means = [], []
            for c, members in chunks.items():
                k = [p for p in members if p in kept]
                m = math.fsum(s[p] for p in members) / len(members)
                if k and len(k) < len(members):
                    partial += 1
                    assert k == members[:len(k)]
                if k:
                    kept_means.append(m)
                else:
                    dropped_means.append(m)
            assert partial <= 1
            if kept_means and dropped_means:
                assert min(kept_means) >= max(dropped_means) - 1e-6


# ------------------------------------------ per-layer budgets (Sec. 5 future work)
def test_layer_budgets_hand_example():
    events_expected = {}
    with open(os.path.join(GOLDEN, "layer_budgets_hand_example.txt")) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            head, *rest = line.split()
            if head == "score":
                score = [float(x) for x in rest]
            elif head == "setup":
                chunk, trigger, P, *budgets = (int(x) for x in rest)
            elif head == "event":
                events_expected[(int(rest[0]), int(rest[2]))] = [int(x) for x in rest[4:]]
    events, final = O.simulate_decode_layers(score, len(score), chunk, budgets, trigger, prefill=P)
    assert len(events) == 2
    for (e, l), after in events_expected.items():
        assert events[e][1][l] == after


def test_equal_layer_budgets_are_the_token_rule():
    rng = np.random.default_rng(31)
    for trial in range(20):
        L = 1000
        s = rng.normal(size=L)
        if trial % 4 == 0:
            s[rng.integers(0, L, size=20)] = np.nan
        K, P = int(rng.integers(20, 300)), int(rng.integers(0, 12))
        chunk = int(rng.integers(1, 40))
        trig = K + int(rng.integers(0, 30))
        ev1, fin1 = O.simulate_decode(s, L, chunk, K, trig, prefill=P)
        evl, finl = O.simulate_decode_layers(s, L, chunk, [K] * 3, trig, prefill=P)
        assert [a for _, a in ev1] == [a[0] for _, a in evl] == [a[2] for _, a in evl]
        assert finl == [fin1] * 3


def _brute_layer(s, K, P, R):
    n = len(s)
    P = min(P, n)
    M = max(0, K - P - R)
    cand = list(range(P, n - R))
    valid = [S for S in itertools.combinations(cand, min(M, len(cand)))
             if all(_better(s, i, j) for i in S for j in cand if j not in S)]
    assert len(valid) == 1
    return sorted(set(range(P)) | set(range(n - R, n)) | set(valid[0]))


def test_layer_selection_equals_brute_force_on_tiny_inputs():
    rng = np.random.default_rng(32)
    for trial in range(300):
        n = int(rng.integers(1, 11))
        P = int(rng.integers(0, 3))
        R = int(rng.integers(0, max(1, n - min(P, n) + 1)))
        K = int(rng.integers(1, 12))
        s = rng.integers(-2, 3, size=n).astype(np.float64)
        if trial % 5 == 0:
            s[rng.integers(0, n)] = np.nan
        assert O.select_kept_layer(s, K, P, R) == _brute_layer(list(s), K, P, R)


def test_layer_caches_stay_nested_on_decode_histories():
    """With one recency window and common events, a layer's cache after every
    event is its own budget's selection from any larger layer's cache, so the
    caches are nested; each keeps the prefill, the shared window and exactly
    min(size, K_l) tokens."""
    rng = np.random.default_rng(33)
    for trial in range(12):
        L = 1200
        s = rng.normal(size=L)
        n_layers = int(rng.integers(2, 6))
        budgets = [int(x) for x in rng.integers(40, 400, size=n_layers)]
        P = int(rng.integers(0, 10))
        chunk = int(rng.integers(1, 50))
        trig = max(budgets) + int(rng.integers(0, 40))
        events, final = O.simulate_decode_layers(s, L, chunk, budgets, trig, prefill=P)
        assert len(events) >= 2
        order = sorted(range(n_layers), key=lambda l: -budgets[l])
        for before, after in events:
            n = max(len(b) for b in before)
            R = min(min(128, min(budgets) // 4), max(0, min(budgets) - min(P, n)))
            for l in range(n_layers):
                assert len(after[l]) == min(len(before[l]), budgets[l])
                assert after[l][:P] == list(range(min(P, n)))
                if R:
                    assert after[l][-R:] == before[l][-R:] == before[order[0]][-R:]
            for a, b in zip(order, order[1:]):
                big, small = after[a], after[b]
                assert set(small) <= set(big)
                sel = O.select_kept_layer([s[p] for p in big], budgets[b], P, R)
                assert [big[i] for i in sel] == small

# ------------------------------------------- the other attention-free variants
def test_hsvar_closed_forms():
    # a walk with constant step a in Band A and b in Band B: g-bar = a, b
    T, D = 150, 8
    ra = np.zeros((T, D)); ra[:, 0] = 3.0 * np.arange(T)
    rb = np.zeros((T, D)); rb[:, 1] = 0.5 * np.arange(T)
    s = O.hsvar_scores([ra], [rb], w=16)
    assert s[0] == 0.0
    np.testing.assert_allclose(s[1:], 2.5, rtol=1e-14)
    # linear drift with a full window: mean = a + b (t - (w - 1) / 2)
    t = np.arange(300, dtype=np.float64)
    g = 2.0 + 0.25 * t
    m = O.rolling_band_mean(g, 64)
    np.testing.assert_allclose(m[70:], 2.0 + 0.25 * (t[70:] - 31.5), rtol=1e-13)
    # warm-up averages positions 1..t only, never position 0
    g2 = np.array([1e9, 1.0, 2.0, 6.0])
    np.testing.assert_allclose(O.rolling_band_mean(g2, 64), [0.0, 1.0, 1.5, 3.0])
    # swapping the bands negates the score
    rng = np.random.default_rng(15)
    A, B = rng.normal(size=(2, 90, 12))
    np.testing.assert_allclose(O.hsvar_scores([B], [A], 8), -O.hsvar_scores([A], [B], 8), rtol=1e-13)


def test_head_variance_closed_forms_and_equivariance():
    x = np.zeros((1, 1, 8))
    x[0, 0, 3] = 4.0                             # one-hot: var = a^2 (d - 1) / d^2
    assert O.head_variance(x) == pytest.approx(16.0 * 7 / 64, rel=1e-15)
    assert O.head_variance(np.full((2, 3, 16), 7.5)) == 0.0
    rng = np.random.default_rng(16)
    X = rng.normal(size=(2, 3, 16))
    v = O.head_variance(X)
    assert O.head_variance(-2.0 * X + 100.0) == pytest.approx(4.0 * v, rel=1e-12)
    # mean over (layer, head), not a sum: a duplicated head keeps it
    assert O.head_variance(np.concatenate([X, X], axis=1)) == pytest.approx(v, rel=1e-14)
    s = O.kv_variance_scores(np.stack([X, 2 * X, 3 * X]), w=64)
    np.testing.assert_allclose(s, [v, 2.5 * v, 14.0 / 3.0 * v], rtol=1e-12)


def test_lag_key_is_the_key_half_of_lagkv():
    K, V, u, _ = _golden_lag()
    # the hand example's V terms vanish at t = 2, 3 and equal 1/4 at t = 4
    uk = [O.lag_key_token_variance(K[t], K[(t // 2 - 1) * 2:(t // 2) * 2], 1e-300) for t in (2, 3, 4)]
    np.testing.assert_allclose(uk, [1 / 64, 1 / 4, 1 / 4], rtol=1e-14)
    rng = np.random.default_rng(17)
    K = rng.normal(size=(64, 2, 2, 8))
    V = rng.normal(size=(64, 2, 2, 8))
    both = O.lagkv_scores(K, V, lag=8)
    np.testing.assert_allclose(O.lag_key_scores(K, lag=8) + O.lag_key_scores(V, lag=8), both, rtol=1e-12)
    np.testing.assert_array_equal(O.lag_key_scores(K, lag=8)[:8], 0.0)
