"""CPU checks of the seeded input generator (numpy side)."""
import numpy as np
import pytest
import torch

from synth import gen, workloads


def test_bf16_rounding_matches_torch_round_to_nearest_even():
    rng = np.random.default_rng(0)
    x = np.concatenate([rng.normal(size=20000).astype(np.float32) * 10,
                        np.array([0.0, -0.0, 1.0, 1.00390625, 1.01171875, 3.0e38, -1e-38], np.float32)])
    # values exactly half-way between two bf16 numbers (ties to even)
    base = rng.integers(0, 0x7F00, size=1000).astype(np.uint32) << 16
    halfway = (base | np.uint32(0x8000)).view(np.float32)
    x = np.concatenate([x, halfway]).astype(np.float32)
    mine = gen.f32_to_bf16_bits(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(mine, ref)
    back = gen.bf16_bits_to_f64(mine)
    np.testing.assert_array_equal(back, torch.from_numpy(x).to(torch.bfloat16).double().numpy())


def test_normal16_moments_and_range():
    h = gen.mix64(np.arange(200000, dtype=np.uint64))
    x = gen.normal16(h)
    assert x.min() >= -131070 and x.max() <= 131070
    assert abs(x.mean()) < 300
    assert x.std() == pytest.approx(gen.IH_SD, rel=0.01)


def test_rows_are_deterministic_and_position_addressable():
    m = workloads.small_model(123)
    tabs = gen.make_tables(m)
    seg = gen.segment_index(m, 0, 200)
    a = gen.hidden_rows(m, tabs, 0, 1, np.arange(0, 200), seg)
    b = gen.hidden_rows(m, tabs, 0, 1, [57, 3, 199], seg)
    np.testing.assert_array_equal(a[[57, 3, 199]], b)
    sp = gen.spike_flags(m, 0, 200)
    k = gen.kv_rows(m, tabs, 0, 0, np.arange(200), sp)
    k2 = gen.kv_rows(m, tabs, 0, 0, [5, 150], sp)
    np.testing.assert_array_equal(k[[5, 150]], k2)
    assert not np.array_equal(gen.kv_rows(m, tabs, 1, 0, [5], sp), k2[:1])   # another sequence
    assert not np.array_equal(gen.kv_rows(m, tabs, 0, 1, [5], sp), k2[:1])   # V differs from K


def test_trace_has_spikes_drift_and_band_a_jumps():
    m = gen.TraceModel(7)
    T = 6000
    sp = gen.spike_flags(m, 0, T)
    assert 0.012 < sp.mean() < 0.028 and not sp[0]
    seg = gen.segment_index(m, 0, T)
    assert np.all(np.diff(seg) >= 0) and seg[-1] == sp.sum()
    tabs = gen.make_tables(m)
    assert tabs.drift[10] < 0 < tabs.drift[21] and tabs.seg_amp[21] == 0 < tabs.seg_amp[10]
    # Band A change at a spike is ~4x the usual one, with no echo at t+1
    t_spike = int(np.nonzero(sp[100:])[0][0]) + 100
    pos = np.array([t_spike - 2, t_spike - 1, t_spike, t_spike + 1])
    rows = gen.bf16_bits_to_f64(gen.hidden_rows(m, tabs, 0, 10, pos, seg))
    g = np.linalg.norm(np.diff(rows, axis=0), axis=1)      # plain check of the recipe
    assert 3.0 < g[1] / g[0] < 5.5
    if not sp[t_spike + 1]:
        assert 0.6 < g[2] / g[0] < 1.6


def test_pyramid_budgets_recipe():
    from synth import workloads as W
    for k_mean, L in ((8192, 32), (4096, 32), (512, 32), (640, 4)):
        b = W.pyramid_budgets(k_mean, L)
        assert len(b) == L and all(x % 16 == 0 for x in b)
        assert all(x >= y for x, y in zip(b, b[1:]))                 # larger budgets for lower layers
        assert abs(sum(b) / L - k_mean) <= 8                          # the mean stays K (rounding to 16)
        assert b[0] == round(1.5 * k_mean / 16) * 16 and b[-1] == round(0.5 * k_mean / 16) * 16
    assert W.pyramid_budgets(100, 1) == (96,)


def test_host_twin_matches_numpy_generator_byte_for_byte():
    """The C twin of the generator (used by the oracle's full-size checks)
    gives the numpy generator's bytes: small and full model shapes, Band A
    layers with segment jumps, spike positions, unordered positions, another
    seed and sequence.  Built by the package build; skipped where it is not."""
    from synth import host
    if host.load() is None:
        pytest.skip("libepikv_synth_host.so not built")
    for m, seq in ((workloads.small_model(11), 0), (gen.TraceModel(0xE91C0003), 5), (gen.TraceModel(99), 2)):
        tabs = gen.make_tables(m)
        T = 3000
        sp = gen.spike_flags(m, seq, T)
        seg = gen.segment_index(m, seq, T)
        spike_pos = np.nonzero(sp)[0][:3]
        pos = np.concatenate([[0, 1, 2, T - 1, 777, 5], spike_pos, spike_pos + 1, np.arange(100, 170)])
        for kind in (0, 1):
            np.testing.assert_array_equal(host.kv_rows(m, tabs, seq, kind, pos, sp),
                                          gen.kv_rows(m, tabs, seq, kind, pos, sp))
        for layer in sorted({0, m.band_a[0], m.band_b[-1], m.num_layers - 1}):
            np.testing.assert_array_equal(host.hidden_rows(m, tabs, seq, layer, pos, seg),
                                          gen.hidden_rows(m, tabs, seq, layer, pos, seg))
