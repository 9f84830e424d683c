"""Claims about the kernels' fp32 arithmetic that the design rests on, checked on the CPU in
numpy fp32 (each operation rounds to fp32; a fused multiply-add is formed exactly in fp64
and rounded once, which is exact for the fp32 operands used here).  No GPU and no oracle:
these check that a rearranged formula decides and rounds as the definition does.

- FWM's pass 2 reads one half-bin table entry per key, {alpha, beta, w^N}, indexed by
  q = floor(v) with v = 2u: q gives the bin r = q >> 1 and the Nearest endpoint (q + 1) >> 1
  with the decisions of r = floor(u), t = u - r, l = r + [t >= 1/2] (Sec. 3, "Reconstruction"),
  and w^L = alpha + v beta stays within a few fp32 units of e_r + t (e_{r+1} - e_r).
- Pass 1 at d = 64 compares the unscaled dot products and scales the row extrema once: the
  scale 2^-3 is exact, so the maximum, its lowest index and its tie count are those of the
  scaled scores for every score of magnitude 2^-123 or more.
"""
import numpy as np
import pytest

f32 = np.float32


def _fma32(a, b, c):
    return (np.float64(a) * np.float64(b) + np.float64(c)).astype(f32)


def _fwm_grid(K, tau):
    """The FWM grid values e_r = exp(-tau + r tau / K), r = 0..K, rounded to fp32 as the host does."""
    return np.array([np.exp(-tau + r * tau / K) for r in range(K + 1)]).astype(f32)


def _line_table(e, K):
    """Entries q = 0..2K of the half-bin table: r = min(q >> 1, K - 1), beta = (e_{r+1} - e_r) / 2,
    alpha = e_r - 2 r beta (one rounding), w^N = e_{(q + 1) >> 1}."""
    q = np.arange(2 * K + 1)
    r = np.minimum(q >> 1, K - 1)
    beta = (f32(0.5) * (e[r + 1] - e[r]).astype(f32)).astype(f32)
    alpha = _fma32((-2.0 * r).astype(f32), beta, e[r])
    return alpha, beta, e[(q + 1) >> 1]


@pytest.mark.parametrize("tau", [3.0, 6.0, 8.0])
@pytest.mark.parametrize("K", [1, 2, 4, 8, 16, 32, 64])
def test_fwm_half_bin_line_table(K, tau):
    rng = np.random.default_rng(K * 100 + int(tau))
    e = _fwm_grid(K, tau)
    alpha, beta, wN_tab = _line_table(e, K)
    # random positions in [0, K], every bin edge and midpoint, and the values just below them
    edges = np.arange(0, 2 * K + 1, dtype=np.float64) / 2
    u = np.concatenate([(rng.random(50000) * K), edges, np.nextafter(edges.astype(f32), f32(-1.0))]).astype(f32)
    u = u[(u >= 0) & (u <= K)]
    v = (f32(2.0) * u).astype(f32)  # exact
    q = np.floor(v).astype(np.int64)  # the round-down add of the kernel
    # the reference decisions: r = floor(u) clipped to K - 1, t = u - r, l = r + [t >= 1/2]
    r = np.minimum(np.floor(u).astype(np.int64), K - 1)
    t = (u - r.astype(f32)).astype(f32)
    ell = r + (t >= 0.5)
    assert np.array_equal(np.minimum(q >> 1, K - 1), r)
    assert np.array_equal((q + 1) >> 1, ell)
    assert np.array_equal(wN_tab[q], e[ell])  # w^N: the same fp32 value as the pair table's endpoint
    # w^L: the line form against the exact value of the same fp32 grid, and against the pair form
    wl_line = _fma32(v, beta[q], alpha[q])
    wl_pair = _fma32(t, (e[r + 1] - e[r]).astype(f32), e[r])
    exact = e[r].astype(np.float64) + (u.astype(np.float64) - r) * (e[r + 1].astype(np.float64) - e[r])
    rel_line = np.abs(wl_line - exact) / exact
    rel_pair = np.abs(wl_pair - exact) / exact
    assert rel_pair.max() <= 2.0 ** -23  # the pair form: about one rounding
    assert rel_line.max() <= 2.0e-6  # the line form: alpha's cancellation costs a few units
    assert np.abs(wl_line - exact).sum() / exact.sum() <= 2.0e-7  # over a row-like sum


def _row_stats(x):
    """Maximum, lowest index of it and tie count of a row."""
    m = x.max()
    hits = np.flatnonzero(x == m)
    return m, hits[0], hits.size


def test_pass1_unscaled_comparison_at_d64():
    rng = np.random.default_rng(7)
    scale = f32(0.125)  # 1 / sqrt(64)
    for trial in range(400):
        n = int(rng.integers(1, 1025))
        mag = 10.0 ** rng.uniform(-30, 3)
        acc = (rng.standard_normal(n) * mag).astype(f32)
        if trial % 3 == 0 and n > 3:  # exact duplicates, some at the maximum
            k = int(rng.integers(1, n))
            acc[rng.integers(0, n, k)] = acc[rng.integers(0, n)]
            acc[rng.integers(0, n)] = acc.max()
        scaled = (acc * scale).astype(f32)
        m_raw, a_raw, n_raw = _row_stats(acc)
        m_sc, a_sc, n_sc = _row_stats(scaled)
        assert f32(m_raw * scale) == m_sc
        assert (a_raw, n_raw) == (a_sc, n_sc)


def test_pass1_unscaled_comparison_limit():
    """Below 2^-123 the scaled scores are subnormal and two distinct dot products can round to the
    same scaled score: the only place the unscaled comparison could count a tie differently."""
    a = np.array([f32(2.0 ** -124), np.nextafter(f32(2.0 ** -124), f32(1.0))], dtype=f32)
    assert a[0] != a[1]
    assert f32(a[0] * f32(0.125)) == f32(a[1] * f32(0.125))
    b = np.array([f32(2.0 ** -123), np.nextafter(f32(2.0 ** -123), f32(1.0))], dtype=f32)
    assert f32(b[0] * f32(0.125)) != f32(b[1] * f32(0.125))
