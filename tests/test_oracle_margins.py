"""Pins for the oracle's boundary-band code (CPU only).

The parity bar excuses a GPU/oracle mismatch only for a user with a decision
whose uniform lies within 1e-6 of what decides it: the acceptance ratio
p_t(d)/q_t(d) of a position that shaped the output, or an edge of the CDF
cell of the token sampled at a_i.  These tests fix, on values worked out by
hand, what the oracle reports as those distances and which positions count:

  * _cdf_margin(w, u, k): min(u*W - C_{k-1}, C_k - u*W) / W with C the
    cumulative weights, W = C_{V-1} and C_{-1} = 0;
  * margin_accept[n] = |u_acc - p_t(d)/q_t(d)| at draft positions, +inf at the
    bonus position;
  * decision_margins: the acceptance tests at t = 0 .. min(a_i, L_i - 1) (the
    accepted drafts and the first rejection) and the resample at a_i; tests at
    later positions never shaped the output and do not count.
"""
import numpy as np

from oracle import decision_margins, spec_verify
from oracle.spec_verify import _cdf_margin


def test_cdf_margin_three_tenths_of_a_millionth_from_an_edge():
    w = np.array([1.0, 2.0, 3.0, 4.0])  # cumulative 1, 3, 6, 10
    # u * W = 3 + 3e-6: token 2, 3e-6 above its lower edge C_1 = 3, i.e. 3e-7 of W
    u = 0.3 + 3e-7
    assert abs(_cdf_margin(w, u, 2) - 3e-7) < 1e-15
    # the same distance below the upper edge C_2 = 6
    u = 0.6 - 3e-7
    assert abs(_cdf_margin(w, u, 2) - 3e-7) < 1e-15


def test_cdf_margin_inside_a_cell_is_the_nearer_edge():
    w = np.array([1.0, 2.0, 3.0, 4.0])
    # u * W = 4: token 2 spans [3, 6); nearer edge 3, distance 1 = 0.1 of W
    assert abs(_cdf_margin(w, 0.4, 2) - 0.1) < 1e-15
    # u * W = 5.5: nearer edge 6, distance 0.5
    assert abs(_cdf_margin(w, 0.55, 2) - 0.05) < 1e-15
    # token 0 spans [0, 1): u * W = 0.2 is 0.2 from its lower edge 0
    assert abs(_cdf_margin(w, 0.02, 0) - 0.02) < 1e-15
    # last token spans [6, 10): u * W = 9.9 is 0.1 from W
    assert abs(_cdf_margin(w, 0.99, 3) - 0.01) < 1e-15
    # unnormalised weights give the same fractions
    assert abs(_cdf_margin(7.0 * w, 0.4, 2) - 0.1) < 1e-15


def test_margin_accept_is_the_distance_to_the_ratio():
    # p = (1/2, 1/2), q = (3/4, 1/4): draft token 0 has p/q = 2/3
    z = np.array([[0.0, 0.0], [0.0, 0.0]])
    w = np.array([[np.log(3.0), 0.0]])
    for delta, accepted in ((4e-7, False), (-4e-7, True), (0.1, False), (-0.25, True)):
        u = np.array([[2.0 / 3.0 + delta, 0.37], [0.5, 0.61]])
        r = spec_verify([1], z, w, [0], u)
        assert abs(r["margin_accept"][0] - abs(delta)) < 1e-13
        assert r["margin_accept"][1] == np.inf  # bonus position: no test
        assert bool(r["accepted"][0]) == accepted
        assert r["accept_len"][0] == (1 if accepted else 0)
    # rejected: residual max(0, p - q) = (0, 1/4), only token 1 has mass,
    # its cell is all of [0, W): margin min(u, 1 - u)
    u = np.array([[0.9, 0.37], [0.5, 0.61]])
    r = spec_verify([1], z, w, [0], u)
    assert r["out_tokens"].tolist() == [1]
    assert abs(r["margin_resample"][0] - 0.37) < 1e-13
    assert abs(r["resample_mass"][0] - 0.25) < 1e-13
    # accepted: bonus from p_1 = (1/2, 1/2) with u_res = 0.61: token 1, 0.11 from C_0 = 1/2
    u = np.array([[0.1, 0.37], [0.5, 0.61]])
    r = spec_verify([1], z, w, [0], u)
    assert r["out_tokens"].tolist() == [0, 1]
    assert abs(r["margin_resample"][0] - 0.11) < 1e-13


def _result(L, accept_len, margin_accept, margin_resample):
    return dict(accept_len=np.asarray(accept_len), margin_accept=np.asarray(margin_accept, dtype=float),
                margin_resample=np.asarray(margin_resample, dtype=float))


def test_decision_margins_count_only_decisions_that_shaped_the_output():
    far, near = 0.3, 5e-7
    L = [3, 3]
    inf = np.inf
    # user 0: a = 1 (position 0 accepted, position 1 rejected); user 1: a = 3 (all accepted)
    base = [far, far, far, inf, far, far, far, inf]
    assert not decision_margins(_result(L, [1, 3], base, [far, far]), L).any()

    # the rejecting position t = a_i is near the band: flagged
    m = list(base)
    m[1] = near
    assert decision_margins(_result(L, [1, 3], m, [far, far]), L).tolist() == [True, False]
    # an accepted position before it: flagged
    m = list(base)
    m[0] = near
    assert decision_margins(_result(L, [1, 3], m, [far, far]), L).tolist() == [True, False]
    # a position after the rejection never shaped the output: not flagged
    m = list(base)
    m[2] = near
    assert decision_margins(_result(L, [1, 3], m, [far, far]), L).tolist() == [False, False]
    # all accepted: the last draft position t = L_i - 1 counts
    m = list(base)
    m[6] = near
    assert decision_margins(_result(L, [1, 3], m, [far, far]), L).tolist() == [False, True]
    # the bonus position t = L_i holds no acceptance test: whatever it holds is ignored
    m = list(base)
    m[7] = near
    assert decision_margins(_result(L, [1, 3], m, [far, far]), L).tolist() == [False, False]
    # the resample at a_i
    assert decision_margins(_result(L, [1, 3], base, [far, near]), L).tolist() == [False, True]
    # the band is strict and scales with the argument
    assert not decision_margins(_result(L, [1, 3], base, [far, 1e-6]), L).any()
    assert decision_margins(_result(L, [1, 3], base, [far, 0.2]), L, band=0.25).tolist() == [False, True]


def test_decision_margins_with_no_drafts_and_offsets():
    # users with L = 0 have only the resample; offsets skip their one position
    L = [0, 2, 0, 1]
    a = [0, 0, 0, 1]
    m = [np.inf, 0.2, 0.2, np.inf, np.inf, 0.2, np.inf]
    assert not decision_margins(_result(L, a, m, [0.3] * 4), L).any()
    m2 = list(m)
    m2[2] = 1e-9  # user 1, position 1: after its rejection at t = 0
    assert not decision_margins(_result(L, a, m2, [0.3] * 4), L).any()
    m3 = list(m)
    m3[5] = 1e-9  # user 3, position 0: accepted, shaped the output
    assert decision_margins(_result(L, a, m3, [0.3] * 4), L).tolist() == [False, False, False, True]
    assert decision_margins(_result(L, a, m, [1e-8, 0.3, 0.3, 0.3]), L).tolist() == [True, False, False, False]
