"""The batch-planning oracle against what the paper prints and against itself.

The paper gives no worked example of one schedule, but Sec. IV-B prints the
optimum throughput for homogeneous users under Table 2's parameters (M = 6,
alpha 0.70 and 0.95) and speedups over the two autoregressive baselines;
the oracle's exact optimum must reproduce them.  Closed forms and an
exhaustive search on tiny instances pin the rest."""
import json
import os

import pytest

import oracle.scheduler as osc

GOLD = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "dipsd_paper_throughput.json")))


def test_utility_is_the_geometric_sum():
    """Eq. u_single: one bonus token plus each of l drafts accepted with prob. a^k."""
    for a in (0.3, 0.78, 0.95):
        for l in range(0, 12):
            assert osc.u(a, l) == pytest.approx(sum(a ** k for k in range(l + 1)), rel=1e-12)
    assert osc.u(0.5, 0) == 1.0


def test_span_of_one_batch_and_of_a_pipeline():
    P = osc.default_params(2)
    l = [4, 2]
    one = osc.span(P, [[0, 1]], l)
    tv = osc.t_verify(P, 2, 4, 512)
    assert one == pytest.approx(4 * osc.t_draft_token(P, 0) + 3.0 + tv)
    two = osc.span(P, [[0], [1]], l)
    tv0, tv1 = osc.t_verify(P, 1, 4, 512), osc.t_verify(P, 1, 2, 512)
    assert two == pytest.approx(max(tv0 + tv1, 4 * osc.t_draft_token(P, 0) + 3.0 + tv0,
                                     2 * osc.t_draft_token(P, 1) + 3.0 + tv1))


def test_cost_primitives_by_hand():
    """Eqs. Fd, Fv at Table 2's model sizes, multiplied out by hand."""
    assert osc.F_d(28, 2048, 6144, 512) == 4 * 28 * 2048 * (4096 + 513 + 6144)
    assert osc.F_v(64, 5120, 25600, 8, 1024) == 4 * 64 * 5120 * 8 * (10240 + 1024 + 8 + 25600)


@pytest.mark.parametrize("alpha,key", [(0.70, "dipsd_alpha_0.70"), (0.95, "dipsd_alpha_0.95")])
def test_homogeneous_optimum_matches_the_paper(alpha, key):
    P = osc.default_params(6, alpha=alpha)
    R, sizes, Ls = osc.homogeneous_optimum(P)
    assert round(1000 * R, 2) == GOLD["alpha_sweep_M6"][key]


def test_speedups_over_the_baselines_match_the_paper():
    P = osc.default_params(6, alpha=0.95)
    R = osc.homogeneous_optimum(P)[0]
    g = GOLD["alpha_sweep_M6"]
    assert round(R / osc.autoregressive(P), 2) == g["speedup_vs_ad_alpha_0.95"]
    assert round(R / osc.autoregressive_greedy(P), 2) == g["speedup_vs_ad_greedy_alpha_0.95"]
    P = osc.default_params(6, alpha=0.78)
    R = osc.homogeneous_optimum(P)[0]
    assert round(R / osc.autoregressive_greedy(P), 2) == GOLD["default_alpha_M6"]["speedup_vs_ad_greedy"]


def test_reduced_enumeration_equals_full_enumeration():
    """For identical users the per-batch-length reduction finds the exhaustive optimum."""
    for M, lmax, a in ((3, 5, 0.7), (4, 4, 0.9), (3, 6, 0.5)):
        P = osc.default_params(M, alpha=a)
        P["l_max"] = lmax
        assert osc.homogeneous_optimum(P)[0] == pytest.approx(osc.exhaustive(P)[0], rel=1e-12)


def test_memory_bound_limits_batch_size():
    """Eq. C_mem_total: with room for two users' KV only, no batch holds three."""
    P = osc.default_params(4)
    J, h1, h2 = P["verify"]
    params = J * (8.0 * h1 * h1 + 4.0 * h1 * h2)
    P["mem_cap"] = params + 4.0 * J * h1 * 2 * 512 + 1.0
    P["l_max"] = 3
    R, part, l = osc.exhaustive(P)
    assert max(len(b) for b in part) <= 2
    assert not osc.fits(P, [0, 1, 2]) and osc.fits(P, [0, 1])
