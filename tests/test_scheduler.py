"""Batch planning (Algorithm 1 with exact sub-solvers) against the oracle and
the paper's printed results."""
import json
import os
import random

import pytest

import oracle.scheduler as osc
from paper_2604_20919_gb300 import scheduler as sc

GOLD = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "dipsd_paper_throughput.json")))


def _oracle_params(p: sc.SystemParams):
    P = osc.default_params(p.M)
    P.update(prefix=list(p.prefix), alpha=list(p.alpha), tau_c=list(p.tau_c), c_m=list(p.c_draft),
             beta_m=list(p.beta_draft), l_max=p.l_max, mem_cap=p.mem_cap)
    return P


@pytest.mark.parametrize("alpha", [0.70, 0.78, 0.95])
def test_homogeneous_plan_is_the_optimum(alpha):
    p = sc.SystemParams.homogeneous(6, alpha=alpha)
    plan = sc.solve(p)
    R_o = osc.homogeneous_optimum(_oracle_params(p))[0]
    assert plan.throughput == pytest.approx(R_o, rel=1e-12)
    # the plan is what it claims: re-evaluated by the oracle's own definitions
    assert osc.throughput(_oracle_params(p), plan.batches, plan.draft_len) == pytest.approx(plan.throughput,
                                                                                            rel=1e-12)
    assert sorted(m for b in plan.batches for m in b) == list(range(6))
    if alpha in (0.70, 0.95):
        key = "dipsd_alpha_0.70" if alpha == 0.70 else "dipsd_alpha_0.95"
        assert round(1000 * plan.throughput, 2) == GOLD["alpha_sweep_M6"][key]


def test_user_sweep_peak_speedup():
    """M = 14 (the sweep's largest, Sec. IV-B): 17.89x over AD."""
    p = sc.SystemParams.homogeneous(14)
    plan = sc.solve(p, starts=(7,), refine_best=False)
    assert round(plan.throughput / sc.autoregressive(p), 2) == GOLD["user_sweep"]["peak_speedup_vs_ad"]


def test_baseline_crossovers():
    """Fixed l = 7 overtakes AD with greedy batching between alpha 0.70 and 0.75,
    DiP-SD without batching between 0.85 and 0.90 (the paper: near 0.75, 0.85)."""
    def gap(alpha, fn):
        p = sc.SystemParams.homogeneous(6, alpha=alpha)
        return fn(p).throughput - sc.autoregressive_greedy(p)
    assert gap(0.70, sc.fixed_lengths) < 0 < gap(0.75, sc.fixed_lengths)
    assert gap(0.85, sc.without_batching) < 0 < gap(0.90, sc.without_batching)


def test_random_small_instances_match_exhaustive_search():
    rng = random.Random(7)
    for _ in range(12):
        M = rng.choice([2, 3, 4])
        lmax = rng.choice([3, 4, 5])
        scale = [rng.choice([0.2, 1.0, 3.0]) for _ in range(M)]
        p = sc.SystemParams([rng.choice([128, 512, 2048]) for _ in range(M)],
                            [rng.uniform(0.5, 0.95) for _ in range(M)], [rng.uniform(0.0, 20.0) for _ in range(M)],
                            [4.0305e-11 * s for s in scale], [33.8151 * s for s in scale], l_max=lmax)
        plan = sc.solve(p)
        R_o, part, l = osc.exhaustive(_oracle_params(p))
        assert plan.throughput == pytest.approx(R_o, rel=1e-12), (p, plan, part, l)


def test_memory_bound_is_respected():
    p = sc.SystemParams.homogeneous(5, l_max=4)
    J, h1 = p.verify.J, p.verify.h1
    p.mem_cap = sc.param_bytes(p) + 4.0 * J * h1 * 2 * 512 + 1.0  # two users' KV per batch
    plan = sc.solve(p)
    assert max(len(b) for b in plan.batches) <= 2
    R_o = osc.exhaustive(_oracle_params(p))[0]
    assert plan.throughput == pytest.approx(R_o, rel=1e-12)


def test_greedy_batching_packs_by_prefix():
    p = sc.SystemParams.homogeneous(4)
    p.prefix = [100, 800, 300, 500]
    assert sc.greedy_batches(p) == [[1, 3, 2, 0]]
    J, h1 = p.verify.J, p.verify.h1
    p.mem_cap = sc.param_bytes(p) + 4.0 * J * h1 * 2 * 800 + 1.0
    assert sc.greedy_batches(p) == [[1, 3], [2, 0]]


def test_command_line_plan(capsys):
    """`python -m paper_2604_20919_gb300.scheduler` prints the plan and the
    baselines; at M = 6, alpha = 0.95 they are the paper's printed figures."""
    out = sc.main(["--users", "6", "--alpha", "0.95"])
    printed = json.loads(capsys.readouterr().out.strip().splitlines()[-1])
    assert printed["N"] == out["N"] and printed["batches"] == out["batches"]
    gold = GOLD["alpha_sweep_M6"]
    assert round(out["throughput_tokens_per_s"], 2) == gold["dipsd_alpha_0.95"]
    base = out["baselines_tokens_per_s"]
    assert round(out["throughput_tokens_per_s"] / base["AD"], 2) == gold["speedup_vs_ad_alpha_0.95"]
    assert round(out["throughput_tokens_per_s"] / base["AD_greedy_batching"], 2) == \
        gold["speedup_vs_ad_greedy_alpha_0.95"]
    assert sorted(m for b in out["batches"] for m in b) == list(range(6))
    # per-user values: one per user, or the run stops with a usage error
    out = sc.main(["--users", "3", "--alpha", "0.7", "0.8", "0.9", "--prefix", "300", "500", "700"])
    assert sorted(m for b in out["batches"] for m in b) == [0, 1, 2]
    with pytest.raises(SystemExit):
        sc.main(["--users", "3", "--alpha", "0.7", "0.8"])
