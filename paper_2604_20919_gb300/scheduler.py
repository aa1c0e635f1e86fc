"""DiP-SD batch planning on the CPU (Sec. III, Algorithm 1): batch count N,
user-to-batch assignment x and integer draft lengths l that maximise the
throughput R = U / S of the pipelined rounds (Eq. R_def).

The system model is the paper's (Sec. II-B..II-F):
  * utility u_m(l) = (1 - a_m^(l+1)) / (1 - a_m) (Eq. u_single), U = sum_m u_m;
  * cost primitives F^d(i) (Eq. Fd), F^v(L, I) (Eq. Fv) and the affine
    latencies G_m(b, F) = c_m b F + beta_m, G^v(b, F) = c^v b F + beta^v
    (Eqs. Gm, Gv);
  * drafting tau_m = l_m G_m(1, F^d(i_m)) (Eq. C_tau_d); batch n is ready at
    t^d_n = max over its users of tau_m + tau^c_m (Eq. C_td) and verified in
    t^v_n = G^v(b_n, F^v(L_n, I_n)) with L_n, I_n the batch maxima (Eq. C_tv);
  * the span S of one round is the least value with S = sum_n T_n,
    T_n >= t^v_n and S >= t^d_n + t^v_n (Eqs. C_T_lb..C_precedence):
    S = max(sum_n t^v_n, max_n (t^d_n + t^v_n));
  * memory: Gamma_p + 4 J_v h1_v b_n I_n <= Gamma_max per batch (Eqs.
    C_mem_param..C_mem_total).

Solver (the structure of Algorithm 1, with exact sub-solvers of our own in
place of the MILPs the paper hands to SCIP): scan N = 2..M; for each N
alternate an x-step (minimise S for fixed l: local search over moves and
swaps of users between batches) and an l-step (maximise U / S for fixed x:
Dinkelbach's method, Eqs. dinkel..dinkel_stop, whose inner problem
max U - q S is solved exactly: per batch the draft lengths are determined by
the batch's longest draft L and its ready time D, dominated (L, D) options
are pruned, and the batches' options are combined as a multiple-choice
knapsack over their verification times); stop when l is unchanged and R no
longer improves; keep the best N (Eq. batch_select).  The alternation starts
from several initial draft lengths (7 as in Table 2, and 1, 3, L_ub), and the
best plan is refined by a local search on R itself (user moves and swaps,
each scored with its exact l-step), since the alternation alone can stop in a
local optimum.  On small instances the result equals the exhaustive optimum
of problem P.

Host-side planning only: it chooses the batches that dipsd_verify_batch
then verifies, one call per pipeline stage.
"""
from __future__ import annotations

import math
from dataclasses import dataclass
from typing import List, Optional, Sequence, Tuple


@dataclass(frozen=True)
class ModelDims:
    """(J, h1, h2): decoder blocks, hidden size, FFN hidden size (Table 1)."""
    J: int
    h1: int
    h2: int


# Table 2 defaults: Qwen3-1.7B drafting on the device, Qwen3-32B verifying.
DRAFT_QWEN3_1P7B = ModelDims(28, 2048, 6144)
VERIFY_QWEN3_32B = ModelDims(64, 5120, 25600)


@dataclass
class SystemParams:
    """Per-user and server parameters (Table 1; defaults of Table 2, times in
    ms, memory in bytes)."""
    prefix: List[int]                 # i_m
    alpha: List[float]                # a_m, in (0, 1)
    tau_c: List[float]                # tau^c_m
    c_draft: List[float]              # c_m
    beta_draft: List[float]           # beta_m
    c_verify: float = 1.2077e-11      # c^v
    beta_verify: float = 95.1074      # beta^v
    draft: ModelDims = DRAFT_QWEN3_1P7B
    verify: ModelDims = VERIFY_QWEN3_32B
    mem_cap: float = 8.0e10           # Gamma_max
    l_max: int = 20                   # L_ub

    @property
    def M(self) -> int:
        return len(self.prefix)

    @staticmethod
    def homogeneous(M: int, alpha: float = 0.78, prefix: int = 512, tau_c: float = 3.0,
                    c_draft: float = 4.0305e-11, beta_draft: float = 33.8151, **kw) -> "SystemParams":
        return SystemParams([prefix] * M, [alpha] * M, [tau_c] * M, [c_draft] * M, [beta_draft] * M, **kw)


# ----------------------------------------------------------------- model
def f_draft(d: ModelDims, i: int) -> float:
    """F^d(i) (Eq. Fd)."""
    return 4.0 * d.J * d.h1 * (2 * d.h1 + i + 1 + d.h2)


def f_verify(v: ModelDims, L: int, I: int) -> float:
    """F^v(L, I) (Eq. Fv)."""
    return 4.0 * v.J * v.h1 * L * (2 * v.h1 + I + L + v.h2)


def utility(alpha: float, l: int) -> float:
    """u(l) = (1 - a^(l+1)) / (1 - a) (Eq. u_single): expected emitted tokens."""
    return (1.0 - alpha ** (l + 1)) / (1.0 - alpha)


def draft_step_ms(p: SystemParams, m: int) -> float:
    """G_m(1, F^d(i_m)): one drafted token of user m (Eqs. Gm, C_tau_d)."""
    return p.c_draft[m] * f_draft(p.draft, p.prefix[m]) + p.beta_draft[m]


def verify_ms(p: SystemParams, b: int, L: int, I: int) -> float:
    """t^v = G^v(b, F^v(L, I)) (Eqs. Gv, C_tv)."""
    return p.c_verify * b * f_verify(p.verify, L, I) + p.beta_verify


def param_bytes(p: SystemParams) -> float:
    """Gamma_p (Eq. C_mem_param)."""
    v = p.verify
    return v.J * (8.0 * v.h1 ** 2 + 4.0 * v.h1 * v.h2)


def batch_fits(p: SystemParams, users: Sequence[int]) -> bool:
    """Memory feasibility of one batch (Eqs. C_mem_kv, C_mem_total)."""
    if not users:
        return False
    v = p.verify
    kv = 4.0 * v.J * v.h1 * len(users) * max(p.prefix[m] for m in users)
    return param_bytes(p) + kv <= p.mem_cap


@dataclass
class Plan:
    """A schedule: batches (lists of user indices, in stage order) and draft lengths."""
    batches: List[List[int]]
    draft_len: List[int]
    U: float = 0.0
    S: float = 0.0

    @property
    def N(self) -> int:
        return len(self.batches)

    @property
    def throughput(self) -> float:
        """R = U / S in tokens per ms (Eq. R_def); x 1000 for tokens/s."""
        return self.U / self.S if self.S > 0 else 0.0


def span(p: SystemParams, batches: Sequence[Sequence[int]], l: Sequence[int]) -> float:
    """S = max(sum_n t^v_n, max_n (t^d_n + t^v_n)) of a schedule (Eqs. C_td..C_precedence)."""
    tv_sum, worst = 0.0, 0.0
    for users in batches:
        L = max(l[m] for m in users)
        I = max(p.prefix[m] for m in users)
        tv = verify_ms(p, len(users), L, I)
        td = max(l[m] * draft_step_ms(p, m) + p.tau_c[m] for m in users)
        tv_sum += tv
        worst = max(worst, td + tv)
    return max(tv_sum, worst)


def evaluate(p: SystemParams, batches: Sequence[Sequence[int]], l: Sequence[int]) -> Plan:
    U = sum(utility(p.alpha[m], l[m]) for users in batches for m in users)
    return Plan([list(b) for b in batches], list(l), U, span(p, batches, l))


# ----------------------------------------------------------------- l-step
@dataclass
class _Option:
    L: int          # the batch's longest draft
    D: float        # the batch's ready time t^d_n
    U: float        # the batch's utility
    tv: float       # its verification time
    lens: Tuple[int, ...]


def _batch_options(p: SystemParams, users: Sequence[int]) -> List[_Option]:
    """Undominated (L, D) choices of one batch: for a cap L on the drafts and a
    ready time D (one user's tau_m + tau^c_m), every user takes the longest
    draft that meets both; an option is kept unless another has at least its
    utility with no larger verification time and no larger D + t^v."""
    I = max(p.prefix[m] for m in users)
    step = {m: draft_step_ms(p, m) for m in users}
    Ds = sorted({l * step[m] + p.tau_c[m] for m in users for l in range(1, p.l_max + 1)})
    opts = []
    for L in range(1, p.l_max + 1):
        tv = verify_ms(p, len(users), L, I)
        for D in Ds:
            lens = []
            for m in users:
                lm = min(L, int(math.floor((D - p.tau_c[m]) / step[m] + 1e-9)))
                if lm < 1:
                    break
                lens.append(lm)
            else:
                if max(lens) != L:
                    continue  # the cap is not reached: the same drafts under a smaller L cost less
                D_real = max(l * step[m] + p.tau_c[m] for l, m in zip(lens, users))
                if abs(D_real - D) > 1e-9:
                    continue
                opts.append(_Option(L, D, sum(utility(p.alpha[m], l) for l, m in zip(lens, users)), tv, tuple(lens)))
    # Pareto pruning on (U up, tv down, D + tv down)
    opts.sort(key=lambda o: (-o.U, o.tv, o.D + o.tv))
    kept: List[_Option] = []
    for o in opts:
        if any(k.U >= o.U and k.tv <= o.tv and k.D + k.tv <= o.D + o.tv for k in kept):
            continue
        kept.append(o)
    return kept


def _frontier(options: List[List[_Option]], cap: float):
    """All undominated (sum t^v, sum U) combinations of one option per batch,
    each option with D + t^v <= cap (multiple-choice knapsack frontier)."""
    front = [(0.0, 0.0, ())]
    for opts in options:
        allowed = [o for o in opts if o.D + o.tv <= cap + 1e-9]
        if not allowed:
            return []
        nxt = [(c + o.tv, u + o.U, pick + (o,)) for c, u, pick in front for o in allowed]
        nxt.sort(key=lambda t: (t[0], -t[1]))
        front = []
        best_u = -1.0
        for c, u, pick in nxt:
            if u > best_u + 1e-12:
                front.append((c, u, pick))
                best_u = u
    return front


def best_lengths(p: SystemParams, batches: Sequence[Sequence[int]], l0: Sequence[int],
                 tol: float = 1e-9, max_iter: int = 50) -> Plan:
    """l-step: draft lengths maximising U / S for a fixed assignment, by
    Dinkelbach's method (Eqs. dinkel..dinkel_stop).  The inner problem
    max U - q S is solved exactly: S = max(sum t^v, max (D + t^v)); for every
    candidate value of the second term the batches' options form a
    multiple-choice knapsack whose undominated frontier is enumerated."""
    options = [_batch_options(p, users) for users in batches]
    if any(not o for o in options):
        return evaluate(p, batches, l0)
    caps = sorted({o.D + o.tv for opts in options for o in opts})

    def inner(q: float):
        best = None
        for cap in caps:
            for c, u, pick in _frontier(options, cap):
                worst = max(o.D + o.tv for o in pick)
                S = max(c, worst)
                val = u - q * S
                if best is None or val > best[0] + 1e-12:
                    best = (val, u, S, pick)
        return best

    cur = evaluate(p, batches, l0)
    q = cur.throughput
    pick = None
    for _ in range(max_iter):
        val, u, S, pick = inner(q)
        if abs(val) <= tol * max(1.0, u):
            break
        q = u / S
    lens = list(l0)
    for users, o in zip(batches, pick):
        for m, lm in zip(users, o.lens):
            lens[m] = lm
    plan = evaluate(p, batches, lens)
    return plan if plan.throughput >= cur.throughput - 1e-15 else cur


# ----------------------------------------------------------------- x-step
def best_assignment(p: SystemParams, N: int, l: Sequence[int], start: Optional[List[List[int]]] = None,
                    max_rounds: int = 100) -> Optional[List[List[int]]]:
    """x-step: an assignment into N non-empty, memory-feasible batches with
    small span S for fixed draft lengths (local search: single-user moves and
    pairwise swaps, each taken when it lowers S, from `start` or from a
    round-robin deal of the users sorted by prefix length)."""
    M = p.M
    if N < 1 or N > M:
        return None
    if start is None:
        order = sorted(range(M), key=lambda m: (-p.prefix[m], -l[m], m))
        start = [[] for _ in range(N)]
        for k, m in enumerate(order):
            start[k % N].append(m)
    batches = [sorted(b) for b in start]
    if not all(batch_fits(p, b) for b in batches):
        return None

    def cost(bs):
        return span(p, bs, l), sum(verify_ms(p, len(b), max(l[m] for m in b), max(p.prefix[m] for m in b))
                                   for b in bs)

    best = cost(batches)
    for _ in range(max_rounds):
        improved = False
        for a in range(N):
            for m in list(batches[a]):
                if len(batches[a]) == 1:
                    break
                for b in range(N):
                    if b == a:
                        continue
                    cand = [list(x) for x in batches]
                    cand[a].remove(m)
                    cand[b] = sorted(cand[b] + [m])
                    if not (batch_fits(p, cand[a]) and batch_fits(p, cand[b])):
                        continue
                    cc = cost(cand)
                    if cc < best:
                        batches, best, improved = cand, cc, True
                        break
                if improved:
                    break
            if improved:
                break
        if improved:
            continue
        for a in range(N):
            for b in range(a + 1, N):
                for ma in batches[a]:
                    for mb in batches[b]:
                        cand = [list(x) for x in batches]
                        cand[a] = sorted([u for u in cand[a] if u != ma] + [mb])
                        cand[b] = sorted([u for u in cand[b] if u != mb] + [ma])
                        if not (batch_fits(p, cand[a]) and batch_fits(p, cand[b])):
                            continue
                        cc = cost(cand)
                        if cc < best:
                            batches, best, improved = cand, cc, True
                            break
                    if improved:
                        break
                if improved:
                    break
            if improved:
                break
        if not improved:
            break
    return batches


# ----------------------------------------------------------------- solver
def solve_fixed_n(p: SystemParams, N: int, l0: Optional[Sequence[int]] = None, max_outer: int = 30,
                  tol: float = 1e-12) -> Optional[Plan]:
    """P(N) (Eq. fixedN_ratio_obj): alternate the x-step and the l-step
    (Eqs. alt_x, alt_lm) from l0 (Table 2: 7) until l is unchanged and R no
    longer improves."""
    l = list(l0) if l0 is not None else [min(7, p.l_max)] * p.M
    batches = None
    plan = None
    for _ in range(max_outer):
        batches = best_assignment(p, N, l, start=batches)
        if batches is None:
            return None
        nxt = best_lengths(p, batches, l)
        if plan is not None and nxt.draft_len == plan.draft_len and nxt.throughput <= plan.throughput + tol:
            break
        plan = nxt
        l = nxt.draft_len
    return plan


def refine(p: SystemParams, plan: Plan, max_rounds: int = 50) -> Plan:
    """Local search on R itself: single-user moves and pairwise swaps between
    batches, each scored with its best draft lengths (the exact l-step), taken
    when R grows.  The alternation above minimises S for fixed l in its
    x-step, which can stop where moving a user would pay off only together
    with new draft lengths."""
    best = plan
    for _ in range(max_rounds):
        improved = False
        bs = best.batches
        N = len(bs)
        cands = []
        for a in range(N):
            for m in bs[a]:
                for b in range(N):
                    if b != a and len(bs[a]) > 1:
                        c = [list(x) for x in bs]
                        c[a].remove(m)
                        c[b] = sorted(c[b] + [m])
                        cands.append(c)
        for a in range(N):
            for b in range(a + 1, N):
                for ma in bs[a]:
                    for mb in bs[b]:
                        c = [list(x) for x in bs]
                        c[a] = sorted([x for x in c[a] if x != ma] + [mb])
                        c[b] = sorted([x for x in c[b] if x != mb] + [ma])
                        cands.append(c)
        for c in cands:
            if not all(batch_fits(p, x) for x in c):
                continue
            cand = best_lengths(p, c, best.draft_len)
            if cand.throughput > best.throughput * (1 + 1e-12):
                best, improved = cand, True
                break
        if not improved:
            break
    return best


def solve(p: SystemParams, n_range: Optional[Sequence[int]] = None, starts: Sequence[int] = (7, 1, 3, 20),
          refine_best: bool = True) -> Plan:
    """Algorithm 1: scan N (2..M by default), alternating from each initial
    draft length in `starts` (clipped to L_ub), keep the best (Eq.
    batch_select), then refine it with `refine`."""
    best = None
    inits = sorted({min(max(1, s), p.l_max) for s in starts}, key=lambda s: (s != 7, s))
    for N in (n_range if n_range is not None else range(2, p.M + 1)):
        for s in inits:
            plan = solve_fixed_n(p, N, [s] * p.M)
            if plan is not None and (best is None or plan.throughput > best.throughput + 1e-15):
                best = plan
    if best is None:
        raise ValueError("no memory-feasible schedule")
    return refine(p, best) if refine_best else best


# ----------------------------------------------------------------- baselines (Sec. IV-A)
def autoregressive(p: SystemParams) -> float:
    """AD: the server decodes each user alone, one token per forward (L = 1),
    users one after another: tokens per ms."""
    return p.M / sum(verify_ms(p, 1, 1, p.prefix[m]) for m in range(p.M))


def greedy_batches(p: SystemParams) -> List[List[int]]:
    """Users by prefix length, longest first, packed into a batch until the
    memory bound would be violated (Sec. IV-A, the greedy batching baseline)."""
    order = sorted(range(p.M), key=lambda m: (-p.prefix[m], m))
    batches: List[List[int]] = []
    for m in order:
        if batches and batch_fits(p, batches[-1] + [m]):
            batches[-1].append(m)
        else:
            batches.append([m])
    return batches


def autoregressive_greedy(p: SystemParams) -> float:
    """AD with greedy batching: one token per user per round, the greedy
    batches verified one after another with L = 1."""
    bs = greedy_batches(p)
    return p.M / sum(verify_ms(p, len(b), 1, max(p.prefix[m] for m in b)) for b in bs)


def without_batching(p: SystemParams) -> Plan:
    """DiP-SD without batching: N = M, one user per batch; only l is optimised."""
    return best_lengths(p, [[m] for m in range(p.M)], [min(7, p.l_max)] * p.M)


def fixed_lengths(p: SystemParams, l: int = 7) -> Plan:
    """DiP-SD with every l_m fixed (7 in the paper); only x (and N) is optimised."""
    best = None
    for N in range(2, p.M + 1):
        bs = best_assignment(p, N, [l] * p.M)
        if bs is None:
            continue
        plan = evaluate(p, bs, [l] * p.M)
        if best is None or plan.throughput > best.throughput:
            best = plan
    return best


# ----------------------------------------------------------------- command line
def main(argv: Optional[Sequence[str]] = None) -> dict:
    """Plans M users under Table 2's defaults (per-user acceptance rates and
    prefix lengths may be given) and prints one JSON line: the plan, its
    throughput and the Sec. IV-A baselines, all in tokens per second."""
    import argparse
    import json
    ap = argparse.ArgumentParser(prog="python -m paper_2604_20919_gb300.scheduler",
                                 description="DiP-SD batch planning (Algorithm 1) under the paper's latency model")
    ap.add_argument("--users", type=int, default=6, help="M")
    ap.add_argument("--alpha", type=float, nargs="+", default=[0.78], help="one acceptance rate, or one per user")
    ap.add_argument("--prefix", type=int, nargs="+", default=[512], help="one prefix length, or one per user")
    ap.add_argument("--l-max", type=int, default=20, help="L_ub")
    ap.add_argument("--mem-cap", type=float, default=8.0e10, help="Gamma_max in bytes")
    args = ap.parse_args(argv)
    M = args.users
    if M < 2:
        ap.error("--users must be at least 2 (the plan has N >= 2 batches)")

    def per_user(v, name):
        if len(v) == 1:
            return list(v) * M
        if len(v) != M:
            ap.error(f"--{name} takes 1 or {M} values")
        return list(v)

    p = SystemParams.homogeneous(M, l_max=args.l_max, mem_cap=args.mem_cap)
    p.alpha = per_user(args.alpha, "alpha")
    p.prefix = per_user(args.prefix, "prefix")
    plan = solve(p)
    out = {"throughput_tokens_per_s": 1000.0 * plan.throughput, "N": plan.N, "batches": plan.batches,
           "draft_len": plan.draft_len, "U": plan.U, "S_ms": plan.S,
           "baselines_tokens_per_s": {
               "AD": 1000.0 * autoregressive(p),
               "AD_greedy_batching": 1000.0 * autoregressive_greedy(p),
               "without_batching": 1000.0 * without_batching(p).throughput,
               "fixed_l7": 1000.0 * fixed_lengths(p, min(7, p.l_max)).throughput}}
    print(json.dumps(out))
    return out


if __name__ == "__main__":
    main()
