"""Oracle for DiP-SD batch planning (Sec. II-B..II-F, problem P of Eq.
global_ratio).  Test infrastructure only: imported by tests/ alone.

Plain definitions written out from the paper, sharing no code with the
package's scheduler:
  * u(l) = (1 - a^(l+1)) / (1 - a)                      Eq. u_single
  * F^d(i) = 4 J_d h1_d (2 h1_d + i + 1 + h2_d)          Eq. Fd
  * F^v(L, I) = 4 J_v h1_v L (2 h1_v + I + L + h2_v)     Eq. Fv
  * G_m(b, F) = c_m b F + beta_m, G^v = c^v b F + beta^v Eqs. Gm, Gv
  * tau_m = l_m G_m(1, F^d(i_m))                         Eq. C_tau_d
  * t^d_n = max_{m in n} (tau_m + tau^c_m)               Eq. C_td (tightest)
  * t^v_n = G^v(b_n, F^v(max l, max i))                  Eq. C_tv
  * S = smallest sum_n T_n with T_n >= t^v_n and S >= t^d_n + t^v_n
      = max(sum_n t^v_n, max_n (t^d_n + t^v_n))          Eqs. C_T_lb..C_precedence
  * memory J_v (8 h1^2 + 4 h1 h2) + 4 J_v h1 b_n I_n <= cap   Eqs. C_mem_*
  * R = U / S                                            Eq. R_def

exhaustive(): the optimum of P by enumerating every N in 2..M, every set
partition of the users into N batches and every draft-length vector in
{1..l_max}^M (tiny M and l_max only).  homogeneous_optimum(): the same
optimum for identical users by a reduced enumeration: batch sizes (an integer
partition of M) and one length per batch.  The reduction is exact: with
identical users a batch's t^v and t^d depend only on its longest draft, so
raising every user of the batch to that length adds utility at no cost.
"""
from __future__ import annotations

import functools
import itertools


def u(alpha, l):
    return (1.0 - alpha ** (l + 1)) / (1.0 - alpha)


def F_d(J, h1, h2, i):
    return 4.0 * J * h1 * (2 * h1 + i + 1 + h2)


def F_v(J, h1, h2, L, I):
    return 4.0 * J * h1 * L * (2 * h1 + I + L + h2)


def default_params(M, alpha=0.78, prefix=512):
    """Table 2 defaults (times in ms, memory in bytes)."""
    return dict(prefix=[prefix] * M, alpha=[alpha] * M, tau_c=[3.0] * M, c_m=[4.0305e-11] * M,
                beta_m=[33.8151] * M, c_v=1.2077e-11, beta_v=95.1074, draft=(28, 2048, 6144),
                verify=(64, 5120, 25600), mem_cap=8.0e10, l_max=20)


def t_verify(P, b, L, I):
    return P["c_v"] * b * F_v(*P["verify"], L, I) + P["beta_v"]


def t_draft_token(P, m):
    return P["c_m"][m] * 1 * F_d(*P["draft"], P["prefix"][m]) + P["beta_m"][m]


def fits(P, users):
    J, h1, h2 = P["verify"]
    params = J * (8.0 * h1 * h1 + 4.0 * h1 * h2)
    kv = 4.0 * J * h1 * len(users) * max(P["prefix"][m] for m in users)
    return params + kv <= P["mem_cap"]


def span(P, batches, l):
    total, worst = 0.0, 0.0
    for users in batches:
        tv = t_verify(P, len(users), max(l[m] for m in users), max(P["prefix"][m] for m in users))
        td = max(l[m] * t_draft_token(P, m) + P["tau_c"][m] for m in users)
        total += tv
        worst = max(worst, td + tv)
    return max(total, worst)


def throughput(P, batches, l):
    """R = U / S in tokens per ms."""
    U = sum(u(P["alpha"][m], l[m]) for users in batches for m in users)
    return U / span(P, batches, l)


def set_partitions(items):
    """Every partition of `items` into non-empty blocks (block order ignored)."""
    if not items:
        yield []
        return
    first, rest = items[0], items[1:]
    for part in set_partitions(rest):
        for k in range(len(part)):
            yield part[:k] + [[first] + part[k]] + part[k + 1:]
        yield [[first]] + part


def exhaustive(P):
    """max R over N in 2..M, every partition into N memory-feasible batches
    and every l in {1..l_max}^M; returns (R, batches, l)."""
    M = len(P["prefix"])
    best = (0.0, None, None)
    for part in set_partitions(list(range(M))):
        if len(part) < 2 or not all(fits(P, b) for b in part):
            continue
        for l in itertools.product(range(1, P["l_max"] + 1), repeat=M):
            R = throughput(P, part, l)
            if R > best[0]:
                best = (R, part, list(l))
    return best


def integer_partitions(n, k, largest=None):
    """Non-increasing k-tuples of positive integers summing to n."""
    largest = n if largest is None else largest
    if k == 0:
        if n == 0:
            yield ()
        return
    for first in range(min(largest, n - (k - 1)), 0, -1):
        for rest in integer_partitions(n - first, k - 1, first):
            yield (first,) + rest


@functools.lru_cache(maxsize=None)
def _homogeneous_cached(key):
    return _homogeneous(dict(key))


def homogeneous_optimum(P):
    """max R for identical users: batch sizes and one draft length per batch;
    returns (R, sizes, lengths)."""
    key = tuple(sorted((k, tuple(v) if isinstance(v, list) else v) for k, v in P.items()))
    return _homogeneous_cached(key)


def _homogeneous(P):
    M = len(P["prefix"])
    a, i = P["alpha"][0], P["prefix"][0]
    step = t_draft_token(P, 0)
    best = (0.0, None, None)
    for N in range(2, M + 1):
        for sizes in integer_partitions(M, N):
            if not all(fits(P, list(range(b))) for b in sizes):
                continue
            # batches of equal size are interchangeable: each group of equal
            # sizes takes a multiset of lengths
            groups = [len(list(g)) for _, g in itertools.groupby(sizes)]
            per_group = [itertools.combinations_with_replacement(range(1, P["l_max"] + 1), k) for k in groups]
            for pick in itertools.product(*[list(g) for g in per_group]):
                Ls = [L for g in pick for L in g]
                tv = [t_verify(P, b, L, i) for b, L in zip(sizes, Ls)]
                S = max(sum(tv), max(L * step + P["tau_c"][0] + t for L, t in zip(Ls, tv)))
                R = sum(b * u(a, L) for b, L in zip(sizes, Ls)) / S
                if R > best[0]:
                    best = (R, sizes, Ls)
    return best


def autoregressive(P):
    """AD: one token per user per target forward (L = 1), users one by one."""
    M = len(P["prefix"])
    return M / sum(t_verify(P, 1, 1, P["prefix"][m]) for m in range(M))


def autoregressive_greedy(P):
    """AD with greedy batching: users by prefix length, longest first, packed
    into a batch until the memory bound would be violated; one L = 1 forward
    per batch per round."""
    M = len(P["prefix"])
    order = sorted(range(M), key=lambda m: (-P["prefix"][m], m))
    batches = []
    for m in order:
        if batches and fits(P, batches[-1] + [m]):
            batches[-1].append(m)
        else:
            batches.append([m])
    return M / sum(t_verify(P, len(b), 1, max(P["prefix"][m] for m in b)) for b in batches)
