"""Pins for the speculative-sampling oracle (CPU only).

What fixes the answer here is mathematics, not the oracle itself:
  * scipy's softmax and numpy's searchsorted (library routines);
  * the output law of speculative sampling: for emitted (y_1..y_{k+1}) with
    k accepted drafts, P = prod_{t<k} min(p_t, q_t)(y_{t+1}) times
    max(0, p_k - q_k)(y_{k+1}) if k < L, or p_L(y_{k+1}) if k = L; it is the
    statement that the target distribution is preserved (Sec. I, refs
    Leviathan et al. / Chen et al.), checked by exhaustive enumeration of
    draft sequences and uniform cells on tiny vocabularies;
  * the expected emitted length (1 - alpha^(L+1)) / (1 - alpha), Eq. (u_single);
  * Monte Carlo: emitted tokens ~ p (chi-square), acceptance = sum min(p, q).
"""
import itertools
import math

import numpy as np
import pytest
import scipy.special
import scipy.stats

from oracle import inverse_cdf, softmax, spec_verify, spec_verify_sparse
from oracle.spec_verify import residual


def test_softmax_matches_scipy_and_invariants():
    rng = np.random.default_rng(1)
    for scale in (0.1, 1.0, 3.0, 30.0):
        x = rng.normal(0, scale, size=(7, 513))
        p = softmax(x)
        np.testing.assert_allclose(p, scipy.special.softmax(x, axis=-1), rtol=1e-12, atol=1e-300)
        np.testing.assert_allclose(p.sum(-1), 1.0, atol=1e-12)
        np.testing.assert_allclose(softmax(x + 123.25), p, rtol=1e-12, atol=1e-300)
    # huge logits do not overflow
    p = softmax(np.array([[1e4, 1e4 - 1.0, -1e4]]))
    np.testing.assert_allclose(p[0, :2], scipy.special.softmax([0.0, -1.0]), rtol=1e-12)


def test_inverse_cdf_matches_searchsorted_and_skips_zero_weights():
    rng = np.random.default_rng(2)
    for _ in range(200):
        V = int(rng.integers(1, 40))
        w = rng.random(V) * (rng.random(V) < 0.6)
        if w.sum() == 0:
            w[rng.integers(V)] = 1.0
        u = float(rng.random())
        k = inverse_cdf(w, u)
        ref = int(np.searchsorted(np.cumsum(w), u * w.sum(), side="right"))
        assert k == min(ref, V - 1) or (ref >= V and w[k] > 0)
        assert w[k] > 0
    # uniform weights: k = floor(u * V)
    for u in (0.0001, 0.2499, 0.25 + 1e-9, 0.9999):
        assert inverse_cdf(np.ones(4), u) == math.floor(u * 4)


def test_residual_fallback_when_p_equals_q():
    p = scipy.special.softmax(np.array([0.3, -1.0, 2.0]))
    np.testing.assert_array_equal(residual(p, p.copy()), p)
    r = residual(p, scipy.special.softmax(np.array([0.3, -1.0, 1.0])))
    assert r[2] > 0 and r[0] == 0 and r[1] == 0


# ---------------------------------------------------------------------------
# exhaustive enumeration of the output law
# ---------------------------------------------------------------------------

def _cells(points):
    """Sorted sub-intervals of [0,1] cut at the given points, with their midpoints and widths."""
    pts = np.unique(np.clip(np.concatenate([[0.0, 1.0], points]), 0.0, 1.0))
    lo, hi = pts[:-1], pts[1:]
    keep = hi - lo > 0
    return (lo[keep] + hi[keep]) / 2, hi[keep] - lo[keep]


def _enumerated_law(zl, wl, L):
    """P(emitted sequence) by enumerating drafts and uniform cells through the oracle."""
    V = zl.shape[1]
    p = scipy.special.softmax(zl, axis=-1)
    q = scipy.special.softmax(wl, axis=-1) if L else np.zeros((0, V))
    with np.errstate(divide="ignore"):  # q(d) = 0: the ratio is +inf and min(1, .) = 1
        acc_cells = [_cells(np.minimum(1.0, p[t] / q[t])) for t in range(L)]
    res_cells = []
    for t in range(L + 1):
        pts = [np.cumsum(p[t])]
        if t < L:
            r = np.maximum(p[t] - q[t], 0)
            if r.sum() > 0:
                pts.append(np.cumsum(r) / r.sum())
        res_cells.append(_cells(np.concatenate(pts)))
    users_d, users_u, weights = [], [], []
    for drafts in itertools.product(range(V), repeat=L):
        w_d = np.prod([q[t, drafts[t]] for t in range(L)]) if L else 1.0
        if w_d == 0:
            continue
        for acc in itertools.product(*[range(len(c[0])) for c in acc_cells]):
            w_a = np.prod([acc_cells[t][1][acc[t]] for t in range(L)]) if L else 1.0
            for res in itertools.product(*[range(len(c[0])) for c in res_cells]):
                w_r = np.prod([res_cells[t][1][res[t]] for t in range(L + 1)])
                u = np.zeros((L + 1, 2))
                for t in range(L):
                    u[t, 0] = acc_cells[t][0][acc[t]]
                for t in range(L + 1):
                    u[t, 1] = res_cells[t][0][res[t]]
                users_d.append(drafts)
                users_u.append(u)
                weights.append(w_d * w_a * w_r)
    n = len(weights)
    out = spec_verify(np.full(n, L), np.tile(zl, (n, 1)), np.tile(wl, (n, 1)),
                      np.array(users_d, dtype=np.int64).reshape(-1),
                      np.concatenate(users_u))
    law = {}
    offs = out["out_offsets"]
    for i in range(n):
        seq = tuple(int(x) for x in out["out_tokens"][offs[i]:offs[i + 1]])
        law[seq] = law.get(seq, 0.0) + weights[i]
    return law, p, q


def _closed_form_law(p, q, L):
    V = p.shape[1]
    law = {}
    for k in range(L + 1):
        for seq in itertools.product(range(V), repeat=k + 1):
            pr = 1.0
            for t in range(k):
                pr *= min(p[t, seq[t]], q[t, seq[t]])
            last = max(0.0, p[k, seq[k]] - q[k, seq[k]]) if k < L else p[L, seq[k]]
            pr *= last
            if pr > 0:
                law[seq] = pr
    return law


@pytest.mark.parametrize("V,L,seed", [(3, 0, 0), (2, 1, 1), (4, 1, 2), (2, 2, 3), (3, 2, 4), (2, 3, 5)])
def test_output_law_matches_closed_form(V, L, seed):
    rng = np.random.default_rng(seed)
    zl = rng.normal(0, 1.5, size=(L + 1, V))
    wl = rng.normal(0, 1.5, size=(L, V))
    law, p, q = _enumerated_law(zl, wl, L)
    ref = _closed_form_law(p, q, L)
    assert set(k for k, v in law.items() if v > 1e-15) == set(ref)
    for k, v in ref.items():
        assert abs(law[k] - v) < 1e-12, (k, law[k], v)
    assert abs(sum(law.values()) - 1.0) < 1e-12
    # the first emitted token is exactly p_0-distributed (target law preserved)
    first = np.zeros(V)
    for k, v in law.items():
        first[k[0]] += v
    np.testing.assert_allclose(first, p[0], atol=1e-12)


def test_output_law_disjoint_and_identical_supports():
    # disjoint supports: every draft is rejected, the residual is p_0 itself
    zl = np.array([[0.0, 0.5, -1e4, -1e4], [0.0, 0.0, 0.0, 0.0]])
    wl = np.array([[-1e4, -1e4, 0.2, 0.0]])
    law, p, q = _enumerated_law(zl, wl, 1)
    assert all(len(s) == 1 for s in law)
    for k, v in law.items():
        assert abs(v - p[0, k[0]]) < 1e-12
    # identical p and q: every draft is accepted, the bonus comes from p_L
    zl = np.array([[0.1, 0.7, -0.3], [0.4, -0.2, 0.0], [1.0, 0.0, 0.5]])
    law, p, q = _enumerated_law(zl, zl[:2].copy(), 2)
    assert all(len(s) == 3 for s in law)
    ref = _closed_form_law(p, q, 2)
    for k, v in ref.items():
        assert abs(law[k] - v) < 1e-12


@pytest.mark.parametrize("L", [0, 1, 2])
def test_expected_length_closed_form_exact(L):
    """Eq. (u_single): E|emitted| = (1 - alpha^(L+1)) / (1 - alpha) for i.i.d. positions."""
    rng = np.random.default_rng(10 + L)
    z = rng.normal(0, 1, size=3)
    w = z + rng.normal(0, 0.8, size=3)
    law, p, q = _enumerated_law(np.tile(z, (L + 1, 1)), np.tile(w, (L, 1)), L)
    alpha = np.minimum(p[0], scipy.special.softmax(w)).sum()
    mean = sum(len(k) * v for k, v in law.items())
    assert abs(mean - (1 - alpha ** (L + 1)) / (1 - alpha)) < 1e-12


# ---------------------------------------------------------------------------
# Monte Carlo
# ---------------------------------------------------------------------------

def _mc_batch(rng, zl, wl, n):
    """n users sharing the same logits rows; drafts drawn from q with numpy."""
    L = wl.shape[0]
    q = scipy.special.softmax(wl, axis=-1)
    d = np.stack([rng.choice(q.shape[1], size=n, p=q[t]) for t in range(L)], axis=1) if L else \
        np.zeros((n, 0), dtype=np.int64)
    u = rng.random((n * (L + 1), 2))
    return spec_verify(np.full(n, L), np.tile(zl, (n, 1)), np.tile(wl, (n, 1)), d.reshape(-1), u)


def test_monte_carlo_target_law_and_acceptance():
    rng = np.random.default_rng(20)
    V, L, n = 16, 4, 100_000
    zl = rng.normal(0, 1.2, size=(L + 1, V))
    wl = zl[:L] + rng.normal(0, 0.9, size=(L, V))
    out = _mc_batch(rng, zl, wl, n)
    p = scipy.special.softmax(zl, axis=-1)
    q = scipy.special.softmax(wl, axis=-1)
    a = out["accept_len"]
    offs = out["out_offsets"]
    toks = out["out_tokens"]
    for k in range(L + 1):
        reached = np.flatnonzero(a >= k)
        obs = np.bincount(toks[offs[reached] + k], minlength=V)
        pv = scipy.stats.chisquare(obs, p[k] * reached.size).pvalue
        assert pv > 1e-4, (k, pv)
        if k < L:
            alpha = np.minimum(p[k], q[k]).sum()
            acc = np.mean(a[reached] > k)
            sd = math.sqrt(alpha * (1 - alpha) / reached.size)
            assert abs(acc - alpha) < 4 * sd, (k, acc, alpha)


@pytest.mark.parametrize("L", [0, 1, 4, 10])
def test_monte_carlo_expected_length(L):
    rng = np.random.default_rng(30 + L)
    V, n = 12, 60_000
    z = rng.normal(0, 1, size=V)
    w = z + rng.normal(0, 1.0, size=V)
    out = _mc_batch(rng, np.tile(z, (L + 1, 1)), np.tile(w, (L, 1)), n)
    alpha = np.minimum(scipy.special.softmax(z), scipy.special.softmax(w)).sum()
    lengths = out["accept_len"] + 1
    expect = (1 - alpha ** (L + 1)) / (1 - alpha)
    assert abs(lengths.mean() - expect) < 4 * lengths.std() / math.sqrt(n) + 1e-12


def test_truncation_and_packing_invariants():
    rng = np.random.default_rng(40)
    B, V = 300, 50
    L = rng.integers(0, 8, size=B)
    T = L + 1
    z = rng.normal(0, 1, size=(T.sum(), V))
    w = rng.normal(0, 1, size=(L.sum(), V))
    d = rng.integers(0, V, size=L.sum())
    u = rng.random((T.sum(), 2))
    out = spec_verify(L, z, w, d, u)
    a, offs, toks, acc = out["accept_len"], out["out_offsets"], out["out_tokens"], out["accepted"]
    assert offs[0] == 0 and np.all(np.diff(offs) == a + 1) and offs[-1] == len(toks)
    qo = lo = 0
    for i in range(B):
        assert 0 <= a[i] <= L[i]
        assert np.all(acc[qo:qo + a[i]])
        if a[i] < L[i]:
            assert not acc[qo + a[i]]
        np.testing.assert_array_equal(toks[offs[i]:offs[i] + a[i]], d[lo:lo + a[i]])
        assert not acc[qo + L[i]]  # bonus position carries no test
        qo += T[i]
        lo += L[i]


# ---------------------------------------------------------------------------
# sparse draft payload (spec_verify_sparse)
# ---------------------------------------------------------------------------

def _sparse_table(q):
    """(topk_idx, topk_q) rows of a dense draft distribution's support, padded
    with zero-probability entries on tokens outside the support."""
    K = int(max((q > 0).sum(axis=1).max(), 1)) if len(q) else 1
    idx = np.zeros((len(q), K), dtype=np.int64)
    val = np.zeros((len(q), K))
    for r in range(len(q)):
        sup = np.flatnonzero(q[r] > 0)
        off = [x for x in range(q.shape[1]) if x not in set(sup)]
        pad = off[:K - len(sup)]
        idx[r] = np.concatenate([sup, pad]).astype(np.int64)
        val[r, :len(sup)] = q[r, sup]
    return idx, val


def _enumerated_law_sparse(zl, q, L):
    """P(emitted sequence) by enumeration through spec_verify_sparse, q dense with zeros."""
    V = zl.shape[1]
    p = scipy.special.softmax(zl, axis=-1)
    acc_cells = [_cells(np.minimum(1.0, np.divide(p[t], q[t], out=np.ones(V), where=q[t] > 0))) for t in range(L)]
    res_cells = []
    for t in range(L + 1):
        pts = [np.cumsum(p[t])]
        if t < L:
            r = np.maximum(p[t] - q[t], 0)
            if r.sum() > 0:
                pts.append(np.cumsum(r) / r.sum())
        res_cells.append(_cells(np.concatenate(pts)))
    idx, val = _sparse_table(q)
    rows_d, rows_u, weights = [], [], []
    for drafts in itertools.product(range(V), repeat=L):
        w_d = np.prod([q[t, drafts[t]] for t in range(L)]) if L else 1.0
        if w_d == 0:
            continue
        for acc in itertools.product(*[range(len(c[0])) for c in acc_cells]):
            w_a = np.prod([acc_cells[t][1][acc[t]] for t in range(L)]) if L else 1.0
            for res in itertools.product(*[range(len(c[0])) for c in res_cells]):
                w_r = np.prod([res_cells[t][1][res[t]] for t in range(L + 1)])
                u = np.zeros((L + 1, 2))
                for t in range(L):
                    u[t, 0] = acc_cells[t][0][acc[t]]
                for t in range(L + 1):
                    u[t, 1] = res_cells[t][0][res[t]]
                rows_d.append(drafts)
                rows_u.append(u)
                weights.append(w_d * w_a * w_r)
    n = len(weights)
    d = np.array(rows_d, dtype=np.int64).reshape(-1)
    logq = np.log(np.tile(q, (n, 1))[np.arange(n * L), d]) if L else np.zeros(0)
    out = spec_verify_sparse(np.full(n, L), np.tile(zl, (n, 1)), d, logq, np.tile(idx, (n, 1)),
                             np.tile(val, (n, 1)), np.concatenate(rows_u))
    law = {}
    offs = out["out_offsets"]
    for i in range(n):
        seq = tuple(int(x) for x in out["out_tokens"][offs[i]:offs[i + 1]])
        law[seq] = law.get(seq, 0.0) + weights[i]
    return law, p


@pytest.mark.parametrize("V,L,K,seed", [(4, 1, 2, 11), (3, 2, 1, 12), (4, 2, 3, 13), (5, 1, 5, 14)])
def test_sparse_output_law_matches_closed_form(V, L, K, seed):
    """A draft distribution on K of V tokens: the enumerated output law equals
    prod_t min(p_t, q_t) x (residual or p), and the first token is p_0."""
    rng = np.random.default_rng(seed)
    zl = rng.normal(0, 1.5, size=(L + 1, V))
    q = np.zeros((L, V))
    for t in range(L):
        sup = rng.choice(V, size=K, replace=False)
        q[t, sup] = rng.dirichlet(np.ones(K))
    law, p = _enumerated_law_sparse(zl, q, L)
    ref = _closed_form_law(p, q, L)
    assert set(k for k, v in law.items() if v > 1e-15) == set(ref)
    for k, v in ref.items():
        assert abs(law[k] - v) < 1e-12, (k, law[k], v)
    first = np.zeros(V)
    for k, v in law.items():
        first[k[0]] += v
    np.testing.assert_allclose(first, p[0], atol=1e-12)


def test_sparse_with_full_support_equals_dense():
    """K = V, q = softmax(w), logq(d) = log q(d): spec_verify_sparse == spec_verify."""
    rng = np.random.default_rng(15)
    L = np.array([3, 0, 5, 2])
    V = 40
    z = rng.normal(0, 2, size=(int((L + 1).sum()), V))
    w = z[np.concatenate([np.arange(o, o + l) for o, l in zip(np.concatenate([[0], np.cumsum(L + 1)[:-1]]), L)])]
    w = w + rng.normal(0, 0.7, size=w.shape)
    q = scipy.special.softmax(w, axis=-1)
    d = np.array([rng.choice(V, p=q[r]) for r in range(len(q))])
    u = rng.random((len(z), 2))
    dense = spec_verify(L, z, w, d, u)
    idx = np.tile(np.arange(V), (len(q), 1))
    sparse = spec_verify_sparse(L, z, d, np.log(q[np.arange(len(q)), d]), idx, q, u)
    for key in ("accept_len", "out_offsets", "out_tokens", "accepted"):
        assert np.array_equal(dense[key], sparse[key]), key
