"""Oracle for the speculative-sampling step (test infrastructure only).

Stage 2 of the paper's four-stage round (Sec. II-A): the server checks each
user's L_i draft tokens with the target distribution, finds the first
mismatched (rejected) draft, discards everything after it, and emits one
more token after the last accepted position, so every round emits at least
one token.  The paper delegates the accept/reject rule to the speculative
sampling it cites (Leviathan et al., ICML 2023; Chen et al., 2023), which
keeps the target distribution exactly; Eq. (u_single) is its expected
output length under i.i.d. acceptance alpha.  The steps, per user i, in
that method's order (positions t = 0 .. L_i; draft d_{t+1} was proposed at
position t):

  1. p_t = softmax(z_t) for every verify position, q_t = softmax(w_t) for
     every draft position (temperature 1, full vocabulary).
  2. draft d_{t+1} is accepted when u_acc(t) * q_t(d) < p_t(d), i.e. with
     probability min(1, p_t(d) / q_t(d)).
  3. a_i = number of leading accepted drafts.
  4. if a_i < L_i: the extra token is drawn from the residual
     norm(max(0, p_a - q_a)); if a_i == L_i (all accepted): the bonus token
     is drawn from p_{L_i}.
  5. emitted_i = d_1 .. d_{a_i}, then that extra token.

Readings where the method leaves a choice:
  * uniforms are inputs: uniforms[n] = (u_acc, u_res) for verify position n;
  * sampling is an inverse CDF in ascending token order: the smallest k with
    cumsum(w)[k] > u * sum(w); if rounding leaves none, the last k with w_k > 0;
  * a residual with no positive mass falls back to p_a.

spec_verify_sparse takes the draft distribution as a sparse table and the
draft tokens' probabilities as given numbers; its steps are the same.

Pins (tests/test_oracle_spec.py): scipy softmax; exact brute force of the
whole output law on tiny vocabularies against the closed form
prod_t min(p_t, q_t) * (residual or p); Monte Carlo chi-square of the
emitted tokens against p; acceptance rate sum_v min(p, q); expected length
(1 - alpha^(L+1)) / (1 - alpha), Eq. (u_single).  The boundary-band helpers
(_cdf_margin, margin_accept, decision_margins) are pinned on hand-worked
values in tests/test_oracle_margins.py.
"""
from __future__ import annotations

import numpy as np


def softmax(x: np.ndarray) -> np.ndarray:
    """Row softmax in fp64, max-subtracted."""
    x = np.asarray(x, dtype=np.float64)
    e = np.exp(x - x.max(axis=-1, keepdims=True))
    return e / e.sum(axis=-1, keepdims=True)


def inverse_cdf(w: np.ndarray, u: float) -> int:
    """Smallest index k with sum_{j<=k} w_j > u * sum_j w_j (w >= 0, unnormalised)."""
    c = np.cumsum(w)
    hit = np.flatnonzero(c > u * c[-1])
    if hit.size:
        return int(hit[0])
    return int(np.flatnonzero(w > 0)[-1])


def residual(p_row: np.ndarray, q_row: np.ndarray) -> np.ndarray:
    """Unnormalised residual max(0, p - q); p itself if that has no positive mass."""
    r = np.maximum(p_row - q_row, 0.0)
    return r if r.sum() > 0 else p_row


def _cdf_margin(w: np.ndarray, u: float, k: int) -> float:
    """Distance of u from the CDF boundaries of the chosen token k (in units of the total)."""
    c = np.cumsum(w)
    total = c[-1]
    lo = c[k - 1] if k > 0 else 0.0
    return float(min(u * total - lo, c[k] - u * total) / total)


def spec_verify(L, target_logits, draft_logits, draft_tokens, uniforms):
    """Speculative verification of one batch.

    L             [B] draft lengths L_i >= 0
    target_logits [sum_i (L_i+1), V] target logits z, users concatenated
    draft_logits  [sum_i L_i, V]     draft logits w
    draft_tokens  [sum_i L_i]        d_{i,1..L_i}
    uniforms      [sum_i (L_i+1), 2] (u_acc, u_res) per verify position

    Returns a dict:
      accept_len [B], out_offsets [B+1], out_tokens [sum_i (a_i+1)]   (the outputs)
      accepted [sum T] bool   acceptance test at every draft position (False at bonus)
      p_d, q_d [sum T]         p_t(d_{t+1}), q_t(d_{t+1}) (0 at the bonus position)
      margin_accept [sum T]    |u_acc - p_t(d)/q_t(d)| (inf at the bonus position)
      margin_resample [B]      distance of u_res from the chosen token's CDF cell edges
      resample_mass [B]        total mass of the distribution sampled at a_i
    """
    dt = np.asarray(draft_tokens, dtype=np.int64)
    p = softmax(target_logits)
    q = softmax(draft_logits) if len(dt) else np.zeros((0, p.shape[1]))
    q_d = q[np.arange(len(dt)), dt] if len(dt) else np.zeros(0)
    return _verify(L, p, q, q_d, dt, uniforms)


def spec_verify_sparse(L, target_logits, draft_tokens, draft_logq, topk_idx, topk_q, uniforms):
    """Speculative verification from a sparse draft payload (Sec. II-A: the
    device sends the drafted tokens and a small amount of probability
    information, e.g. draft-token log-probabilities).

    The draft distribution of draft position r is the table (topk_idx[r],
    topk_q[r]): q_r(topk_idx[r, j]) = topk_q[r, j] and 0 elsewhere (exact for
    a device that samples from its top K).  The acceptance test reads
    q_r(d) = exp(draft_logq[r]); the residual is max(0, p - q_r) over the whole
    vocabulary.  Everything else is spec_verify.

    draft_logq [sum_i L_i]; topk_idx, topk_q [sum_i L_i, K] (distinct indices)
    """
    dt = np.asarray(draft_tokens, dtype=np.int64)
    p = softmax(target_logits)
    idx = np.asarray(topk_idx, dtype=np.int64)
    q = np.zeros((len(dt), p.shape[1]))
    for r in range(len(dt)):
        q[r, idx[r]] = np.asarray(topk_q[r], dtype=np.float64)
    q_d = np.exp(np.asarray(draft_logq, dtype=np.float64))
    return _verify(L, p, q, q_d, dt, uniforms)


def _verify(L, p, q, q_d_all, dt, uniforms):
    """Steps 2-5 for target distributions p [sum T, V], draft distributions
    q [sum L, V] and the draft tokens' draft probabilities q_d_all [sum L]."""
    L = np.asarray(L, dtype=np.int64)
    B = L.shape[0]
    uni = np.asarray(uniforms, dtype=np.float64)
    sT = p.shape[0]

    accepted = np.zeros(sT, dtype=bool)
    p_d = np.zeros(sT)
    q_d = np.zeros(sT)
    margin_accept = np.full(sT, np.inf)
    accept_len = np.zeros(B, dtype=np.int64)
    margin_resample = np.zeros(B)
    resample_mass = np.zeros(B)
    emitted = []

    qo = lo = 0
    for i in range(B):
        Li = int(L[i])
        # step 2: acceptance test at every draft position
        for t in range(Li):
            d = dt[lo + t]
            pd, qd = p[qo + t, d], q_d_all[lo + t]
            p_d[qo + t], q_d[qo + t] = pd, qd
            accepted[qo + t] = uni[qo + t, 0] * qd < pd
            margin_accept[qo + t] = abs(uni[qo + t, 0] - pd / qd) if qd > 0 else np.inf
        # step 3: leading accepted drafts
        a = 0
        while a < Li and accepted[qo + a]:
            a += 1
        accept_len[i] = a
        # step 4: residual at the first rejection, else p at the bonus position
        w = residual(p[qo + a], q[lo + a]) if a < Li else p[qo + Li]
        u = uni[qo + a, 1]
        y = inverse_cdf(w, u)
        margin_resample[i] = _cdf_margin(w, u, y)
        resample_mass[i] = w.sum()
        # step 5: emitted tokens
        emitted.append(np.concatenate([dt[lo:lo + a], [y]]))
        qo += Li + 1
        lo += Li

    out_offsets = np.zeros(B + 1, dtype=np.int64)
    out_offsets[1:] = np.cumsum(accept_len + 1)
    out_tokens = np.concatenate(emitted) if emitted else np.zeros(0, dtype=np.int64)
    return dict(accept_len=accept_len, out_offsets=out_offsets, out_tokens=out_tokens,
                accepted=accepted, p_d=p_d, q_d=q_d, margin_accept=margin_accept,
                margin_resample=margin_resample, resample_mass=resample_mass)


def decision_margins(result, L, band=1e-6):
    """Per user: True when a decision that shaped its output lay within `band`.

    Decisions that shaped user i's output: the acceptance tests at positions
    0 .. min(a_i, L_i - 1) and the resample at a_i.
    """
    L = np.asarray(L, dtype=np.int64)
    near = np.zeros(len(L), dtype=bool)
    qo = 0
    for i, Li in enumerate(L):
        a = int(result["accept_len"][i])
        last = min(a, int(Li) - 1)
        if last >= 0 and np.min(result["margin_accept"][qo:qo + last + 1]) < band:
            near[i] = True
        if result["margin_resample"][i] < band:
            near[i] = True
        qo += int(Li) + 1
    return near
