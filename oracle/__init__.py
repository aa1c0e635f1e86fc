"""CPU fp64 oracle for DiP-SD batched verification -- TEST INFRASTRUCTURE ONLY.

Plain, slow, obviously correct NumPy restatements of what the edge server
computes in one batch-verification round (paper Sec. II-A, stage 2):

  * attention.verify_attention -- causal GQA attention of each user's L_i+1
    verify tokens over that user's paged KV cache (plain definition).
  * attention.kv_append        -- the round's state update: each verify
    token's key/value row written to its page and slot (plain scatter).
  * spec_verify.spec_verify    -- speculative sampling: accept/reject each
    draft token, truncate at the first rejection, resample from the residual
    or from p at the bonus position, pack the emitted tokens.
  * spec_verify.spec_verify_sparse -- the same from a sparse draft payload
    (draft-token log-probabilities and a top-K draft distribution).

Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline / reference
leg may import this package.  It shares no code with the CUDA library and
never imports it.  Every function is pinned by tests/test_oracle_*.py against
closed forms, invariants, library routines or brute force (see each
function's docstring for its pin).
"""
from .attention import kv_append, verify_attention
from .spec_verify import softmax, inverse_cdf, spec_verify, spec_verify_sparse, decision_margins

__all__ = ["kv_append", "verify_attention", "softmax", "inverse_cdf", "spec_verify", "spec_verify_sparse", "decision_margins"]
