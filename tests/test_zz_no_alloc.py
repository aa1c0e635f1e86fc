"""dipsd_spec_verify_noalloc: the entry point for callers that cannot allocate
device memory (it keeps its scratch in a static device array instead of a
caller workspace).  Called through the C ABI on two calls in a row, and
compared with the fp64 oracle (the same parity bar as every spec test) and
with dipsd_spec_verify on the same inputs.

This file is collected last on purpose, so that a run stopping at the first
failure has already run every other test.
"""
import ctypes

import numpy as np
import pytest
import torch

from parity import PROB_ATOL, check_spec, valid_spec_outputs
from workloads import make_batch, make_config

pytestmark = pytest.mark.gpu
DEV = "cuda"
_I32P = ctypes.POINTER(ctypes.c_int)


def _noalloc(lib, b, z, w, d, stream):
    L = np.ascontiguousarray(b.L, dtype=np.int32)
    uid = np.ascontiguousarray(b.user_ids, dtype=np.int32)
    sum_t = int(b.T.sum())
    acc = torch.full((b.B,), -7, dtype=torch.int32, device=DEV)
    offs = torch.full((b.B + 1,), -7, dtype=torch.int32, device=DEV)
    toks = torch.full((sum_t,), -7, dtype=torch.int32, device=DEV)
    probs = torch.full((sum_t, 2), -7.0, dtype=torch.float32, device=DEV)
    dtype = 0 if z.dtype == torch.bfloat16 else 1
    st = lib.dipsd_spec_verify_noalloc(
        b.B, L.ctypes.data_as(_I32P), uid.ctypes.data_as(_I32P), b.seed, b.V, dtype, z.data_ptr(),
        w.data_ptr() if w.numel() else None, d.data_ptr() if d.numel() else None,
        acc.data_ptr(), offs.data_ptr(), toks.data_ptr(), probs.data_ptr(), stream.cuda_stream)
    return st, (acc, offs, toks, probs)


def test_noalloc_matches_oracle_and_workspace_entry_point_on_two_calls(cuda_lib):
    lib = cuda_lib.load()
    stream = torch.cuda.current_stream()
    batches = [make_config(2, seed=0, spec_only=True),
               make_batch([3, 0, 9, 1, 5], [0] * 5, Hq=8, Hkv=1, D=64, V=32000, logit_std=1.0,
                          noise_sigma=0.8, seed=31, spec_only=True)]
    for b in batches:  # two calls in a row through the shared scratch
        g = lambda t: t.to(DEV)
        z, w, d = g(b.target_logits), g(b.draft_logits), g(b.draft_tokens)
        st, got = _noalloc(lib, b, z, w, d, stream)
        assert st == 0, cuda_lib.status_string(st)
        torch.cuda.synchronize()
        print(check_spec(b, *got))
        ref = cuda_lib.dipsd_spec_verify(b.L, b.user_ids, b.seed, z, w, d)
        torch.cuda.synchronize()
        g_acc, g_offs, g_toks, g_probs = valid_spec_outputs(*got)
        r_acc, r_offs, r_toks, r_probs = valid_spec_outputs(*ref)
        assert torch.equal(g_acc, r_acc)
        assert torch.equal(g_offs, r_offs)
        assert torch.equal(g_toks, r_toks)
        assert torch.allclose(g_probs, r_probs, atol=PROB_ATOL, rtol=0)


def test_noalloc_rejects_batches_beyond_its_scratch(cuda_lib):
    lib = cuda_lib.load()
    dummy = torch.zeros(16, dtype=torch.int32, device=DEV)
    p = dummy.data_ptr()
    n0 = cuda_lib.dipsd_launch_count()
    # 6300 verify positions > 4096
    L = np.full(300, 20, dtype=np.int32)
    uid = np.arange(300, dtype=np.int32)
    st = lib.dipsd_spec_verify_noalloc(300, L.ctypes.data_as(_I32P), uid.ctypes.data_as(_I32P), 0, 64, 0,
                                       p, p, p, p, p, p, None, None)
    assert st == 2  # DIPSD_ERR_UNSUPPORTED, nothing launched
    # 4096 positions, but fp32 logits at V = 151936: the plan's scratch exceeds 8 MiB
    L = np.full(128, 31, dtype=np.int32)
    uid = np.arange(128, dtype=np.int32)
    st = lib.dipsd_spec_verify_noalloc(128, L.ctypes.data_as(_I32P), uid.ctypes.data_as(_I32P), 0, 151936, 1,
                                       p, p, p, p, p, p, None, None)
    assert st == 2
    assert cuda_lib.dipsd_launch_count() == n0
