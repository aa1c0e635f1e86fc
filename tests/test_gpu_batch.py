"""dipsd_verify_batch (one pipeline stage's users) vs the oracle, incl. the
pipelined schedule of four stages on two streams."""
import numpy as np
import pytest
import torch

import oracle
from parity import attention_subset_reference, check_attention, check_spec, valid_spec_outputs
from workloads import make_batch, make_config

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _launch(dipsd, b, L_all, ctx_all, kc, vc, bt, stream):
    g = lambda t: t.to(DEV, non_blocking=True)
    with torch.cuda.stream(stream):
        res = dipsd.dipsd_verify_batch(b.members, L_all, ctx_all, g(b.q), kc, vc, bt, b.scale,
                                       g(b.target_logits), g(b.draft_logits), g(b.draft_tokens),
                                       b.seed, stream=stream)
    return res


def test_pipelined_stages_on_two_streams(cuda_lib):
    """Workload 5: 128 users dealt into 4 batches of 32, verified back to back on two streams."""
    batches = make_config(5, seed=0, device="cpu", kv_device=DEV)
    from workloads import config_shape
    s = config_shape(5)
    L_all, ctx_all = s["L"], s["ctx"]
    kc, vc = batches[0].k_cache, batches[0].v_cache
    bt = batches[0].block_table.to(DEV)
    streams = [torch.cuda.Stream(), torch.cuda.Stream()]
    results = [_launch(cuda_lib, b, L_all, ctx_all, kc, vc, bt, streams[n % 2]) for n, b in enumerate(batches)]
    torch.cuda.synchronize()
    for n, (b, (attn, acc, offs, toks, probs)) in enumerate(zip(batches, results)):
        st = check_spec(b, acc, offs, toks, probs)
        users = [0, int(np.argmax(b.ctx)), b.B - 1]
        rows, ref, ref_abs = attention_subset_reference(b, users, with_abs=True)
        err = check_attention(attn[torch.from_numpy(rows).to(DEV)], ref, ref_abs)
        print(f"stage {n}: {st}, attention max err {err:.3e}")


@pytest.mark.parametrize("fork", [1, 2])
def test_batch_matches_separate_calls(cuda_lib, fork):
    """verify_batch equals the two separate calls, with the decision and
    sampling kernels on the library's second stream (1) or on the caller's (2)."""
    b = make_config(2, seed=4)
    g = lambda t: t.to(DEV)
    q, kc, vc, bt = g(b.q), g(b.k_cache), g(b.v_cache), g(b.block_table)
    z, w, d = g(b.target_logits), g(b.draft_logits), g(b.draft_tokens)
    attn_a = cuda_lib.dipsd_verify_attention(b.L, b.ctx, q, kc, vc, bt, b.scale)
    sv = cuda_lib.dipsd_spec_verify(b.L, b.members, b.seed, z, w, d)
    with cuda_lib.plan_override(batch_fork=fork):
        res = cuda_lib.dipsd_verify_batch(b.members, b.L, b.ctx, q, kc, vc, bt, b.scale, z, w, d, b.seed)
    torch.cuda.synchronize()
    assert torch.equal(attn_a, res[0])
    for x, y in zip(valid_spec_outputs(*sv), valid_spec_outputs(*res[1:])):
        assert torch.equal(x, y)


def test_batch_with_permuted_membership(cuda_lib):
    """Members name rows of a larger user table, in any order."""
    # table of 6 users: batch users sit at rows 4, 0, 5, 2 (their Philox key words)
    perm = np.array([4, 0, 5, 2])
    from workloads import config_shape
    s = config_shape(1)
    b = make_batch(s["L"], s["ctx"], Hq=s["Hq"], Hkv=s["Hkv"], D=s["D"], V=s["V"], logit_std=s["logit_std"],
                   noise_sigma=s["noise_sigma"], logit_dtype=s["logit_dtype"], seed=5, user_ids=perm)
    L_all = np.zeros(6, np.int32)
    ctx_all = np.zeros(6, np.int32)
    L_all[perm], ctx_all[perm] = b.L, b.ctx
    bt_all = torch.full((6, b.block_table.shape[1]), -1, dtype=torch.int32)
    bt_all[torch.from_numpy(perm)] = b.block_table
    g = lambda t: t.to(DEV)
    attn, acc, offs, toks, probs = cuda_lib.dipsd_verify_batch(
        perm, L_all, ctx_all, g(b.q), g(b.k_cache), g(b.v_cache), g(bt_all), b.scale, g(b.target_logits),
        g(b.draft_logits), g(b.draft_tokens), b.seed)
    torch.cuda.synchronize()
    ref = oracle.verify_attention(b.q.double().numpy(), b.k_cache.double().numpy(), b.v_cache.double().numpy(),
                                  b.block_table.numpy(), b.ctx, b.L, b.scale)
    ref_abs = oracle.verify_attention(b.q.double().numpy(), b.k_cache.double().numpy(),
                                      np.abs(b.v_cache.double().numpy()), b.block_table.numpy(), b.ctx, b.L, b.scale)
    check_attention(attn, ref, ref_abs)
    check_spec(b, acc, offs, toks, probs)


def test_batch_captured_in_a_graph(cuda_lib):
    """verify_batch captured into a CUDA graph (both streams) and replayed:
    the replays give the outputs of a plain call."""
    b = make_config(2, seed=9)
    g = lambda t: t.to(DEV)
    q, kc, vc, bt = g(b.q), g(b.k_cache), g(b.v_cache), g(b.block_table)
    z, w, d = g(b.target_logits), g(b.draft_logits), g(b.draft_tokens)
    ws = cuda_lib.workspace(cuda_lib.dipsd_verify_batch_workspace_size(b.members, b.L, b.ctx, b.Hq, b.Hkv, b.D, b.V),
                            DEV)
    attn = torch.empty_like(q)
    outs = cuda_lib.spec_outputs(b.L, DEV)
    call = lambda: cuda_lib.dipsd_verify_batch(b.members, b.L, b.ctx, q, kc, vc, bt, b.scale, z, w, d, b.seed,
                                               attn_out=attn, outputs=outs, ws=ws)
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        call()  # the first call from this stream, outside the capture
    torch.cuda.synchronize()
    ref = [attn.clone()] + [t.clone() for t in valid_spec_outputs(*outs)]
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=s):  # a stream that made a plain call first
        call()
    for _ in range(3):
        attn.zero_()
        for t in outs[:3]:
            t.fill_(-1)
        graph.replay()
        torch.cuda.synchronize()
        got = [attn] + valid_spec_outputs(*outs)
        for x, y in zip(ref, got):
            assert torch.equal(x, y)
    assert cuda_lib.device_status(ws) == 0


def test_batch_from_many_streams(cuda_lib):
    """Calls from more caller streams than the library keeps second streams
    for (each new stream takes over the oldest set): every call still gives
    the outputs of the first, and the status word stays clear."""
    b = make_config(2, seed=11)
    g = lambda t: t.to(DEV)
    q, kc, vc, bt = g(b.q), g(b.k_cache), g(b.v_cache), g(b.block_table)
    z, w, d = g(b.target_logits), g(b.draft_logits), g(b.draft_tokens)
    ref = cuda_lib.dipsd_verify_batch(b.members, b.L, b.ctx, q, kc, vc, bt, b.scale, z, w, d, b.seed)
    torch.cuda.synchronize()
    ref = [ref[0]] + valid_spec_outputs(*ref[1:])
    streams = [torch.cuda.Stream() for _ in range(10)]
    results = []
    for _ in range(2):
        for s in streams:
            with torch.cuda.stream(s):
                results.append(cuda_lib.dipsd_verify_batch(b.members, b.L, b.ctx, q, kc, vc, bt, b.scale, z, w,
                                                           d, b.seed, stream=s))
    torch.cuda.synchronize()
    for res in results:
        got = [res[0]] + valid_spec_outputs(*res[1:])
        for x, y in zip(ref, got):
            assert torch.equal(x, y)
