"""Python binding of libdipsd.so (the C ABI in include/dipsd.h).

Argument marshalling only: every step of verification runs in the library's
CUDA kernels.  Functions carry the C names; tensors are torch CUDA tensors
(device memory and streams come from PyTorch), per-user lengths are host
sequences.  If the library is missing this module raises instead of falling
back to anything else.
"""
from __future__ import annotations

import contextlib
import ctypes
import os
from typing import Optional, Sequence

import numpy as np
import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libdipsd.so")

DIPSD_OK = 0
DIPSD_BF16 = 0
DIPSD_F32 = 1
PAGE_SIZE = 16
MAX_USERS = 512
MAX_DRAFT = 31
DEVERR_WAIT_TIMEOUT = 1
DEVERR_BAD_TOKEN = 2
DEVERR_BAD_BLOCK = 4

EXPORTS = (
    "dipsd_status_string", "dipsd_abi_version", "dipsd_launch_count",
    "dipsd_verify_attention_workspace_size", "dipsd_verify_attention",
    "dipsd_spec_verify_workspace_size", "dipsd_spec_verify",
    "dipsd_verify_batch_workspace_size", "dipsd_verify_batch", "dipsd_spec_verify_noalloc",
    "dipsd_verify_attention_append", "dipsd_verify_batch_append",
    "dipsd_spec_verify_sparse_workspace_size", "dipsd_spec_verify_sparse", "dipsd_verify_attention_plan",
    "dipsd_philox_words", "dipsd_verify_uniforms", "dipsd_test_set_override",
)
NOALLOC_MAX_POSITIONS = 4096
# dipsd_test_set_override codes
TEST_OVERRIDES = {"attn_split_tiles": 1, "attn_cluster": 2, "attn_persist": 3, "attn_grid": 4,
                  "spec_nk1": 5, "spec_nk2": 6, "spec_grid1": 7, "batch_fork": 8}

_lib: Optional[ctypes.CDLL] = None
_i32p = ctypes.c_void_p  # host int32 arrays, passed by address
_vp = ctypes.c_void_p
_sz = ctypes.c_size_t
_i = ctypes.c_int
_u64 = ctypes.c_uint64


class AttentionPlan(ctypes.Structure):
    """dipsd_attention_plan of include/dipsd.h."""
    _fields_ = [("n_items", _i), ("grid", _i), ("cluster", _i), ("n_merge", _i), ("stream_chunks", _i),
                ("ws_bytes", _sz)]


class DipsdError(RuntimeError):
    def __init__(self, status: int, where: str):
        super().__init__(f"{where}: {status_string(status)} (status {status})")
        self.status = status


def load(path: str = LIB_PATH) -> ctypes.CDLL:
    """Loads the library once; raises if it has not been built."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is missing: build it with __graft_entry__.build()")
    lib = ctypes.CDLL(path)
    lib.dipsd_status_string.restype = ctypes.c_char_p
    lib.dipsd_status_string.argtypes = [_i]
    lib.dipsd_abi_version.restype = _i
    lib.dipsd_launch_count.restype = ctypes.c_longlong
    lib.dipsd_verify_attention_workspace_size.restype = _sz
    lib.dipsd_verify_attention_workspace_size.argtypes = [_i, _i32p, _i32p, _i, _i, _i]
    lib.dipsd_verify_attention.restype = _i
    lib.dipsd_verify_attention.argtypes = [_i, _i32p, _i32p, _vp, _vp, _vp, _i, _vp, _i, _i, _i, _i,
                                           ctypes.c_float, _vp, _vp, _sz, _vp]
    lib.dipsd_spec_verify_workspace_size.restype = _sz
    lib.dipsd_spec_verify_workspace_size.argtypes = [_i, _i32p, _i]
    lib.dipsd_spec_verify.restype = _i
    lib.dipsd_spec_verify.argtypes = [_i, _i32p, _i32p, _u64, _i, _i, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _sz,
                                      _vp]
    lib.dipsd_verify_batch_workspace_size.restype = _sz
    lib.dipsd_verify_batch_workspace_size.argtypes = [_i, _i32p, _i, _i32p, _i32p, _i, _i, _i, _i]
    lib.dipsd_verify_batch.restype = _i
    lib.dipsd_verify_batch.argtypes = [_i, _i32p, _i, _i32p, _i32p, _vp, _vp, _vp, _i, _vp, _i, _i, _i, _i,
                                       ctypes.c_float, _vp, _i, _i, _vp, _vp, _vp, _u64, _vp, _vp, _vp, _vp,
                                       _vp, _sz, _vp]
    lib.dipsd_verify_attention_append.restype = _i
    lib.dipsd_verify_attention_append.argtypes = [_i, _i32p, _i32p, _vp, _vp, _vp, _vp, _vp, _i, _vp, _i, _i, _i,
                                                  _i, ctypes.c_float, _vp, _vp, _sz, _vp]
    lib.dipsd_verify_batch_append.restype = _i
    lib.dipsd_verify_batch_append.argtypes = [_i, _i32p, _i, _i32p, _i32p, _vp, _vp, _vp, _vp, _vp, _i, _vp, _i,
                                              _i, _i, _i, ctypes.c_float, _vp, _i, _i, _vp, _vp, _vp, _u64, _vp,
                                              _vp, _vp, _vp, _vp, _sz, _vp]
    lib.dipsd_spec_verify_sparse_workspace_size.restype = _sz
    lib.dipsd_spec_verify_sparse_workspace_size.argtypes = [_i, _i32p, _i]
    lib.dipsd_spec_verify_sparse.restype = _i
    lib.dipsd_spec_verify_sparse.argtypes = [_i, _i32p, _i32p, _u64, _i, _i, _i, _vp, _vp, _vp, _vp, _vp, _vp, _vp,
                                             _vp, _vp, _vp, _sz, _vp]
    lib.dipsd_verify_attention_plan.restype = _i
    lib.dipsd_verify_attention_plan.argtypes = [_i, _i32p, _i32p, _i, _i, _i, _i, _i,
                                                ctypes.POINTER(AttentionPlan), _i32p, _i32p, _i32p]
    lib.dipsd_spec_verify_noalloc.restype = _i
    lib.dipsd_spec_verify_noalloc.argtypes = [_i, _i32p, _i32p, _u64, _i, _i, _vp, _vp, _vp, _vp, _vp, _vp, _vp,
                                              _vp]
    lib.dipsd_philox_words.restype = _i
    lib.dipsd_philox_words.argtypes = [_u64, _i, ctypes.c_longlong, _vp, _vp]
    lib.dipsd_verify_uniforms.restype = _i
    lib.dipsd_verify_uniforms.argtypes = [_i, _i32p, _i32p, _u64, _vp, _vp]
    lib.dipsd_test_set_override.restype = _i
    lib.dipsd_test_set_override.argtypes = [_i, _i]
    _lib = lib
    return lib


def dipsd_launch_count() -> int:
    """Kernels launched by the library from this host thread so far."""
    return int(load().dipsd_launch_count())


@contextlib.contextmanager
def plan_override(**overrides):
    """Test hook: plan overrides (names of TEST_OVERRIDES, 0 = the planner's
    own choice) held for the duration of the block, process-wide."""
    lib = load()
    for k, v in overrides.items():
        _check(lib.dipsd_test_set_override(TEST_OVERRIDES[k], int(v)), "dipsd_test_set_override")
    try:
        yield
    finally:
        for k in overrides:
            lib.dipsd_test_set_override(TEST_OVERRIDES[k], 0)


def status_string(status: int) -> str:
    return load().dipsd_status_string(int(status)).decode()


def _check(status: int, where: str) -> None:
    if status != DIPSD_OK:
        raise DipsdError(status, where)


def _host_i32(x: Sequence[int]):
    """A C-contiguous int32 host array of x (x itself when it already is one)
    and its address; the array must outlive the call that gets the address."""
    if type(x) is np.ndarray and x.dtype == np.int32 and x.flags.c_contiguous:
        a = x
    else:
        a = np.ascontiguousarray(x, dtype=np.int32)
    return a, a.ctypes.data


def _dptr(t: Optional[torch.Tensor], name: str, dtype=None) -> int:
    """Device address of a contiguous CUDA tensor (of dtype, if given)."""
    if t is None:
        return 0
    if not (t.is_cuda and t.is_contiguous()):
        raise ValueError(f"{name} must be a contiguous CUDA tensor")
    if dtype is not None and t.dtype is not dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
    return t.data_ptr()


def _stream(stream) -> int:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)


def _logit_dtype(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return DIPSD_BF16
    if t.dtype == torch.float32:
        return DIPSD_F32
    raise ValueError(f"logits must be bf16 or fp32, got {t.dtype}")


def workspace(nbytes: int, device) -> torch.Tensor:
    """Zero-filled device buffer usable as a workspace (status word starts at 0)."""
    return torch.zeros(max(int(nbytes), 256), dtype=torch.uint8, device=device)


def device_status(ws: torch.Tensor) -> int:
    """Device status word (DEVERR_* bits) of a workspace; synchronises on its stream."""
    return int(ws[:4].view(torch.int32).item())


# ---------------------------------------------------------------- attention
def dipsd_verify_attention_workspace_size(L, ctx, Hq: int, Hkv: int, D: int) -> int:
    a, pa = _host_i32(L)
    b, pb = _host_i32(ctx)
    return int(load().dipsd_verify_attention_workspace_size(len(a), pa, pb, Hq, Hkv, D))


def dipsd_verify_attention_plan(L, ctx, Hq: int, Hkv: int, D: int, num_sms: int, append: bool = False) -> dict:
    """The work plan the attention entry points make for a device with
    num_sms SMs (host only).  Returns n_items, grid, cluster, n_merge,
    stream_chunks, ws_bytes, per user nsplit and split_len, and (page-stream
    plans) chunk_bound."""
    a, pa = _host_i32(L)
    b, pb = _host_i32(ctx)
    plan = AttentionPlan()
    nsplit, pn = _host_i32(np.zeros(len(a)))
    split_len, ps = _host_i32(np.zeros(len(a)))
    bounds, pbd = _host_i32(np.zeros(int(num_sms) + 1))
    _check(load().dipsd_verify_attention_plan(len(a), pa, pb, Hq, Hkv, D, int(num_sms), 1 if append else 0,
                                              ctypes.byref(plan), pn, ps, pbd), "dipsd_verify_attention_plan")
    return {"n_items": plan.n_items, "grid": plan.grid, "cluster": plan.cluster, "n_merge": plan.n_merge,
            "stream_chunks": plan.stream_chunks, "ws_bytes": int(plan.ws_bytes), "nsplit": nsplit,
            "split_len": split_len, "chunk_bound": bounds[:plan.stream_chunks + 1] if plan.stream_chunks else None}


def dipsd_verify_attention(L, ctx, q, k_cache, v_cache, block_table, softmax_scale: float, out=None,
                           ws=None, stream=None) -> torch.Tensor:
    """Causal GQA attention of every verify token over its user's paged KV cache."""
    lib = load()
    a, pa = _host_i32(L)
    b, pb = _host_i32(ctx)
    sum_t = int((a + 1).sum())
    nb, Hkv, page, D = k_cache.shape
    Hq = q.shape[1]
    if page != PAGE_SIZE or tuple(q.shape) != (sum_t, Hq, D) or tuple(v_cache.shape) != tuple(k_cache.shape):
        raise ValueError("shape mismatch between q, caches and lengths")
    if block_table.dim() != 2 or block_table.shape[0] != len(a):
        raise ValueError("block_table must be [B][max_blocks]")
    if out is None:
        out = torch.empty_like(q)
    if ws is None:
        ws = workspace(dipsd_verify_attention_workspace_size(a, b, Hq, Hkv, D), q.device)
    st = lib.dipsd_verify_attention(len(a), pa, pb, _dptr(q, "q", torch.bfloat16),
                                    _dptr(k_cache, "k_cache", torch.bfloat16),
                                    _dptr(v_cache, "v_cache", torch.bfloat16), nb,
                                    _dptr(block_table, "block_table", torch.int32), block_table.shape[1],
                                    Hq, Hkv, D, float(softmax_scale), _dptr(out, "out", torch.bfloat16),
                                    _dptr(ws, "workspace"), ws.numel(), _stream(stream))
    _check(st, "dipsd_verify_attention")
    return out


def dipsd_verify_attention_append(L, ctx, q, new_k, new_v, k_cache, v_cache, block_table, softmax_scale: float,
                                  out=None, ws=None, stream=None) -> torch.Tensor:
    """As dipsd_verify_attention, first writing the verify tokens' K/V rows
    (new_k, new_v [sum T][Hkv][D]) into their pages (positions C_i + t)."""
    lib = load()
    a, pa = _host_i32(L)
    b, pb = _host_i32(ctx)
    sum_t = int((a + 1).sum())
    nb, Hkv, page, D = k_cache.shape
    Hq = q.shape[1]
    if page != PAGE_SIZE or tuple(q.shape) != (sum_t, Hq, D) or tuple(v_cache.shape) != tuple(k_cache.shape):
        raise ValueError("shape mismatch between q, caches and lengths")
    if tuple(new_k.shape) != (sum_t, Hkv, D) or tuple(new_v.shape) != (sum_t, Hkv, D):
        raise ValueError("new_k / new_v must be [sum T][Hkv][D]")
    if block_table.dim() != 2 or block_table.shape[0] != len(a):
        raise ValueError("block_table must be [B][max_blocks]")
    if out is None:
        out = torch.empty_like(q)
    if ws is None:
        ws = workspace(dipsd_verify_attention_workspace_size(a, b, Hq, Hkv, D), q.device)
    st = lib.dipsd_verify_attention_append(len(a), pa, pb, _dptr(q, "q", torch.bfloat16),
                                           _dptr(new_k, "new_k", torch.bfloat16), _dptr(new_v, "new_v", torch.bfloat16),
                                           _dptr(k_cache, "k_cache", torch.bfloat16),
                                           _dptr(v_cache, "v_cache", torch.bfloat16), nb,
                                           _dptr(block_table, "block_table", torch.int32), block_table.shape[1],
                                           Hq, Hkv, D, float(softmax_scale), _dptr(out, "out", torch.bfloat16),
                                           _dptr(ws, "workspace"), ws.numel(), _stream(stream))
    _check(st, "dipsd_verify_attention_append")
    return out


# ---------------------------------------------------------- spec verification
def dipsd_spec_verify_workspace_size(L, V: int) -> int:
    a, pa = _host_i32(L)
    return int(load().dipsd_spec_verify_workspace_size(len(a), pa, V))


def spec_outputs(L, device, with_probs=True):
    """Output tensors of one spec-verify call: accept_len, out_offsets, out_tokens, draft_probs."""
    B = len(L)
    sum_t = int(np.asarray(L).sum()) + B
    return (torch.empty(B, dtype=torch.int32, device=device),
            torch.empty(B + 1, dtype=torch.int32, device=device),
            torch.empty(sum_t, dtype=torch.int32, device=device),
            torch.empty(sum_t, 2, dtype=torch.float32, device=device) if with_probs else None)


def _user_ids(user_ids, B):
    u, pu = _host_i32(user_ids)
    if u.shape != (B,):
        raise ValueError("user_ids must hold one id per user")
    return u, pu


def dipsd_philox_words(seed: int, user_id: int, n_blocks: int, out=None, stream=None) -> torch.Tensor:
    """Words of counter blocks 0 .. n_blocks-1 of the Philox4x64-10 stream with
    key (seed, user_id), as int64 bit patterns [n_blocks * 4] on the current device."""
    if out is None:
        out = torch.empty(4 * int(n_blocks), dtype=torch.int64, device="cuda")
    _check(load().dipsd_philox_words(int(seed), int(user_id), int(n_blocks), _dptr(out, "out", torch.int64),
                                     _stream(stream)), "dipsd_philox_words")
    return out


def dipsd_verify_uniforms(L, user_ids, seed: int, out=None, stream=None) -> torch.Tensor:
    """The (u_acc, u_res) pairs spec verification draws for this batch, [sum T][2] fp32."""
    a, pa = _host_i32(L)
    u, pu = _user_ids(user_ids, len(a))
    if out is None:
        out = torch.empty(int((a + 1).sum()), 2, dtype=torch.float32, device="cuda")
    _check(load().dipsd_verify_uniforms(len(a), pa, pu, int(seed), _dptr(out, "out", torch.float32),
                                        _stream(stream)), "dipsd_verify_uniforms")
    return out


def dipsd_spec_verify(L, user_ids, seed, target_logits, draft_logits, draft_tokens, outputs=None, ws=None,
                      stream=None):
    """Speculative verification with in-kernel Philox uniforms keyed on
    (seed, user_ids[i]); returns (accept_len, out_offsets, out_tokens, draft_probs)."""
    lib = load()
    a, pa = _host_i32(L)
    u, pu = _user_ids(user_ids, len(a))
    sum_t, sum_l = int((a + 1).sum()), int(a.sum())
    V = target_logits.shape[1]
    dt = _logit_dtype(target_logits)
    if target_logits.shape[0] != sum_t:
        raise ValueError("target_logits do not match the draft lengths")
    if draft_logits.shape != (sum_l, V) or draft_logits.dtype != target_logits.dtype or draft_tokens.numel() != sum_l:
        raise ValueError("draft_logits / draft_tokens do not match the draft lengths")
    acc, offs, toks, probs = outputs if outputs is not None else spec_outputs(a, target_logits.device)
    if ws is None:
        ws = workspace(dipsd_spec_verify_workspace_size(a, V), target_logits.device)
    st = lib.dipsd_spec_verify(len(a), pa, pu, int(seed), V, dt, _dptr(target_logits, "target_logits"),
                               _dptr(draft_logits, "draft_logits") if sum_l else 0,
                               _dptr(draft_tokens, "draft_tokens", torch.int32) if sum_l else 0,
                               _dptr(acc, "accept_len", torch.int32), _dptr(offs, "out_offsets", torch.int32),
                               _dptr(toks, "out_tokens", torch.int32),
                               _dptr(probs, "draft_probs", torch.float32), _dptr(ws, "workspace"), ws.numel(),
                               _stream(stream))
    _check(st, "dipsd_spec_verify")
    return acc, offs, toks, probs


def dipsd_spec_verify_sparse_workspace_size(L, V: int) -> int:
    a, pa = _host_i32(L)
    return int(load().dipsd_spec_verify_sparse_workspace_size(len(a), pa, V))


def dipsd_spec_verify_sparse(L, user_ids, seed, target_logits, draft_tokens, draft_logq, topk_idx, topk_q,
                             outputs=None, ws=None, stream=None):
    """Speculative verification from a sparse draft payload; returns
    (accept_len, out_offsets, out_tokens, draft_probs)."""
    lib = load()
    a, pa = _host_i32(L)
    u, pu = _user_ids(user_ids, len(a))
    sum_t, sum_l = int((a + 1).sum()), int(a.sum())
    V = target_logits.shape[1]
    K = int(topk_idx.shape[1]) if topk_idx.dim() == 2 else 0
    if target_logits.shape[0] != sum_t:
        raise ValueError("target_logits do not match the draft lengths")
    if (draft_tokens.numel() != sum_l or draft_logq.numel() != sum_l or tuple(topk_idx.shape) != (sum_l, K)
            or tuple(topk_q.shape) != (sum_l, K)):
        raise ValueError("draft tokens / log-probabilities / table do not match the draft lengths")
    acc, offs, toks, probs = outputs if outputs is not None else spec_outputs(a, target_logits.device)
    if ws is None:
        ws = workspace(dipsd_spec_verify_sparse_workspace_size(a, V), target_logits.device)
    st = lib.dipsd_spec_verify_sparse(len(a), pa, pu, int(seed), V, max(K, 1), _logit_dtype(target_logits),
                                      _dptr(target_logits, "target_logits"),
                                      _dptr(draft_tokens, "draft_tokens", torch.int32) if sum_l else 0,
                                      _dptr(draft_logq, "draft_logq", torch.float32) if sum_l else 0,
                                      _dptr(topk_idx, "topk_idx", torch.int32) if sum_l else 0,
                                      _dptr(topk_q, "topk_q", torch.float32) if sum_l else 0,
                                      _dptr(acc, "accept_len", torch.int32), _dptr(offs, "out_offsets", torch.int32),
                                      _dptr(toks, "out_tokens", torch.int32),
                                      _dptr(probs, "draft_probs", torch.float32), _dptr(ws, "workspace"), ws.numel(),
                                      _stream(stream))
    _check(st, "dipsd_spec_verify_sparse")
    return acc, offs, toks, probs


# ---------------------------------------------------------------- one stage
def dipsd_verify_batch_workspace_size(members, L_all, ctx_all, Hq, Hkv, D, V) -> int:
    m, pm = _host_i32(members)
    a, pa = _host_i32(L_all)
    b, pb = _host_i32(ctx_all)
    return int(load().dipsd_verify_batch_workspace_size(len(m), pm, len(a), pa, pb, Hq, Hkv, D, V))


def _verify_batch(members, L_all, ctx_all, q, k_cache, v_cache, block_table_all, softmax_scale, target_logits,
                  draft_logits, draft_tokens, seed, attn_out, outputs, ws, stream, new_kv):
    """Attention then speculative verification for the users `members` of one stage.

    Returns (attn_out, accept_len, out_offsets, out_tokens, draft_probs).
    """
    lib = _lib if _lib is not None else load()
    m, pm = _host_i32(members)
    a, pa = _host_i32(L_all)
    b, pb = _host_i32(ctx_all)
    sum_l = int(a[m].sum())  # (a member outside the tables raises IndexError here)
    sum_t = sum_l + len(m)
    nb, Hkv, page, D = k_cache.shape
    Hq, V = q.shape[1], target_logits.shape[1]
    if page != PAGE_SIZE or q.shape != (sum_t, Hq, D):
        raise ValueError("q does not match the members' draft lengths")
    if target_logits.shape[0] != sum_t or draft_logits.shape != (sum_l, V):
        raise ValueError("logits do not match the members' draft lengths")
    if attn_out is None:
        attn_out = torch.empty_like(q)
    acc, offs, toks, probs = outputs if outputs is not None else spec_outputs(a[m], q.device)
    if ws is None:
        ws = workspace(dipsd_verify_batch_workspace_size(m, a, b, Hq, Hkv, D, V), q.device)
    if new_kv is not None:
        new_k, new_v = new_kv
        if tuple(new_k.shape) != (sum_t, Hkv, D) or tuple(new_v.shape) != (sum_t, Hkv, D):
            raise ValueError("new_k / new_v must be [sum T][Hkv][D]")
        fn, name = lib.dipsd_verify_batch_append, "dipsd_verify_batch_append"
        head = (_dptr(q, "q", torch.bfloat16), _dptr(new_k, "new_k", torch.bfloat16),
                _dptr(new_v, "new_v", torch.bfloat16))
    else:
        fn, name = lib.dipsd_verify_batch, "dipsd_verify_batch"
        head = (_dptr(q, "q", torch.bfloat16),)
    st = fn(len(m), pm, len(a), pa, pb, *head,
                                _dptr(k_cache, "k_cache", torch.bfloat16), _dptr(v_cache, "v_cache", torch.bfloat16),
                                nb, _dptr(block_table_all, "block_table", torch.int32), block_table_all.shape[1],
                                Hq, Hkv, D, float(softmax_scale), _dptr(attn_out, "attn_out", torch.bfloat16), V,
                                _logit_dtype(target_logits), _dptr(target_logits, "target_logits"),
                                _dptr(draft_logits, "draft_logits") if sum_l else 0,
                                _dptr(draft_tokens, "draft_tokens", torch.int32) if sum_l else 0, int(seed),
                                _dptr(acc, "accept_len", torch.int32), _dptr(offs, "out_offsets", torch.int32),
                                _dptr(toks, "out_tokens", torch.int32), _dptr(probs, "draft_probs", torch.float32),
                                _dptr(ws, "workspace"), ws.numel(), _stream(stream))
    _check(st, name)
    return attn_out, acc, offs, toks, probs


def dipsd_verify_batch(members, L_all, ctx_all, q, k_cache, v_cache, block_table_all, softmax_scale,
                       target_logits, draft_logits, draft_tokens, seed, attn_out=None, outputs=None,
                       ws=None, stream=None):
    """Attention then speculative verification for the users `members` of one
    stage (each member's Philox key is (seed, member index)).

    Returns (attn_out, accept_len, out_offsets, out_tokens, draft_probs).
    """
    return _verify_batch(members, L_all, ctx_all, q, k_cache, v_cache, block_table_all, softmax_scale,
                         target_logits, draft_logits, draft_tokens, seed, attn_out, outputs, ws, stream, None)


def dipsd_verify_batch_append(members, L_all, ctx_all, q, new_k, new_v, k_cache, v_cache, block_table_all,
                              softmax_scale, target_logits, draft_logits, draft_tokens, seed, attn_out=None,
                              outputs=None, ws=None, stream=None):
    """As dipsd_verify_batch, first writing the verify tokens' K/V rows into their pages."""
    return _verify_batch(members, L_all, ctx_all, q, k_cache, v_cache, block_table_all, softmax_scale,
                         target_logits, draft_logits, draft_tokens, seed, attn_out, outputs, ws, stream,
                         (new_k, new_v))
