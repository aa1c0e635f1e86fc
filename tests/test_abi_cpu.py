"""The C-ABI library builds, loads and exports every symbol include/dipsd.h
declares; host-side validation rejects bad arguments before touching the GPU."""
import ctypes
import os
import re

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2604_20919_gb300 import build, dipsd
    build.build()
    return dipsd.load()


def _declared():
    hdr = open(os.path.join(ROOT, "include", "dipsd.h")).read()
    hdr = re.sub(r"/\*.*?\*/", "", hdr, flags=re.S)
    return sorted(set(re.findall(r"\b(dipsd_\w+)\s*\(", hdr)))


def test_header_declarations_are_exported(lib):
    from paper_2604_20919_gb300 import dipsd
    names = _declared()
    assert names == sorted(dipsd.EXPORTS)
    for n in names:
        assert hasattr(lib, n), n


def test_status_strings_and_version(lib):
    assert lib.dipsd_abi_version() == 2
    from paper_2604_20919_gb300 import dipsd
    assert dipsd.status_string(0) == "ok"
    assert "invalid" in dipsd.status_string(1)
    assert "unknown" in dipsd.status_string(99)


def _i32(x):
    a = np.ascontiguousarray(np.asarray(x, dtype=np.int32))
    return a, a.ctypes.data_as(ctypes.POINTER(ctypes.c_int))


FAKE = 1 << 20  # 16-byte aligned, never dereferenced: validation fails first


@pytest.mark.parametrize("B,L,ctx,Hq,Hkv,D,want", [
    (0, [], [], 8, 2, 128, 1),               # empty batch
    (2, [1, -1], [4, 4], 8, 2, 128, 1),      # negative draft length
    (2, [1, 32], [4, 4], 8, 2, 128, 1),      # draft length above 31
    (2, [1, 2], [4, -3], 8, 2, 128, 1),      # negative context
    (2, [1, 2], [4, 4], 8, 3, 128, 1),       # Hq not a multiple of Hkv
    (2, [1, 2], [4, 4], 8, 2, 96, 2),        # head_dim not built
    (1, [0], [10 ** 6], 8, 2, 128, 1),       # context beyond the block table (max_blocks = 4)
])
def test_attention_rejects_bad_arguments(lib, B, L, ctx, Hq, Hkv, D, want):
    a, pa = _i32(L if L else [0])
    c, pc = _i32(ctx if ctx else [0])
    st = lib.dipsd_verify_attention(B, pa, pc, FAKE, FAKE, FAKE, 16, FAKE, 4, Hq, Hkv, D, 0.1, FAKE + 4096,
                                    FAKE, 1 << 20, None)
    assert st == want


def test_attention_rejects_null_and_misaligned_pointers(lib):
    a, pa = _i32([1])
    c, pc = _i32([3])
    assert lib.dipsd_verify_attention(1, pa, pc, None, FAKE, FAKE, 16, FAKE, 4, 8, 2, 128, 0.1, FAKE, FAKE,
                                      1 << 20, None) == 1
    assert lib.dipsd_verify_attention(1, pa, pc, FAKE + 2, FAKE, FAKE, 16, FAKE, 4, 8, 2, 128, 0.1, FAKE,
                                      FAKE, 1 << 20, None) == 1
    assert lib.dipsd_verify_attention(1, pa, pc, FAKE, FAKE, FAKE, 0, FAKE, 4, 8, 2, 128, 0.1, FAKE + 64,
                                      FAKE, 1 << 20, None) == 1


def test_spec_verify_rejects_bad_arguments(lib):
    u, pu = _i32([0, 1])
    a, pa = _i32([2, 40])
    assert lib.dipsd_spec_verify(2, pa, pu, 7, 100, 0, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, None, FAKE, 1 << 20,
                                 None) == 1
    a, pa = _i32([2, 3])
    assert lib.dipsd_spec_verify(2, pa, pu, 7, 0, 0, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, None, FAKE, 1 << 20,
                                 None) == 1
    assert lib.dipsd_spec_verify(2, pa, pu, 7, 100, 7, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, None, FAKE, 1 << 20,
                                 None) == 1
    assert lib.dipsd_spec_verify(2, pa, pu, 7, 100, 0, FAKE, None, FAKE, FAKE, FAKE, FAKE, None, FAKE, 1 << 20,
                                 None) == 1
    # user ids: required, non-negative
    assert lib.dipsd_spec_verify(2, pa, None, 7, 100, 0, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, None, FAKE, 1 << 20,
                                 None) == 1
    bad, pbad = _i32([0, -4])
    assert lib.dipsd_spec_verify(2, pa, pbad, 7, 100, 0, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, None, FAKE, 1 << 20,
                                 None) == 1
    # workspace too small / missing
    assert lib.dipsd_spec_verify(2, pa, pu, 7, 100, 0, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, None, FAKE, 8,
                                 None) == 4
    assert lib.dipsd_spec_verify(2, pa, pu, 7, 100, 0, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, None, None, 1 << 20,
                                 None) == 4


def test_noalloc_rejects_batches_beyond_its_positions_before_any_launch(lib):
    a, pa = _i32([31] * 128 + [0])  # 4097 verify positions > DIPSD_NOALLOC_MAX_POSITIONS
    u, pu = _i32(range(129))
    n0 = lib.dipsd_launch_count()
    assert lib.dipsd_spec_verify_noalloc(129, pa, pu, 3, 1024, 0, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, None,
                                         None) == 2
    assert lib.dipsd_launch_count() == n0


def test_philox_entry_points_reject_bad_arguments(lib):
    assert lib.dipsd_philox_words(1, -1, 4, FAKE, None) == 1
    assert lib.dipsd_philox_words(1, 0, -4, FAKE, None) == 1
    assert lib.dipsd_philox_words(1, 0, 4, FAKE + 8, None) == 1  # not 16-byte aligned
    assert lib.dipsd_philox_words(1, 0, 0, None, None) == 0      # nothing to write
    a, pa = _i32([2, 3])
    u, pu = _i32([0, -1])
    assert lib.dipsd_verify_uniforms(2, pa, pu, 5, FAKE, None) == 1
    u, pu = _i32([0, 1])
    assert lib.dipsd_verify_uniforms(2, pa, pu, 5, None, None) == 1


def test_test_overrides_are_explicit(lib):
    """The planner never reads the environment: only dipsd_test_set_override moves it."""
    import os
    from paper_2604_20919_gb300 import dipsd
    L, ctx = [5, 0, 8, 2, 20, 1], [1500, 3000, 333, 64, 700, 0]
    base = dipsd.dipsd_verify_attention_plan(L, ctx, 64, 8, 128, 152)
    os.environ["DIPSD_ATTN_CLUSTER"] = "3"
    try:
        assert dipsd.dipsd_verify_attention_plan(L, ctx, 64, 8, 128, 152)["cluster"] == base["cluster"]
    finally:
        del os.environ["DIPSD_ATTN_CLUSTER"]
    with dipsd.plan_override(attn_cluster=3):
        assert dipsd.dipsd_verify_attention_plan(L, ctx, 64, 8, 128, 152)["cluster"] == 3
    assert dipsd.dipsd_verify_attention_plan(L, ctx, 64, 8, 128, 152)["cluster"] == base["cluster"]
    assert lib.dipsd_test_set_override(0, 1) == 1
    assert lib.dipsd_test_set_override(9, 1) == 1
    assert lib.dipsd_test_set_override(1, -1) == 1


def test_spec_workspace_size_is_host_only(lib):
    a, pa = _i32([3, 0, 5])
    n = lib.dipsd_spec_verify_workspace_size(3, pa, 151936)
    assert n >= 256 + 11 * 16 + 11
    assert lib.dipsd_spec_verify_workspace_size(0, pa, 151936) == 0


def test_verify_batch_rejects_bad_membership(lib):
    m, pm = _i32([0, 2, 2])
    a, pa = _i32([1, 2, 3])
    c, pc = _i32([4, 4, 4])
    args = (FAKE, FAKE, FAKE, 16, FAKE, 4, 8, 2, 128, 0.1, FAKE + 4096, 100, 0, FAKE, FAKE, FAKE, 7,
            FAKE, FAKE, FAKE, None, FAKE, 1 << 20, None)
    assert lib.dipsd_verify_batch(3, pm, 3, pa, pc, *args) == 1   # duplicate member
    m, pm = _i32([0, 3])
    assert lib.dipsd_verify_batch(2, pm, 3, pa, pc, *args) == 1   # member out of range
