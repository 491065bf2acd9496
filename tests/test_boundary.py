"""CPU checks of the C-ABI boundary: the library loads without a GPU, exports every entry
point include/domino.h declares, and rejects bad arguments before touching the device."""
import os
import re

import pytest

from paper_2605_29707_gb300 import binding

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _lib():
    if not os.path.exists(binding.LIB_PATH):
        from paper_2605_29707_gb300 import build
        build.build()
    return binding.load()


def declared_entry_points():
    with open(os.path.join(ROOT, "include", "domino.h")) as f:
        text = f.read()
    return re.findall(r"DOMINO_API\s+[\w\s\*]+?\b(domino_\w+)\s*\(", text)


def test_header_and_binding_agree():
    names = declared_entry_points()
    assert len(names) >= 8
    assert sorted(names) == sorted(binding.SYMBOLS)


def test_library_loads_and_exports_every_declared_symbol():
    lib = _lib()
    for name in declared_entry_points():
        assert hasattr(lib, name), name
    assert binding.domino_abi_version() == 2


def test_status_strings():
    _lib()
    assert binding.domino_status_string(0) == "DOMINO_OK"
    assert binding.domino_status_string(-5) == "DOMINO_ERR_BAD_TOKEN"
    assert binding.domino_status_string(-4) == "DOMINO_ERR_TIMEOUT"
    assert binding.domino_status_string(12345) == "DOMINO_ERR_UNKNOWN"


def test_invalid_sizes_rejected_without_device():
    _lib()
    good = dict(B=1, K=16, H=4096, V=151936, Ds=1024, R=256, k=8, N=16)
    for bad in (dict(B=0), dict(K=-1), dict(H=0), dict(V=0), dict(k=0), dict(N=0), dict(k=200, V=100),
                dict(K=2, k=2, N=7), dict(H=4100), dict(k=33), dict(N=257), dict(K=65), dict(V=1 << 22),
                dict(Ds=1000), dict(R=100), dict(Ds=4096)):
        args = dict(good, **bad)
        assert binding.domino_workspace_bytes(*args.values()) == 0, bad


def test_null_pointers_rejected_before_any_cuda_call():
    _lib()
    rc = binding.domino_draft_step(None, None, None, None, 1, 4, 64, 100, 2, 3, None, None, None, None, None,
                                   None, None, 0)
    assert rc == binding.DOMINO_ERR_INVALID_ARG


def test_input_table_size_and_argument_checks():
    """The input-projection table is V x 3 Ds fp32; NULL pointers and bad sizes are refused
    before any device query."""
    _lib()
    assert binding.domino_input_table_bytes(151936, 1024) == 151936 * 3 * 1024 * 4
    assert binding.domino_input_table_bytes(0, 1024) == 0
    assert binding.domino_input_table_bytes(10, 0) == 0
    bad = binding.DOMINO_ERR_INVALID_ARG
    assert binding.domino_build_input_table(None, None, 10, 8, 8, None) == bad
    one = 16  # a non-null stand-in; never dereferenced because validation fails first
    assert binding.domino_build_input_table(one, one, 0, 8, 8, one) == bad
    assert binding.domino_build_input_table(one, one, 10, 8, -8, one) == bad
    assert binding.domino_build_input_table(one, one, 10, 12, 8, one) == binding.DOMINO_ERR_UNSUPPORTED
    assert binding.domino_build_input_table(one, one, 10, 8, 4096, one) == binding.DOMINO_ERR_UNSUPPORTED
    # pointers must be 16-byte aligned (TMA); refused before any device query
    assert binding.domino_build_input_table(one + 2, one, 10, 8, 8, one) == binding.DOMINO_ERR_UNSUPPORTED
    assert binding.domino_build_input_table(one, one, 10, 8, 8, one + 4) == binding.DOMINO_ERR_UNSUPPORTED


def test_rollout_refuses_a_misaligned_input_table_before_any_device_call():
    _lib()
    one = 16  # non-null, 16-byte aligned stand-ins; never dereferenced
    head = binding.make_head(one, one, one, None, None, one, None, one, None, 16, 8, x_table=one + 4)
    rc = binding.domino_rollout_greedy(one, one, one, head, 1, 2, 64, 100, one, one, one, 1 << 20, None)
    assert rc == binding.DOMINO_ERR_INVALID_ARG


def test_launch_count_query():
    _lib()
    # B = 1: the GRU (with its own projections), the vocab GEMM, merge + tree
    assert binding.domino_launches_per_step(1, 16, 4096, 151936, 1024, 256, 8, 16) == 3
    # B = 4 (M = 64, no overlap): gather, X GEMM, W1-hidden GEMM, GRU, vocab GEMM, merge + tree
    assert binding.domino_launches_per_step(4, 16, 4096, 151936, 1024, 256, 8, 16) == 6
    # B = 32 (tokens on M): gather, X GEMM, GRU, W1 GEMM, u finalize, vocab GEMM, merge + tree
    assert binding.domino_launches_per_step(32, 16, 4096, 151936, 1024, 256, 8, 16) == 7
    assert binding.domino_launches_per_step(1, 16, 4096, 151936, 0, 0, 8, 16) == 3
    assert binding.domino_launches_per_step(0, 16, 4096, 151936, 1024, 256, 8, 16) < 0
    # with an input-projection table the X GEMM is not launched
    assert binding.domino_launches_per_step_table(1, 16, 4096, 151936, 1024, 256, 8, 16) == 3
    assert binding.domino_launches_per_step_table(4, 16, 4096, 151936, 1024, 256, 8, 16) == 5
    assert binding.domino_launches_per_step_table(32, 16, 4096, 151936, 1024, 256, 8, 16) == 6
    assert binding.domino_launches_per_step_table(1, 16, 4096, 151936, 0, 0, 8, 16) == 3
    assert binding.domino_launches_per_step_table(0, 16, 4096, 151936, 1024, 256, 8, 16) < 0


def test_verify_rejects_bad_arguments_before_launch():
    """Argument errors of domino_verify_tree_greedy come back before anything is enqueued."""
    f = binding.domino_verify_tree_greedy
    bad = binding.DOMINO_ERR_INVALID_ARG
    one = 1  # a non-null stand-in; never dereferenced because validation fails first
    assert f(one, one, one, 0, 4, 10, one, one, one, one) == bad        # B < 1
    assert f(one, one, one, 1, -1, 10, one, one, one, one) == bad       # N < 0
    assert f(one, one, one, 1, 4, 0, one, one, one, one) == bad         # V < 1
    assert f(None, one, one, 1, 4, 10, one, one, one, one) == bad       # no logits
    assert f(one, None, one, 1, 4, 10, one, one, one, one) == bad       # N > 0 without a tree
    assert f(one, one, one, 1, 4, 10, one, None, one, one) == bad       # no accepted_nodes


def test_verify_sample_rejects_bad_arguments_before_launch():
    """Argument errors of domino_verify_tree_sample (sizes, pointers, temperature, a vocabulary past
    the shared-memory staging limit) come back before anything is enqueued."""
    f = binding.domino_verify_tree_sample
    bad, unsup = binding.DOMINO_ERR_INVALID_ARG, binding.DOMINO_ERR_UNSUPPORTED
    one = 1  # a non-null stand-in; never dereferenced because validation fails first
    assert f(one, one, one, one, 1.0, 0, 4, 10, one, one, one, one) == bad       # B < 1
    assert f(one, one, one, one, 1.0, 1, -1, 10, one, one, one, one) == bad      # N < 0
    assert f(one, one, one, one, 1.0, 1, 4, 0, one, one, one, one) == bad        # V < 1
    assert f(one, one, one, None, 1.0, 1, 4, 10, one, one, one, one) == bad      # no uniforms
    assert f(one, None, one, one, 1.0, 1, 4, 10, one, one, one, one) == bad      # N > 0 without a tree
    assert f(one, one, one, one, 1.0, 1, 4, 10, None, one, one, one) == bad      # no row_sample
    for T in (0.0, -1.0, float("inf"), float("nan"), 1e-40):                     # 1 / 1e-40 overflows
        assert f(one, one, one, one, T, 1, 4, 10, one, one, one, one) == bad
    assert f(one, one, one, one, 1.0, 1, 4, 8 * 53248 + 1, one, one, one, one) == unsup


def test_rollout_rejects_bad_sizes_before_any_device_work():
    f = binding.domino_rollout_workspace_bytes
    assert f(0, 4, 256, 100, 64, 64) == 0       # B < 1
    assert f(9, 4, 256, 100, 64, 64) == 0       # B above the rollout's 8
    assert f(1, 4, 250, 100, 64, 64) == 0       # H not a multiple of 8
    assert f(1, 4, 256, 100, 60, 64) == 0       # d_s not a multiple of 8
    assert binding.domino_rollout_greedy(None, None, None, None, 1, 4, 256, 100, None, None, None, 0) == \
        binding.DOMINO_ERR_INVALID_ARG
    assert binding.domino_rollout_sample_gumbel(None, None, 1, None, None, 1, 4, 256, 100, None, None, None, 0) == \
        binding.DOMINO_ERR_INVALID_ARG
    assert binding.domino_rollout_sample_gumbel(None, None, (1 << 64) - 1, None, None, 1, 4, 256, 100, None, None,
                                                None, 0) == binding.DOMINO_ERR_INVALID_ARG


def test_debug_hold_argument_checks_and_header_constants():
    """The failure-detection hook refuses unknown kinds and negative CTAs / positions before any
    device call, and its constants match the header's."""
    _lib()
    with open(os.path.join(ROOT, "include", "domino.h")) as f:
        text = f.read()
    for name in ("DOMINO_HOLD_OFF", "DOMINO_HOLD_STATE", "DOMINO_HOLD_CLEAR_BARRIER"):
        m = re.search(name + r"\s*=\s*(\d+)", text)
        assert m and int(m.group(1)) == getattr(binding, name), name
    bad = binding.DOMINO_ERR_INVALID_ARG
    assert binding.domino_debug_hold(7, 0, 0) == bad
    assert binding.domino_debug_hold(-1, 0, 0) == bad
    assert binding.domino_debug_hold(binding.DOMINO_HOLD_STATE, -1, 0) == bad
    assert binding.domino_debug_hold(binding.DOMINO_HOLD_STATE, 0, -1) == bad
    assert binding.domino_debug_hold(binding.DOMINO_HOLD_STATE, 0, 64) == bad
    assert binding.domino_debug_hold(binding.DOMINO_HOLD_CLEAR_BARRIER, -3) == bad
