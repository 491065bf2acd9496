"""ctypes binding of the C ABI in include/domino.h (argument marshalling only).

Every function here has the name of the C entry point it calls.  Tensor arguments may be
torch tensors (their data_ptr() is passed) or raw integer addresses; the library itself
does all the work.  Loading fails loudly when libdomino.so has not been built: there is no
fallback implementation.
"""
from __future__ import annotations

import ctypes
import os

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libdomino.so")

DOMINO_OK = 0
DOMINO_ERR_INVALID_ARG = -1
DOMINO_ERR_UNSUPPORTED = -2
DOMINO_ERR_CUDA = -3
DOMINO_ERR_TIMEOUT = -4
DOMINO_ERR_BAD_TOKEN = -5

# every entry point declared in include/domino.h
SYMBOLS = ("domino_workspace_bytes", "domino_draft_step", "domino_workspace_bytes_host",
           "domino_draft_step_host", "domino_check_status", "domino_status_string",
           "domino_abi_version", "domino_launches_per_step", "domino_timing_begin", "domino_timing_end",
           "domino_draft_step_static_scratch", "domino_verify_tree_greedy", "domino_rollout_workspace_bytes",
           "domino_rollout_greedy", "domino_rollout_sample", "domino_input_table_bytes",
           "domino_build_input_table", "domino_launches_per_step_table", "domino_debug_hold",
           "domino_verify_tree_sample", "domino_rollout_sample_gumbel")

DOMINO_STATIC_SCRATCH_BYTES = 16 << 20

# domino_debug_hold: what a GRU CTA withholds (a failure-detection test hook)
DOMINO_HOLD_OFF = 0
DOMINO_HOLD_STATE = 1
DOMINO_HOLD_CLEAR_BARRIER = 2

KERNEL_KINDS = ("gather", "gru_input_proj", "w1_hidden_proj", "gru", "vocab_gemm_softmax_topk", "merge_tree",
                "rollout_base_gemm", "rollout_steps", "tree_verify")


class domino_head_weights(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in
                ("emb", "w_ih", "w_hh", "b_ih", "b_hh", "w1", "b1", "w2", "b2")] + \
               [("Ds", ctypes.c_int), ("R", ctypes.c_int), ("x_table", ctypes.c_void_p)]


class DominoError(RuntimeError):
    def __init__(self, code: int, what: str = ""):
        super().__init__(f"{what}: {domino_status_string(code)} ({code})" if what else domino_status_string(code))
        self.code = code


_lib = None


def load():
    """Load libdomino.so (raises if it is missing)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is missing: build it with __graft_entry__.build() "
                           "(there is no non-CUDA implementation)")
    lib = ctypes.CDLL(LIB_PATH)
    P, I, S = ctypes.c_void_p, ctypes.c_int, ctypes.c_size_t
    lib.domino_workspace_bytes.argtypes = [I] * 8
    lib.domino_workspace_bytes.restype = S
    lib.domino_workspace_bytes_host.argtypes = [I] * 8
    lib.domino_workspace_bytes_host.restype = S
    step_args = [P, P, P, ctypes.POINTER(domino_head_weights)] + [I] * 6 + [P] * 6 + [P, S, P]
    lib.domino_draft_step.argtypes = step_args
    lib.domino_draft_step.restype = I
    lib.domino_draft_step_host.argtypes = step_args
    lib.domino_draft_step_host.restype = I
    lib.domino_check_status.argtypes = [P, P]
    lib.domino_check_status.restype = I
    lib.domino_status_string.argtypes = [I]
    lib.domino_status_string.restype = ctypes.c_char_p
    lib.domino_abi_version.argtypes = []
    lib.domino_abi_version.restype = I
    lib.domino_launches_per_step.argtypes = [I] * 8
    lib.domino_launches_per_step.restype = I
    lib.domino_launches_per_step_table.argtypes = [I] * 8
    lib.domino_launches_per_step_table.restype = I
    lib.domino_timing_begin.argtypes = [I]
    lib.domino_timing_begin.restype = I
    lib.domino_timing_end.argtypes = [P, P, I]
    lib.domino_timing_end.restype = I
    lib.domino_draft_step_static_scratch.argtypes = [P, P, P, ctypes.POINTER(domino_head_weights)] + [I] * 6 + \
        [P] * 6 + [P, P]
    lib.domino_draft_step_static_scratch.restype = I
    lib.domino_verify_tree_greedy.argtypes = [P, P, P, I, I, I, P, P, P, P, P]
    lib.domino_verify_tree_greedy.restype = I
    lib.domino_verify_tree_sample.argtypes = [P, P, P, P, ctypes.c_float, I, I, I, P, P, P, P, P]
    lib.domino_verify_tree_sample.restype = I
    lib.domino_rollout_workspace_bytes.argtypes = [I] * 6
    lib.domino_rollout_workspace_bytes.restype = ctypes.c_size_t
    lib.domino_rollout_greedy.argtypes = [P, P, P, ctypes.POINTER(domino_head_weights)] + [I] * 4 + [P, P, P,
                                                                                               ctypes.c_size_t, P]
    lib.domino_rollout_greedy.restype = I
    lib.domino_rollout_sample.argtypes = [P, P, P, P, ctypes.POINTER(domino_head_weights)] + [I] * 4 + [
        P, P, P, ctypes.c_size_t, P]
    lib.domino_rollout_sample.restype = I
    lib.domino_rollout_sample_gumbel.argtypes = [P, P, ctypes.c_uint64, P, ctypes.POINTER(domino_head_weights)] + [
        I] * 4 + [P, P, P, ctypes.c_size_t, P]
    lib.domino_rollout_sample_gumbel.restype = I
    lib.domino_input_table_bytes.argtypes = [I, I]
    lib.domino_input_table_bytes.restype = S
    lib.domino_build_input_table.argtypes = [P, P, I, I, I, P, P]
    lib.domino_build_input_table.restype = I
    lib.domino_debug_hold.argtypes = [I, I, I]
    lib.domino_debug_hold.restype = I
    _lib = lib
    return lib


def _addr(x):
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if hasattr(x, "data_ptr"):
        return x.data_ptr()
    if hasattr(x, "ctypes"):  # numpy array
        return x.ctypes.data
    raise TypeError(f"cannot take the address of {type(x)}")


def _stream(s):
    if s is None:
        return None
    if isinstance(s, int):
        return s
    return s.cuda_stream  # torch.cuda.Stream


def make_head(emb=None, w_ih=None, w_hh=None, b_ih=None, b_hh=None, w1=None, b1=None, w2=None, b2=None,
              Ds=0, R=0, x_table=None) -> domino_head_weights:
    return domino_head_weights(_addr(emb), _addr(w_ih), _addr(w_hh), _addr(b_ih), _addr(b_hh), _addr(w1),
                               _addr(b1), _addr(w2), _addr(b2), int(Ds), int(R), _addr(x_table))


def domino_input_table_bytes(V, Ds) -> int:
    return int(load().domino_input_table_bytes(V, Ds))


def domino_build_input_table(emb, w_ih, V, H, Ds, table, stream=None) -> int:
    """table [V, 3 Ds] fp32 = emb . W_ih^T (device); synchronises the stream."""
    return int(load().domino_build_input_table(_addr(emb), _addr(w_ih), V, H, Ds, _addr(table), _stream(stream)))


def domino_workspace_bytes(B, K, H, V, Ds, R, k, N) -> int:
    return int(load().domino_workspace_bytes(B, K, H, V, Ds, R, k, N))


def domino_workspace_bytes_host(B, K, H, V, Ds, R, k, N) -> int:
    return int(load().domino_workspace_bytes_host(B, K, H, V, Ds, R, k, N))


def domino_draft_step(hidden, prefix_ids, w_lm, head, B, K, H, V, k, N, topk_ids, topk_logp, tree_parent,
                      tree_token, tree_depth, tree_score, workspace, workspace_bytes, stream=None) -> int:
    h = ctypes.byref(head) if head is not None else None
    return int(load().domino_draft_step(_addr(hidden), _addr(prefix_ids), _addr(w_lm), h, B, K, H, V, k, N,
                                        _addr(topk_ids), _addr(topk_logp), _addr(tree_parent),
                                        _addr(tree_token), _addr(tree_depth), _addr(tree_score),
                                        _addr(workspace), int(workspace_bytes), _stream(stream)))


def domino_draft_step_host(hidden_host, prefix_ids_host, w_lm, head, B, K, H, V, k, N, topk_ids_host,
                           topk_logp_host, tree_parent_host, tree_token_host, tree_depth_host, tree_score_host,
                           workspace, workspace_bytes, stream=None) -> int:
    h = ctypes.byref(head) if head is not None else None
    return int(load().domino_draft_step_host(
        _addr(hidden_host), _addr(prefix_ids_host), _addr(w_lm), h, B, K, H, V, k, N, _addr(topk_ids_host),
        _addr(topk_logp_host), _addr(tree_parent_host), _addr(tree_token_host), _addr(tree_depth_host),
        _addr(tree_score_host), _addr(workspace), int(workspace_bytes), _stream(stream)))


def domino_check_status(workspace, stream=None) -> int:
    return int(load().domino_check_status(_addr(workspace), _stream(stream)))


def domino_status_string(code: int) -> str:
    return load().domino_status_string(int(code)).decode()


def domino_abi_version() -> int:
    return int(load().domino_abi_version())


def domino_launches_per_step(B, K, H, V, Ds, R, k, N) -> int:
    return int(load().domino_launches_per_step(B, K, H, V, Ds, R, k, N))


def domino_launches_per_step_table(B, K, H, V, Ds, R, k, N) -> int:
    return int(load().domino_launches_per_step_table(B, K, H, V, Ds, R, k, N))


def domino_timing_begin(max_launches: int) -> int:
    return int(load().domino_timing_begin(int(max_launches)))


def domino_timing_end() -> dict:
    """Stops per-kernel timing; returns {kind name: (total ms, launches)}."""
    n = len(KERNEL_KINDS)
    ms = (ctypes.c_float * n)()
    cnt = (ctypes.c_int * n)()
    rc = int(load().domino_timing_end(ctypes.cast(ms, ctypes.c_void_p), ctypes.cast(cnt, ctypes.c_void_p), n))
    if rc != 0:
        raise DominoError(rc, "domino_timing_end")
    return {KERNEL_KINDS[i]: (float(ms[i]), int(cnt[i])) for i in range(n)}


def domino_draft_step_static_scratch(hidden, prefix_ids, w_lm, head, B, K, H, V, k, N, topk_ids, topk_logp,
                                     tree_parent, tree_token, tree_depth, tree_score, device_status=None,
                                     stream=None) -> int:
    """The draft step for callers that cannot allocate device memory: no workspace argument;
    the library's own static 16 MiB device array serves as scratch (see include/domino.h)."""
    h = ctypes.byref(head) if head is not None else None
    return int(load().domino_draft_step_static_scratch(
        _addr(hidden), _addr(prefix_ids), _addr(w_lm), h, B, K, H, V, k, N, _addr(topk_ids), _addr(topk_logp),
        _addr(tree_parent), _addr(tree_token), _addr(tree_depth), _addr(tree_score), _addr(device_status),
        _stream(stream)))


def domino_verify_tree_greedy(target_logits, tree_parent, tree_token, B, N, V, row_argmax, accepted_nodes,
                              accepted_count, bonus_token, stream=None) -> int:
    """Greedy verification of B draft trees against the target's fp32 logits [B, N+1, V] (device)."""
    return int(load().domino_verify_tree_greedy(_addr(target_logits), _addr(tree_parent), _addr(tree_token), B, N, V,
                                                _addr(row_argmax), _addr(accepted_nodes), _addr(accepted_count),
                                                _addr(bonus_token), _stream(stream)))


def domino_verify_tree_sample(target_logits, tree_parent, tree_token, uniforms, temperature, B, N, V, row_sample,
                              accepted_nodes, accepted_count, bonus_token, stream=None) -> int:
    """Verification at temperature T > 0 of B draft trees against the target's fp32 logits
    [B, N+1, V] with one uniform per row [B, N+1] (device)."""
    return int(load().domino_verify_tree_sample(_addr(target_logits), _addr(tree_parent), _addr(tree_token),
                                                _addr(uniforms), float(temperature), B, N, V, _addr(row_sample),
                                                _addr(accepted_nodes), _addr(accepted_count), _addr(bonus_token),
                                                _stream(stream)))


def domino_rollout_workspace_bytes(B, K, H, V, Ds, R) -> int:
    return int(load().domino_rollout_workspace_bytes(B, K, H, V, Ds, R))


def domino_rollout_greedy(hidden, anchors, w_lm, head, B, K, H, V, tokens, logp, workspace, workspace_bytes,
                          stream=None) -> int:
    """Greedy sequential draft loop: tokens t_1..t_K [B, K] and their log-probabilities (device)."""
    h = ctypes.byref(head) if head is not None else None
    return int(load().domino_rollout_greedy(_addr(hidden), _addr(anchors), _addr(w_lm), h, B, K, H, V,
                                            _addr(tokens), _addr(logp), _addr(workspace), int(workspace_bytes),
                                            _stream(stream)))


def domino_rollout_sample(hidden, anchors, uniforms, w_lm, head, B, K, H, V, tokens, logp, workspace,
                          workspace_bytes, stream=None) -> int:
    """Sampled sequential draft loop: ``uniforms`` device float32 [B, K] in [0, 1)."""
    h = ctypes.byref(head) if head is not None else None
    return int(load().domino_rollout_sample(_addr(hidden), _addr(anchors), _addr(uniforms), _addr(w_lm), h, B, K, H,
                                            V, _addr(tokens), _addr(logp), _addr(workspace), int(workspace_bytes),
                                            _stream(stream)))


def domino_rollout_sample_gumbel(hidden, anchors, seed, w_lm, head, B, K, H, V, tokens, logp, workspace,
                                 workspace_bytes, stream=None) -> int:
    """Sampled sequential draft loop by the exponential race under a 64-bit ``seed``."""
    h = ctypes.byref(head) if head is not None else None
    return int(load().domino_rollout_sample_gumbel(_addr(hidden), _addr(anchors), int(seed) & ((1 << 64) - 1),
                                                   _addr(w_lm), h, B, K, H, V, _addr(tokens), _addr(logp),
                                                   _addr(workspace), int(workspace_bytes), _stream(stream)))


def domino_debug_hold(what, gru_cta=-1, step=-1) -> int:
    """Test hook: the next GRU launch's CTA ``gru_cta`` withholds its states of position ``step``
    (DOMINO_HOLD_STATE) or its clear-barrier arrival (DOMINO_HOLD_CLEAR_BARRIER); DOMINO_HOLD_OFF
    disarms.  The step then reports DOMINO_ERR_TIMEOUT through its device status."""
    return int(load().domino_debug_hold(int(what), int(gru_cta), int(step)))
