"""Python access to the fp64 CPU oracle of the Domino draft-side block step.

TEST INFRASTRUCTURE ONLY.  The oracle is a plain C library (``domino_oracle.c``)
that writes out each step of the method as the paper defines it (Domino,
arXiv 2605.29707, sections 4.1.1 and 4.1.2; the tree as a best-first selection).
It is imported by the tests, by ``__graft_entry__.smoke()`` and by the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py``; the product path
never imports it.  It shares no code with the CUDA library and does not import
the package.

bf16 tensors travel as numpy ``uint16`` bit patterns; activations are float64.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "domino_oracle.c")
_LIB_PATH = os.path.join(_HERE, "liboracle.so")
_lib = None

ERR_ARG = -1
ERR_TOKEN = -2


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (OpenMP, IEEE double, no FMA contraction)."""
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp", "-ffp-contract=off",
               "-o", _LIB_PATH + ".tmp", _SRC, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(_LIB_PATH + ".tmp", _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    if _lib is None:
        build()
        _lib = ctypes.CDLL(_LIB_PATH)
        P = ctypes.c_void_p
        I = ctypes.c_int
        _lib.oracle_bf16_to_double.restype = ctypes.c_double
        _lib.oracle_bf16_to_double.argtypes = [ctypes.c_uint16]
        _lib.oracle_embed.argtypes = [P, I, I, P, I, P]
        _lib.oracle_gru.argtypes = [P, I, I, I, P, P, P, P, P]
        _lib.oracle_lowrank.argtypes = [P, P, I, I, I, I, P, P, P]
        _lib.oracle_logits.argtypes = [P, P, I, I, I, I, P, P, P, P, I]
        _lib.oracle_log_softmax.argtypes = [P, I, I, P, P]
        _lib.oracle_topk.argtypes = [P, I, I, I, P, P]
        _lib.oracle_tree.argtypes = [P, P, I, I, I, P, P, P, P]
        _lib.oracle_draft_step.argtypes = [P] * 12 + [I] * 8 + [P, I] + [P] * 8 + [I]
        _lib.oracle_verify_greedy.argtypes = [P, I, I, P, P, P, P, P, P]
        _lib.oracle_tree_walk.argtypes = [I, P, P, P, P, P, P]
        _lib.oracle_row_sample.argtypes = [P, I, ctypes.c_double, ctypes.c_double, P]
        _lib.oracle_verify_sample.argtypes = [P, I, I, ctypes.c_double, P, P, P, P, P, P, P]
        _lib.oracle_rollout_greedy.argtypes = [P] * 12 + [I] * 6 + [P, I, P, P, I]
        _lib.oracle_rollout_sample.argtypes = [P] * 13 + [I] * 6 + [P, I, P, P, I]
        U64 = ctypes.c_uint64
        _lib.oracle_philox4x32_10.restype = None
        _lib.oracle_philox4x32_10.argtypes = [P, P, P]
        _lib.oracle_gumbel_row.argtypes = [U64, I, I, I, P]
        _lib.oracle_rollout_sample_gumbel.argtypes = [P, P, U64] + [P] * 10 + [I] * 6 + [P, I, P, P, I]
        _lib.oracle_max_threads.restype = I
        for name in ("oracle_embed", "oracle_gru", "oracle_lowrank", "oracle_logits",
                     "oracle_log_softmax", "oracle_topk", "oracle_tree", "oracle_draft_step"):
            getattr(_lib, name).restype = I
    return _lib


def _p(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _u16(a):
    if a is None:
        return None
    a = np.ascontiguousarray(a)
    assert a.dtype == np.uint16, a.dtype
    return a


def _f64(a):
    return np.ascontiguousarray(a, dtype=np.float64)


def _i32(a):
    return np.ascontiguousarray(a, dtype=np.int32)


def _check(rc, what):
    if rc != 0:
        raise OracleError(rc, what)


class OracleError(RuntimeError):
    def __init__(self, rc, what):
        super().__init__(f"{what} returned {rc}")
        self.rc = rc


def max_threads() -> int:
    return int(_load().oracle_max_threads())


def bf16_to_double(b: int) -> float:
    return float(_load().oracle_bf16_to_double(int(b)))


def embed(emb, ids):
    emb = _u16(emb); ids = _i32(ids)
    V, H = emb.shape
    E = np.empty((ids.size, H), np.float64)
    _check(_load().oracle_embed(_p(emb), V, H, _p(ids), ids.size, _p(E)), "oracle_embed")
    return E


def gru(E, w_ih, w_hh, b_ih=None, b_hh=None):
    E = _f64(E); w_ih = _u16(w_ih); w_hh = _u16(w_hh); b_ih = _u16(b_ih); b_hh = _u16(b_hh)
    K, Hin = E.shape
    Ds = w_hh.shape[1]
    S = np.empty((K, Ds), np.float64)
    _check(_load().oracle_gru(_p(E), K, Hin, Ds, _p(w_ih), _p(w_hh), _p(b_ih), _p(b_hh), _p(S)),
           "oracle_gru")
    return S


def lowrank(hidden, S, w1, b1=None):
    hidden = _f64(hidden); S = _f64(S); w1 = _u16(w1); b1 = _u16(b1)
    K, H = hidden.shape
    Ds = S.shape[1]
    R = w1.shape[0]
    u = np.empty((K, R), np.float64)
    _check(_load().oracle_lowrank(_p(hidden), _p(S), K, H, Ds, R, _p(w1), _p(b1), _p(u)),
           "oracle_lowrank")
    return u


def logits(hidden, u, w_lm, w2=None, b2=None, nthreads=0):
    hidden = _f64(hidden); w_lm = _u16(w_lm); w2 = _u16(w2); b2 = _u16(b2)
    K, H = hidden.shape
    V = w_lm.shape[0]
    R = 0 if w2 is None else w2.shape[1]
    u = None if u is None else _f64(u)
    z = np.empty((K, V), np.float64)
    _check(_load().oracle_logits(_p(hidden), _p(u), K, H, V, R, _p(w_lm), _p(w2), _p(b2), _p(z),
                                 nthreads), "oracle_logits")
    return z


def log_softmax(z):
    z = _f64(z)
    n, V = z.shape
    lp = np.empty_like(z)
    lse = np.empty(n, np.float64)
    _check(_load().oracle_log_softmax(_p(z), n, V, _p(lp), _p(lse)), "oracle_log_softmax")
    return lp, lse


def topk(logp, k):
    logp = _f64(logp)
    n, V = logp.shape
    ids = np.empty((n, k), np.int32)
    vals = np.empty((n, k), np.float64)
    _check(_load().oracle_topk(_p(logp), n, V, k, _p(ids), _p(vals)), "oracle_topk")
    return ids, vals


def tree(topk_ids, topk_logp, N):
    topk_ids = _i32(topk_ids); topk_logp = _f64(topk_logp)
    K, k = topk_ids.shape
    par = np.empty(N, np.int32); tok = np.empty(N, np.int32); dep = np.empty(N, np.int32)
    sc = np.empty(N, np.float64)
    _check(_load().oracle_tree(_p(topk_ids), _p(topk_logp), K, k, N, _p(par), _p(tok), _p(dep),
                               _p(sc)), "oracle_tree")
    return par, tok, dep, sc


def verify_greedy(target, parent, token):
    """Greedy tree verification of one sequence: target fp32 [N+1, V], parent/token [N].
    Returns (row_argmax [N+1], accepted nodes [n_acc], bonus token)."""
    target = np.ascontiguousarray(target, np.float32)
    parent = _i32(parent); token = _i32(token)
    N = parent.shape[0]
    V = target.shape[1]
    if target.shape[0] != N + 1:
        raise OracleError(-1, "oracle_verify_greedy: target must have N + 1 rows")
    ra = np.empty(N + 1, np.int32); nodes = np.empty(max(N, 1), np.int32)
    n = np.zeros(1, np.int32); bonus = np.zeros(1, np.int32)
    _check(_load().oracle_verify_greedy(_p(target), N, V, _p(parent), _p(token), _p(ra), _p(nodes), _p(n),
                                        _p(bonus)), "oracle_verify_greedy")
    return ra, nodes[: int(n[0])].copy(), int(bonus[0])


def tree_walk(parent, token, row_choice):
    """The verification walk of one tree for given per-row target choices [N+1].
    Returns (accepted nodes [n_acc], bonus token)."""
    parent = _i32(parent); token = _i32(token); row_choice = _i32(row_choice)
    N = parent.shape[0]
    if row_choice.shape[0] != N + 1:
        raise OracleError(-1, "oracle_tree_walk: row_choice must have N + 1 entries")
    nodes = np.empty(max(N, 1), np.int32)
    n = np.zeros(1, np.int32); bonus = np.zeros(1, np.int32)
    _check(_load().oracle_tree_walk(N, _p(parent), _p(token), _p(row_choice), _p(nodes), _p(n), _p(bonus)),
           "oracle_tree_walk")
    return nodes[: int(n[0])].copy(), int(bonus[0])


def row_sample(row, T, u):
    """One draw from softmax(row / T) with uniform u in [0, 1) (first id whose cumulative
    probability in id order exceeds u)."""
    row = np.ascontiguousarray(row, np.float32)
    out = np.zeros(1, np.int32)
    _check(_load().oracle_row_sample(_p(row), row.shape[0], float(T), float(u), _p(out)), "oracle_row_sample")
    return int(out[0])


def verify_sample(target, parent, token, T, uniforms):
    """Tree verification of one sequence at temperature T > 0: target fp32 [N+1, V],
    parent/token [N], uniforms fp32 [N+1].  Returns (row_sample [N+1], accepted nodes, bonus)."""
    target = np.ascontiguousarray(target, np.float32)
    parent = _i32(parent); token = _i32(token)
    uniforms = np.ascontiguousarray(uniforms, np.float32)
    N = parent.shape[0]
    V = target.shape[1]
    if target.shape[0] != N + 1 or uniforms.shape[0] != N + 1:
        raise OracleError(-1, "oracle_verify_sample: target and uniforms must have N + 1 rows")
    rs = np.empty(N + 1, np.int32); nodes = np.empty(max(N, 1), np.int32)
    n = np.zeros(1, np.int32); bonus = np.zeros(1, np.int32)
    _check(_load().oracle_verify_sample(_p(target), N, V, float(T), _p(uniforms), _p(parent), _p(token), _p(rs),
                                        _p(nodes), _p(n), _p(bonus)), "oracle_verify_sample")
    return rs, nodes[: int(n[0])].copy(), int(bonus[0])


def rollout_greedy(w, hidden, anchors, seqs=None, nthreads=0):
    """Greedy sequential draft loop.  ``w`` and ``hidden`` as for draft_step; anchors int32 [B].
    Returns (tokens int32 [nseq, K], logp float64 [nseq, K])."""
    hidden = _u16(hidden)
    B, K, H = hidden.shape
    anchors = _i32(anchors)
    g = lambda n: _u16(w[n]) if w.get(n) is not None else None  # noqa: E731
    w_lm = g("w_lm")
    V = w_lm.shape[0]
    w2 = g("w2")
    R = w2.shape[1] if w2 is not None else 0
    w_hh = g("w_hh")
    Ds = w_hh.shape[1] if w_hh is not None else 0
    sq = None if seqs is None else _i32(seqs)
    nseq = B if sq is None else sq.shape[0]
    tokens = np.empty((nseq, K), np.int32)
    logp = np.empty((nseq, K), np.float64)
    _check(_load().oracle_rollout_greedy(_p(hidden), _p(anchors), _p(w_lm), _p(g("emb")), _p(g("w_ih")), _p(w_hh),
                                         _p(g("b_ih")), _p(g("b_hh")), _p(g("w1")), _p(g("b1")), _p(w2),
                                         _p(g("b2")), B, K, H, V, Ds, R, _p(sq), nseq, _p(tokens), _p(logp),
                                         nthreads), "oracle_rollout_greedy")
    return tokens, logp


def rollout_sample(w, hidden, anchors, uniforms, seqs=None, nthreads=0):
    """Sampled sequential draft loop: ``uniforms`` float32 [B, K] in [0, 1), the caller's random
    draws (one per sequence and step).  Otherwise as rollout_greedy."""
    hidden = _u16(hidden)
    B, K, H = hidden.shape
    anchors = _i32(anchors)
    uni = np.ascontiguousarray(uniforms, dtype=np.float32).reshape(B, K)
    g = lambda n: _u16(w[n]) if w.get(n) is not None else None  # noqa: E731
    w_lm = g("w_lm")
    V = w_lm.shape[0]
    w2 = g("w2")
    R = w2.shape[1] if w2 is not None else 0
    w_hh = g("w_hh")
    Ds = w_hh.shape[1] if w_hh is not None else 0
    sq = None if seqs is None else _i32(seqs)
    nseq = B if sq is None else sq.shape[0]
    tokens = np.empty((nseq, K), np.int32)
    logp = np.empty((nseq, K), np.float64)
    _check(_load().oracle_rollout_sample(_p(hidden), _p(anchors), _p(uni), _p(w_lm), _p(g("emb")), _p(g("w_ih")),
                                         _p(w_hh), _p(g("b_ih")), _p(g("b_hh")), _p(g("w1")), _p(g("b1")), _p(w2),
                                         _p(g("b2")), B, K, H, V, Ds, R, _p(sq), nseq, _p(tokens), _p(logp),
                                         nthreads), "oracle_rollout_sample")
    return tokens, logp


def philox4x32_10(ctr, key):
    """Philox-4x32-10 of a 4-word counter and a 2-word key (uint32 each); returns 4 words."""
    c = np.ascontiguousarray(ctr, dtype=np.uint32).reshape(4)
    k = np.ascontiguousarray(key, dtype=np.uint32).reshape(2)
    out = np.empty(4, np.uint32)
    _load().oracle_philox4x32_10(_p(c), _p(k), _p(out))
    return out


def gumbel_row(seed, b, j, V):
    """The exponential-race perturbations g[0 .. V-1] of sequence b at step j (float64 [V])."""
    g = np.empty(V, np.float64)
    _check(_load().oracle_gumbel_row(int(seed), int(b), int(j), int(V), _p(g)), "oracle_gumbel_row")
    return g


def rollout_sample_gumbel(w, hidden, anchors, seed, seqs=None, nthreads=0):
    """Sampled sequential draft loop by the exponential race (Gumbel-max) under a 64-bit seed:
    t_{j+1} = argmax_v L_j[v] + gumbel_row(seed, b, j, V)[v].  Otherwise as rollout_greedy."""
    hidden = _u16(hidden)
    B, K, H = hidden.shape
    anchors = _i32(anchors)
    g = lambda n: _u16(w[n]) if w.get(n) is not None else None  # noqa: E731
    w_lm = g("w_lm")
    V = w_lm.shape[0]
    w2 = g("w2")
    R = w2.shape[1] if w2 is not None else 0
    w_hh = g("w_hh")
    Ds = w_hh.shape[1] if w_hh is not None else 0
    sq = None if seqs is None else _i32(seqs)
    nseq = B if sq is None else sq.shape[0]
    tokens = np.empty((nseq, K), np.int32)
    logp = np.empty((nseq, K), np.float64)
    _check(_load().oracle_rollout_sample_gumbel(_p(hidden), _p(anchors), int(seed), _p(w_lm), _p(g("emb")),
                                                _p(g("w_ih")), _p(w_hh), _p(g("b_ih")), _p(g("b_hh")), _p(g("w1")),
                                                _p(g("b1")), _p(w2), _p(g("b2")), B, K, H, V, Ds, R, _p(sq), nseq,
                                                _p(tokens), _p(logp), nthreads), "oracle_rollout_sample_gumbel")
    return tokens, logp


def draft_step(w, hidden, prefix_ids, k, N, seqs=None, want_logp_full=False, nthreads=0):
    """Run the whole step.

    ``w`` maps weight names (``w_lm emb w_ih w_hh b_ih b_hh w1 b1 w2 b2``) to uint16
    arrays or None; ``hidden`` is uint16 [B, K, H]; ``prefix_ids`` int32 [B, K].
    Returns a dict of numpy arrays indexed by the position in ``seqs``.
    """
    hidden = _u16(hidden); ids = _i32(prefix_ids)
    B, K, H = hidden.shape
    w_lm = _u16(w["w_lm"])
    V = w_lm.shape[0]
    w2 = _u16(w.get("w2"))
    R = 0 if w2 is None else w2.shape[1]
    w_hh = _u16(w.get("w_hh"))
    Ds = 0 if w_hh is None else w_hh.shape[1]
    sel = None if seqs is None else _i32(np.asarray(seqs))
    nseq = B if sel is None else sel.size
    out = {
        "logp_full": np.empty((nseq, K, V), np.float64) if want_logp_full else None,
        "lse": np.empty((nseq, K), np.float64),
        "topk_ids": np.empty((nseq, K, k), np.int32),
        "topk_logp": np.empty((nseq, K, k), np.float64),
        "tree_parent": np.empty((nseq, N), np.int32),
        "tree_token": np.empty((nseq, N), np.int32),
        "tree_depth": np.empty((nseq, N), np.int32),
        "tree_score": np.empty((nseq, N), np.float64),
    }
    args = [_p(hidden), _p(ids), _p(w_lm)] + [_p(_u16(w.get(n))) for n in
                                              ("emb", "w_ih", "w_hh", "b_ih", "b_hh", "w1", "b1")]
    args += [_p(w2), _p(_u16(w.get("b2")))]
    args += [B, K, H, V, Ds, R, k, N, _p(sel), nseq]
    args += [_p(out[n]) for n in ("logp_full", "lse", "topk_ids", "topk_logp", "tree_parent",
                                  "tree_token", "tree_depth", "tree_score")]
    args += [nthreads]
    _check(_load().oracle_draft_step(*args), "oracle_draft_step")
    return out
