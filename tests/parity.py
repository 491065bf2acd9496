"""Gap-aware comparison of the CUDA step's outputs with the fp64 oracle.

Rules (floating point: bf16 inputs, fp32 accumulation on the GPU, fp64 in the oracle):
  * every refined log-prob the GPU reports is within LOGP_TOL of the oracle's log-prob of
    the same token;
  * top-k ids: rank q's token must be distinct, and its oracle log-prob within GAP of the
    oracle's q-th value; it must equal the oracle's token wherever the oracle's gaps around
    rank q (to ranks q-1, q+1 and k+1) exceed GAP;
  * tree: replaying the GPU's picks in order, each pick must be a not-yet-picked child (from
    the GPU's own top-k lists) of the anchor or of an earlier pick, and its oracle cumulative
    score must be within GAP of the best such candidate; where the best candidate leads by more
    than GAP the pick is that candidate.  GPU scores match the oracle's cumulative score of the
    same path within LOGP_TOL (the same bound as a single log-prob, at every depth).
Differences that these rules excuse are counted and returned.
"""
from __future__ import annotations

import numpy as np

LOGP_TOL = 2e-2
GAP = 4e-2


def check_topk(gpu_ids, gpu_logp, logp_full, k, logp_tol=LOGP_TOL, gap=GAP):
    """gpu_ids / gpu_logp: [rows, k]; logp_full: oracle [rows, V].  Returns #excused mismatches."""
    rows = gpu_ids.shape[0]
    excused = 0
    for r in range(rows):
        lp = logp_full[r]
        order = np.lexsort((np.arange(lp.size), -lp))[: k + 1]
        ovals = lp[order]
        ids = gpu_ids[r]
        assert len(set(ids.tolist())) == k, f"row {r}: duplicate ids {ids}"
        assert np.all((ids >= 0) & (ids < lp.size)), f"row {r}: id out of range {ids}"
        for q in range(k):
            g = int(ids[q])
            assert abs(lp[g] - ovals[q]) <= gap, (
                f"row {r} rank {q}: gpu token {g} (oracle logp {lp[g]:.5f}) vs oracle rank value {ovals[q]:.5f}")
            assert abs(float(gpu_logp[r, q]) - lp[g]) <= logp_tol, (
                f"row {r} rank {q}: gpu logp {gpu_logp[r, q]:.5f} vs oracle {lp[g]:.5f}")
            lo = ovals[q] - ovals[q + 1] if q + 1 < ovals.size else np.inf
            hi = ovals[q - 1] - ovals[q] if q > 0 else np.inf
            if min(lo, hi) > gap:
                assert g == int(order[q]), f"row {r} rank {q}: gpu {g} != oracle {int(order[q])} (clear gap)"
            elif g != int(order[q]):
                excused += 1
    return excused


def check_tree(par, tok, dep, score, gpu_topk_ids, logp_full, K, N, logp_tol=LOGP_TOL, gap=GAP,
               oracle_tree=None):
    """One sequence.  gpu_topk_ids: [K, k]; logp_full: oracle [K, V].  Returns #excused."""
    par = np.asarray(par); tok = np.asarray(tok); dep = np.asarray(dep)
    k = gpu_topk_ids.shape[1]
    oscore = []                      # oracle cumulative score of each GPU node
    picked = set()                   # (parent, token)
    expanded = [(-1, 0, 0.0)]        # (node index or -1 for the anchor, depth, oracle score)
    for i in range(N):
        p, t, d = int(par[i]), int(tok[i]), int(dep[i])
        assert -1 <= p < i, f"node {i}: parent {p}"
        pd = 0 if p < 0 else int(dep[p])
        assert d == pd + 1 and 1 <= d <= K, f"node {i}: depth {d} under parent depth {pd}"
        assert t in gpu_topk_ids[d - 1].tolist(), f"node {i}: token {t} not in the position's top-k"
        assert (p, t) not in picked, f"node {i}: duplicate"
        base = 0.0 if p < 0 else oscore[p]
        cand = []
        for (n, nd, ns) in expanded:
            if nd >= K:
                continue
            for c in gpu_topk_ids[nd].tolist():
                if (n, c) not in picked:
                    cand.append((ns + logp_full[nd, c], n, c))
        best = max(c[0] for c in cand)
        mine = base + logp_full[d - 1, t]
        assert mine >= best - gap, f"node {i}: oracle score {mine:.5f} vs frontier best {best:.5f}"
        ranked = sorted(cand, key=lambda c: -c[0])
        if len(ranked) > 1 and ranked[0][0] - ranked[1][0] > gap:
            assert (ranked[0][1], ranked[0][2]) == (p, t), f"node {i}: clear best not picked"
        if score is not None:
            assert abs(float(score[i]) - mine) <= logp_tol, (
                f"node {i} (depth {d}): score {score[i]:.5f} vs oracle path score {mine:.5f}")
        oscore.append(mine)
        picked.add((p, t))
        expanded.append((i, d, mine))
    excused = 0
    if oracle_tree is not None:
        op, ot = oracle_tree
        excused = int(np.sum((np.asarray(op) != par) | (np.asarray(ot) != tok)))
    return excused
