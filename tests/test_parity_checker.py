"""The gap-aware parity checker (tests/parity.py) on the CPU: the oracle's own outputs pass with
nothing excused, every kind of planted mistake fails, and a swap across a near-tie is excused and
counted -- so the GPU parity tests can fail for the reasons they are meant to."""
import numpy as np
import pytest

import oracle
from tests.parity import GAP, LOGP_TOL, check_topk, check_tree

K, V, k, N = 4, 60, 4, 10


def _logp(rng, ties_at=None):
    """log-softmax rows whose k + 1 best values are more than 0.1 apart; with ties_at = (row, q),
    ranks q and q + 1 of that row are 0.01 apart."""
    z = rng.normal(0.0, 0.3, size=(K, V))
    for r in range(K):
        top = rng.choice(V, size=k + 1, replace=False)
        z[r, top] = 5.0 - 0.5 * np.arange(k + 1)
    if ties_at is not None:
        r, q = ties_at
        top = np.argsort(-z[r], kind="stable")[: k + 1]
        z[r, top[q + 1]] = z[r, top[q]] - 0.01
    lp, _ = oracle.log_softmax(z)
    return lp


def _reference(lp):
    ids, vals = oracle.topk(lp, k)
    par, tok, dep, sc = oracle.tree(ids, vals, N)
    return ids, vals, (par, tok, dep, sc)


def test_the_oracles_own_outputs_pass():
    lp = _logp(np.random.default_rng(1))
    ids, vals, (par, tok, dep, sc) = _reference(lp)
    assert check_topk(ids, vals, lp, k) == 0
    assert check_tree(par, tok, dep, sc, ids, lp, K, N, oracle_tree=(par, tok)) == 0


def test_topk_mistakes_fail():
    lp = _logp(np.random.default_rng(2))
    ids, vals, _ = _reference(lp)
    bad = ids.copy()
    bad[1, [0, 1]] = bad[1, [1, 0]]  # ranks 0 and 1 swapped across a 0.5 gap
    with pytest.raises(AssertionError):
        check_topk(bad, vals, lp, k)
    off = vals.copy()
    off[2, 3] += 2.5 * LOGP_TOL  # a log-prob outside the tolerance
    with pytest.raises(AssertionError):
        check_topk(ids, off, lp, k)
    dup = ids.copy()
    dup[0, 2] = dup[0, 1]  # a duplicate id
    with pytest.raises(AssertionError):
        check_topk(dup, vals, lp, k)


def test_near_tie_swap_is_excused_and_counted():
    """Ranks 1 and 2 of one row 0.01 apart: the swapped order passes, each differing rank counted."""
    lp = _logp(np.random.default_rng(3), ties_at=(2, 1))
    ids, vals, _ = _reference(lp)
    assert abs(vals[2, 1] - vals[2, 2]) < GAP
    swapped = ids.copy()
    swapped[2, [1, 2]] = swapped[2, [2, 1]]
    swapped_vals = vals.copy()
    swapped_vals[2, [1, 2]] = vals[2, [2, 1]]
    assert check_topk(swapped, swapped_vals, lp, k) == 2  # ranks 1 and 2 each differ, both excused


def test_tree_mistakes_fail():
    lp = _logp(np.random.default_rng(4))
    ids, vals, (par, tok, dep, sc) = _reference(lp)
    # a token that is not in its position's top-k list
    t = tok.copy()
    t[0] = next(v for v in range(V) if v not in ids[0].tolist())
    with pytest.raises(AssertionError):
        check_tree(par, t, dep, sc, ids, lp, K, N)
    # the first pick replaced by a worse depth-1 candidate across a clear gap
    t = tok.copy()
    t[0] = ids[0, k - 1]
    with pytest.raises(AssertionError):
        check_tree(par, t, dep, sc, ids, lp, K, N)
    # a parent that is not an earlier node
    p = par.copy()
    p[1] = 1
    with pytest.raises(AssertionError):
        check_tree(p, tok, dep, sc, ids, lp, K, N)
    # a cumulative score off by more than the tolerance, at the deepest node: the bound does not
    # grow with depth
    s = sc.copy()
    deep = int(np.argmax(dep))
    assert dep[deep] >= 2
    s[deep] += 1.5 * LOGP_TOL
    with pytest.raises(AssertionError):
        check_tree(par, tok, dep, s, ids, lp, K, N)
    s = sc.copy()
    s[deep] += 0.5 * LOGP_TOL
    check_tree(par, tok, dep, s, ids, lp, K, N)
