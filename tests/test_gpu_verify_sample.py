"""Tree verification at temperature T > 0 on the GPU (domino_verify_tree_sample) against the oracle.

Section 3.1: the target keeps draft tokens by the speculative sampling rule; for a tree of fixed
children that is one draw from the target's softmax(logits / T) per visited node, kept when a
child carries it (oracle_verify_sample states the reading).

A draw is an integer decided by floating point: the GPU sums in fp32, the oracle in fp64, so
where the uniform lies within rounding of a boundary of the cumulative distribution both
neighbours are correct.  Bound: the GPU's normalised cumulative sum at any id differs from the
exact one by at most about (75 + 8 + 8 + 3) fp32 roundings of the total (a thread's run of at
most 75 terms at 151936 ids, the thread scan, the eight slices, u Z) plus the exp and argument
roundings of the terms (relative 2 ulp, and 1.2e-7 |x - max| / T for the few terms that carry
mass): under 1e-5 of the total; the tests allow EPS = 2e-5.  So a GPU draw y is accepted when it
equals the oracle's, or when y lies between the oracle's draws at u - EPS and u + EPS (the draw
is monotone in u) and has non-zero probability.  The walk is integer logic: it must equal the
oracle's walk on the GPU's draws exactly, and the oracle's own walk whenever every draw agrees.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2605_29707_gb300 import binding, inputs

pytestmark = pytest.mark.gpu

EPS = 2e-5
BELOW_ONE = float(np.nextafter(np.float32(1.0), np.float32(0.0)))


def _run_gpu(case, u, T):
    dev = torch.device("cuda:0")
    B, N = case.parent.shape
    V = case.target.shape[2]
    t = torch.from_numpy(case.target).to(dev)
    par = torch.from_numpy(case.parent).to(dev)
    tok = torch.from_numpy(case.token).to(dev)
    uu = torch.from_numpy(np.ascontiguousarray(u, np.float32)).to(dev)
    rs = torch.full((B, N + 1), -7, dtype=torch.int32, device=dev)
    nodes = torch.full((B, max(N, 1)), -7, dtype=torch.int32, device=dev)
    cnt = torch.full((B,), -7, dtype=torch.int32, device=dev)
    bon = torch.full((B,), -7, dtype=torch.int32, device=dev)
    rc = binding.domino_verify_tree_sample(t, par if N else None, tok if N else None, uu, T, B, N, V, rs,
                                           nodes if N else None, cnt, bon, torch.cuda.current_stream(dev))
    assert rc == 0, binding.domino_status_string(rc)
    torch.cuda.synchronize(dev)
    return rs.cpu().numpy(), nodes.cpu().numpy(), cnt.cpu().numpy(), bon.cpu().numpy()


def _clamp(u):
    u = float(u)
    if not (u >= 0.0):
        return 0.0
    return min(u, BELOW_ONE)


def _check(case, u, T):
    """Returns the number of rows whose draw differs from the oracle's (each within EPS)."""
    rs, nodes, cnt, bon = _run_gpu(case, u, T)
    B, N = case.parent.shape
    differ = 0
    for b in range(B):
        uc = np.array([_clamp(x) for x in u[b]], np.float32)
        e_rs, e_nodes, e_bonus = oracle.verify_sample(case.target[b], case.parent[b], case.token[b], T, uc)
        same = True
        for r in range(N + 1):
            y = int(rs[b, r])
            if y == int(e_rs[r]):
                continue
            same = False
            differ += 1
            row = case.target[b, r]
            lo = oracle.row_sample(row, T, max(0.0, float(uc[r]) - EPS))
            hi = oracle.row_sample(row, T, min(BELOW_ONE, float(uc[r]) + EPS))
            assert lo <= y <= hi and np.isfinite(row[y]), (b, r, y, int(e_rs[r]), lo, hi)
        w_nodes, w_bonus = oracle.tree_walk(case.parent[b], case.token[b], rs[b])
        assert int(cnt[b]) == len(w_nodes), (b, cnt[b], w_nodes)
        if N:
            np.testing.assert_array_equal(nodes[b, : len(w_nodes)], w_nodes)
            assert (nodes[b, len(w_nodes):N] == -1).all()
        assert int(bon[b]) == w_bonus
        if same:
            assert w_nodes.tolist() == e_nodes.tolist() and w_bonus == e_bonus
    return differ


def _uniforms(B, N, seed):
    return inputs.uniform01(B * (N + 1), (seed, "verify-sample-u")).astype(np.float32).reshape(B, N + 1)


@pytest.mark.parametrize("B,N,V,seed,T,margin,chain", [
    (3, 16, 1000, 31, 1.0, 6.0, False),    # V multiple of 4 (vector loads)
    (2, 20, 999, 32, 0.7, 5.0, False),     # ragged V (scalar loads), T < 1
    (1, 12, 257, 33, 1.5, 8.0, True),      # a chain, T > 1
    (4, 40, 4096, 34, 1.0, 7.0, False),    # more than 32 nodes
    (2, 1, 5, 35, 1.0, 1.0, False),        # V smaller than the cluster: empty slices
    (2, 3, 37, 36, 20.0, 1.0, False),      # a very flat distribution
    (2, 6, 300, 37, 0.05, 0.5, False),     # a very sharp one
])
def test_verify_sample_matches_oracle(B, N, V, seed, T, margin, chain):
    c = inputs.make_verify_case(B, N, V, seed, p_plant=0.9, chain=chain, margin=margin)
    differ = _check(c, _uniforms(B, N, seed), T)
    assert differ <= max(1, B * (N + 1) // 10)


@pytest.mark.parametrize("B,N,T", [(2, 16, 1.0), (1, 32, 0.6)])
def test_verify_sample_full_vocabulary(B, N, T):
    """The 8B-shaped target vocabulary (151936 ids: eight slices of 18992), planted tokens with
    about two thirds of the mass at T = 1, so that accepted paths of several lengths occur."""
    c = inputs.make_verify_case(B, N, 151936, 40 + N, p_plant=0.9, margin=9.0)
    _check(c, _uniforms(B, N, 40 + N), T)


def test_verify_sample_interval_ends_masks_and_clamping():
    """u = 0 and u just below 1 give the first and last ids of non-zero probability; -inf logits
    are never drawn; a row of -inf only gives id 0; uniforms outside [0, 1) (and NaN) are clamped."""
    V, N = 1000, 5
    c = inputs.make_verify_case(1, N, V, 41, p_plant=0.5, margin=3.0)
    t = c.target.copy()
    t[0, 0, :7] = -np.inf
    t[0, 0, 990:] = -np.inf
    t[0, 1, ::2] = -np.inf
    t[0, 2, :] = -np.inf
    c = inputs.VerifyCase(c.parent, c.token, t)
    u = np.array([[0.0, BELOW_ONE, 0.3, -0.5, 1.5, np.nan]], np.float32)
    rs, _, _, _ = _run_gpu(c, u, 1.0)
    assert rs[0, 0] == 7 and rs[0, 2] == 0
    assert rs[0, 1] % 2 == 1
    _check(c, u, 1.0)
    rs2, _, _, _ = _run_gpu(c, np.array([[0.0, BELOW_ONE, 0.3, 0.0, BELOW_ONE, 0.0]], np.float32), 1.0)
    np.testing.assert_array_equal(rs, rs2)


def test_verify_sample_at_low_temperature_is_the_greedy_verification():
    """Every row's maximum at least 1 above the rest and T = 0.01: all but e^-100 of the mass is on
    the argmax, so the GPU's draws and walk equal its greedy verification's."""
    B, N, V = 3, 16, 4096
    c = inputs.make_verify_case(B, N, V, 42, p_plant=0.8)
    t = c.target.copy()
    for b in range(B):
        for r in range(N + 1):
            a = int(np.argmax(t[b, r]))
            t[b, r, a] = np.float32(np.max(np.delete(t[b, r], a)) + 1.0)
    c = inputs.VerifyCase(c.parent, c.token, t)
    u = _uniforms(B, N, 42) * np.float32(0.999)
    rs, nodes, cnt, bon = _run_gpu(c, u, 0.01)
    dev = torch.device("cuda:0")
    ra = torch.empty((B, N + 1), dtype=torch.int32, device=dev)
    gn = torch.empty((B, N), dtype=torch.int32, device=dev)
    gc = torch.empty((B,), dtype=torch.int32, device=dev)
    gb = torch.empty((B,), dtype=torch.int32, device=dev)
    tt = torch.from_numpy(t).to(dev)
    rc = binding.domino_verify_tree_greedy(tt, torch.from_numpy(c.parent).to(dev), torch.from_numpy(c.token).to(dev),
                                           B, N, V, ra, gn, gc, gb, torch.cuda.current_stream(dev))
    assert rc == 0
    torch.cuda.synchronize(dev)
    np.testing.assert_array_equal(rs, ra.cpu().numpy())
    np.testing.assert_array_equal(cnt, gc.cpu().numpy())
    np.testing.assert_array_equal(bon, gb.cpu().numpy())
    np.testing.assert_array_equal(nodes, gn.cpu().numpy())
    _check(c, u, 0.01)


def test_verify_sample_no_nodes():
    t = np.zeros((2, 1, 64), np.float32)
    t[1, 0, :] = -np.inf
    case = inputs.VerifyCase(np.zeros((2, 0), np.int32), np.zeros((2, 0), np.int32), t)
    u = np.array([[0.51], [0.2]], np.float32)
    rs, _, cnt, bon = _run_gpu(case, u, 1.0)
    assert rs[0, 0] == 32 and rs[1, 0] == 0
    assert cnt.tolist() == [0, 0] and bon.tolist() == [32, 0]
