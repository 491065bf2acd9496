"""Greedy tree verification on the GPU (domino_verify_tree_greedy) against the oracle.

Section 3.1: one target pass checks the whole draft and the draft tokens are kept up to the
first one the target rejects; at temperature 0 a draft token is kept when it equals the target's
most likely next token.  The argmax decisions are taken on the same fp32 logits on both sides, so every output
(row argmaxes, accepted nodes, their count, the bonus token) must match exactly.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2605_29707_gb300 import binding, inputs

pytestmark = pytest.mark.gpu


def _run_gpu(case):
    dev = torch.device("cuda:0")
    B, N = case.parent.shape
    V = case.target.shape[2]
    t = torch.from_numpy(case.target).to(dev)
    par = torch.from_numpy(case.parent).to(dev)
    tok = torch.from_numpy(case.token).to(dev)
    ra = torch.full((B, N + 1), -7, dtype=torch.int32, device=dev)
    nodes = torch.full((B, max(N, 1)), -7, dtype=torch.int32, device=dev)
    cnt = torch.full((B,), -7, dtype=torch.int32, device=dev)
    bon = torch.full((B,), -7, dtype=torch.int32, device=dev)
    rc = binding.domino_verify_tree_greedy(t, par if N else None, tok if N else None, B, N, V, ra,
                                           nodes if N else None, cnt, bon, torch.cuda.current_stream(dev))
    assert rc == 0, binding.domino_status_string(rc)
    torch.cuda.synchronize(dev)
    return ra.cpu().numpy(), nodes.cpu().numpy(), cnt.cpu().numpy(), bon.cpu().numpy()


def _check(case):
    ra, nodes, cnt, bon = _run_gpu(case)
    B, N = case.parent.shape
    for b in range(B):
        e_ra, e_nodes, e_bonus = oracle.verify_greedy(case.target[b], case.parent[b], case.token[b])
        np.testing.assert_array_equal(ra[b], e_ra)
        assert int(cnt[b]) == len(e_nodes), (b, cnt[b], e_nodes)
        if N:
            np.testing.assert_array_equal(nodes[b, : len(e_nodes)], e_nodes)
            assert (nodes[b, len(e_nodes):N] == -1).all()
        assert int(bon[b]) == e_bonus


@pytest.mark.parametrize("B,N,V,seed,p,chain", [
    (3, 16, 1000, 11, 0.7, False),     # V multiple of 4 (vector loads)
    (2, 20, 999, 12, 0.9, False),      # ragged V (scalar loads)
    (1, 12, 257, 13, 1.0, True),       # a chain, every row planted: all accepted
    (4, 40, 4096, 14, 0.5, False),     # more than 32 nodes (two ballot chunks)
    (2, 1, 5, 15, 1.0, False),
])
def test_verify_matches_oracle(B, N, V, seed, p, chain):
    _check(inputs.make_verify_case(B, N, V, seed, p_plant=p, chain=chain))


def test_verify_no_nodes_and_ties():
    # N = 0: only the anchor row; exact ties in it resolve to the lowest id
    t = np.zeros((2, 1, 64), np.float32)
    t[0, 0, [5, 9, 40]] = 3.0
    t[1, 0, :] = -np.inf
    case = inputs.VerifyCase(np.zeros((2, 0), np.int32), np.zeros((2, 0), np.int32), t)
    _check(case)
    # ties between a child's token and a lower non-child id: the lower id wins, so no acceptance
    c = inputs.make_verify_case(1, 6, 128, 16, p_plant=0.0)
    r = 0
    kids = [i for i in range(6) if c.parent[0, i] == -1]
    top = float(c.target[0, r].max()) + 5.0
    c.target[0, r, c.token[0, kids[0]]] = top
    lower = [v for v in range(int(c.token[0, kids[0]])) if v not in c.token[0]]
    if lower:
        c.target[0, r, lower[0]] = top
    _check(c)


def test_verify_on_trees_of_the_oracle_draft_step():
    """Trees built by the oracle's draft step on the tiny configuration, synthetic target logits."""
    wl = inputs.make_workload("tiny")
    c = wl.cfg
    ref = oracle.draft_step(wl.weights, wl.hidden, wl.prefix_ids, c.k, c.N)
    trees = [(ref["tree_parent"][b], ref["tree_token"][b]) for b in range(c.B)]
    _check(inputs.make_verify_case(c.B, c.N, c.V, 17, p_plant=0.8, trees=trees))


@pytest.mark.parametrize("B,N", [(2, 16), (1, 32)])
def test_verify_full_vocabulary(B, N):
    _check(inputs.make_verify_case(B, N, 151936, 18 + N, p_plant=0.8))
