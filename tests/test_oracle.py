"""Pins for the fp64 CPU oracle (CPU only).

Each test ties one oracle step to something other than the oracle itself: a
hand-worked example from tests/golden/, a library routine that computes a special
case (torch.nn.GRU, scipy's log-softmax, a stable library sort), brute-force
enumeration, an invariant the method guarantees, or the parameter count the paper
states.
"""
import itertools
import json
import math
import os

import numpy as np
import pytest
import torch

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def bf16(x):
    """float values that are exact in bf16 -> uint16 bit patterns (truncation is exact here)."""
    a = np.asarray(x, dtype=np.float32)
    bits = a.view(np.uint32)
    assert np.all((bits & 0xFFFF) == 0), "value not exactly representable in bf16"
    return (bits >> 16).astype(np.uint16)


def rand_bf16(rng, shape, std):
    x = torch.from_numpy(rng.standard_normal(shape).astype(np.float32) * std)
    return x.to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)


def to_f64(b):
    return (np.asarray(b, np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def _ev(expr):
    return eval(expr, {"__builtins__": {}}, {"log": math.log, "exp": math.exp})


def load(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


# ----------------------------------------------------------------------------- hand cases

def test_bf16_widening_exact():
    assert oracle.bf16_to_double(0x3F80) == 1.0
    assert oracle.bf16_to_double(0xC000) == -2.0
    assert oracle.bf16_to_double(0x3F00) == 0.5
    assert oracle.bf16_to_double(0x3C23) == float(np.float32(np.uint32(0x3C230000).view(np.float32)))


@pytest.mark.parametrize("name", ["hand_case_a.json", "hand_case_b.json"])
def test_hand_cases_head_off(name):
    g = load(name)
    V, H, K, k, N = g["V"], g["H"], g["K"], g["k"], g["N"]
    w = {"w_lm": bf16(g["w_lm"])}
    hidden = bf16(g["hidden"]).reshape(1, K, H)
    ids = np.asarray(g["prefix_ids"], np.int32).reshape(1, K)
    out = oracle.draft_step(w, hidden, ids, k, N, want_logp_full=True)
    assert out["topk_ids"][0].tolist() == g["expect_topk_ids"]
    assert out["tree_parent"][0].tolist() == g["expect_tree_parent"]
    assert out["tree_token"][0].tolist() == g["expect_tree_token"]
    assert out["tree_depth"][0].tolist() == g["expect_tree_depth"]
    for i, e in enumerate(g["expect_tree_score"]):
        assert out["tree_score"][0, i] == pytest.approx(_ev(e), abs=1e-12)
    if "expect_lse" in g:
        for j, e in enumerate(g["expect_lse"]):
            assert out["lse"][0, j] == pytest.approx(_ev(e), abs=1e-12)
    if "expect_logp" in g:
        for j in range(K):
            for v in range(V):
                assert out["logp_full"][0, j, v] == pytest.approx(_ev(g["expect_logp"][j][v]), abs=1e-12)


def test_hand_case_c_head_on():
    g = load("hand_case_c.json")
    K, k, N, tol = g["K"], g["k"], g["N"], g["tolerance"]
    w = {n: bf16(g[n]) for n in ("w_lm", "emb", "w_ih", "w_hh", "b_ih", "b_hh", "w1", "b1", "w2", "b2")}
    hidden = bf16(g["hidden"]).reshape(1, K, g["H"])
    ids = np.asarray(g["prefix_ids"], np.int32).reshape(1, K)
    # step by step
    E = oracle.embed(w["emb"], ids[0])
    assert E.tolist() == [[1.0, 0.0], [0.0, 1.0]]
    S = oracle.gru(E, w["w_ih"], w["w_hh"], w["b_ih"], w["b_hh"])
    assert S[:, 0] == pytest.approx(g["expect_S"], abs=tol)
    u = oracle.lowrank(to_f64(hidden[0]), S, w["w1"], w["b1"])
    assert u[:, 0] == pytest.approx(g["expect_u"], abs=tol)
    # whole step
    out = oracle.draft_step(w, hidden, ids, k, N, want_logp_full=True)
    assert out["logp_full"][0] == pytest.approx(np.asarray(g["expect_logp"]), abs=tol)
    assert out["topk_ids"][0].tolist() == g["expect_topk_ids"]
    assert out["tree_parent"][0].tolist() == g["expect_tree_parent"]
    assert out["tree_token"][0].tolist() == g["expect_tree_token"]
    assert out["tree_depth"][0].tolist() == g["expect_tree_depth"]
    assert out["tree_score"][0] == pytest.approx(g["expect_tree_score"], abs=tol)


# ----------------------------------------------------------------------------- GRU

@pytest.mark.parametrize("Hin,Ds,K", [(12, 8, 5), (40, 24, 7), (8, 1, 3)])
def test_gru_matches_torch_nn_gru_fp64(Hin, Ds, K):
    """torch.nn.GRU (a library GRU) in float64 is the reference for the recurrence."""
    rng = np.random.default_rng(Hin * 100 + Ds)
    w_ih = rand_bf16(rng, (3 * Ds, Hin), 0.3)
    w_hh = rand_bf16(rng, (3 * Ds, Ds), 0.3)
    b_ih = rand_bf16(rng, (3 * Ds,), 0.3)
    b_hh = rand_bf16(rng, (3 * Ds,), 0.3)
    E = rng.standard_normal((K, Hin))
    S = oracle.gru(E, w_ih, w_hh, b_ih, b_hh)
    gru = torch.nn.GRU(Hin, Ds, bias=True).double()
    with torch.no_grad():
        gru.weight_ih_l0.copy_(torch.from_numpy(to_f64(w_ih)))
        gru.weight_hh_l0.copy_(torch.from_numpy(to_f64(w_hh)))
        gru.bias_ih_l0.copy_(torch.from_numpy(to_f64(b_ih)))
        gru.bias_hh_l0.copy_(torch.from_numpy(to_f64(b_hh)))
        ref, _ = gru(torch.from_numpy(E).unsqueeze(1))
    np.testing.assert_allclose(S, ref[:, 0].numpy(), atol=1e-12, rtol=0)
    # and without biases (NULL means zero)
    S0 = oracle.gru(E, w_ih, w_hh)
    with torch.no_grad():
        gru.bias_ih_l0.zero_(); gru.bias_hh_l0.zero_()
        ref0, _ = gru(torch.from_numpy(E).unsqueeze(1))
    np.testing.assert_allclose(S0, ref0[:, 0].numpy(), atol=1e-12, rtol=0)


# ----------------------------------------------------------------------------- softmax / top-k

def test_log_softmax_matches_scipy_and_normalises():
    from scipy.special import log_softmax as sp_lsm
    rng = np.random.default_rng(1)
    z = rng.standard_normal((6, 1000)) * 5
    lp, lse = oracle.log_softmax(z)
    np.testing.assert_allclose(lp, sp_lsm(z, axis=1), atol=1e-12, rtol=0)
    np.testing.assert_allclose(np.exp(lp).sum(1), 1.0, atol=1e-12)
    assert np.all(lp <= 0)
    # shift invariance and the uniform special case
    lp2, _ = oracle.log_softmax(z + 123.25)
    np.testing.assert_allclose(lp2, lp, atol=1e-10)
    lpu, lseu = oracle.log_softmax(np.zeros((2, 77)))
    np.testing.assert_allclose(lpu, -math.log(77), atol=1e-14)
    np.testing.assert_allclose(lseu, math.log(77), atol=1e-14)


def test_topk_matches_stable_library_sort_with_ties():
    rng = np.random.default_rng(2)
    lp = np.round(rng.standard_normal((10, 300)) * 2) / 4  # coarse grid -> many exact ties
    for k in (1, 5, 17, 300):
        ids, vals = oracle.topk(lp, k)
        for i in range(lp.shape[0]):
            order = np.lexsort((np.arange(300), -lp[i]))  # value desc, then id asc
            assert ids[i].tolist() == order[:k].tolist()
            assert vals[i].tolist() == lp[i, order[:k]].tolist()


# ----------------------------------------------------------------------------- tree

def _random_lists(rng, K, k, V=50, ties=False):
    ids = np.stack([rng.choice(V, size=k, replace=False) for _ in range(K)]).astype(np.int32)
    lp = -np.sort(rng.exponential(1.0, size=(K, k)), axis=1)
    if ties:
        lp = np.round(lp * 4) / 4
        # keep each list ordered by (value desc, id asc)
        for j in range(K):
            o = np.lexsort((ids[j], -lp[j]))
            ids[j], lp[j] = ids[j][o], lp[j][o]
    return ids, lp


def _paths(K, k):
    for d in range(1, K + 1):
        yield from itertools.product(range(k), repeat=d)


def _node_path(par, tok, dep, i, ids):
    path = []
    while i >= 0:
        d = dep[i]
        path.append(int(np.where(ids[d - 1] == tok[i])[0][0]))
        i = par[i]
    return tuple(reversed(path))


@pytest.mark.parametrize("K,k", [(3, 3), (2, 4), (4, 2), (1, 5)])
def test_tree_matches_brute_force_enumeration(K, k):
    rng = np.random.default_rng(K * 10 + k)
    ids, lp = _random_lists(rng, K, k)
    allp = list(_paths(K, k))
    scores = {p: sum(lp[d, c] for d, c in enumerate(p)) for p in allp}
    ranked = sorted(allp, key=lambda p: -scores[p])
    for N in range(1, len(allp) + 1):
        par, tok, dep, sc = oracle.tree(ids, lp, N)
        got = {_node_path(par, tok, dep, i, ids) for i in range(N)}
        assert got == set(ranked[:N])
        np.testing.assert_allclose(sc, sorted((scores[p] for p in ranked[:N]), reverse=True),
                                   atol=1e-12)


@pytest.mark.parametrize("ties", [False, True])
def test_tree_invariants(ties):
    rng = np.random.default_rng(7 + ties)
    K, k, N = 5, 4, 40
    ids, lp = _random_lists(rng, K, k, ties=ties)
    par, tok, dep, sc = oracle.tree(ids, lp, N)
    for i in range(N):
        assert par[i] < i
        d = dep[i]
        assert 1 <= d <= K
        q = int(np.where(ids[d - 1] == tok[i])[0][0])
        base = 0.0 if par[i] < 0 else sc[par[i]]
        assert (d == 1) == (par[i] < 0)
        if par[i] >= 0:
            assert dep[par[i]] == d - 1
        assert sc[i] == base + lp[d - 1, q]  # cumulative score = parent's + own log-prob
        if i:
            assert sc[i] <= sc[i - 1]
    # no node appears twice
    assert len({(par[i], tok[i]) for i in range(N)}) == N


def _tree_by_frontier_scan(ids, lp, N):
    """The best-first tree by its definition, slowly: before every pop the frontier is rebuilt
    from scratch (every depth-1 candidate and every child of a selected node that is not selected
    yet), and the pop is the greatest (score, lower token, lower parent index)."""
    K, k = lp.shape
    nodes = []  # (parent, token, depth, score, list index)
    taken = set()  # (parent, list index)
    for _ in range(N):
        best = None
        for parent in [-1] + list(range(len(nodes))):
            d = 1 if parent < 0 else nodes[parent][2] + 1
            if d > K:
                continue
            base = 0.0 if parent < 0 else nodes[parent][3]
            for q in range(k):
                if (parent, q) in taken:
                    continue
                key = (base + lp[d - 1, q], -int(ids[d - 1, q]), -parent)
                if best is None or key > best[0]:
                    best = (key, parent, q, d)
        (score, _, _), parent, q, d = best
        taken.add((parent, q))
        nodes.append((parent, int(ids[d - 1, q]), d, score, q))
    return (np.array([n[0] for n in nodes]), np.array([n[1] for n in nodes]), np.array([n[2] for n in nodes]),
            np.array([n[3] for n in nodes]))


@pytest.mark.parametrize("seed", range(6))
def test_tree_with_ties_matches_a_frontier_scan(seed):
    """Tie-heavy lists (log-probs on a 1/4 grid, so equal scores are common at every depth):
    the oracle's tree equals the definition computed by rescanning the whole frontier."""
    rng = np.random.default_rng(100 + seed)
    K, k = [(3, 3), (4, 2), (2, 4), (5, 3), (3, 4), (6, 2)][seed]
    ids, lp = _random_lists(rng, K, k, ties=True)
    total = sum(k ** d for d in range(1, K + 1))
    for N in sorted({1, 2, 3, min(total, 12), min(total, 31), total}):
        par, tok, dep, sc = oracle.tree(ids, lp, N)
        rpar, rtok, rdep, rsc = _tree_by_frontier_scan(ids, lp, N)
        assert par.tolist() == rpar.tolist() and tok.tolist() == rtok.tolist() and dep.tolist() == rdep.tolist()
        np.testing.assert_array_equal(sc, rsc)


def test_tree_special_cases():
    rng = np.random.default_rng(11)
    K, k = 6, 4
    ids, lp = _random_lists(rng, K, k)
    # k = 1, N = K: the chain of per-position argmaxes
    par, tok, dep, sc = oracle.tree(ids[:, :1], lp[:, :1], K)
    assert tok.tolist() == ids[:, 0].tolist()
    assert par.tolist() == [-1] + list(range(K - 1))
    np.testing.assert_allclose(sc, np.cumsum(lp[:, 0]), atol=1e-12)
    # K = 1: the top-N of position 0
    par, tok, dep, sc = oracle.tree(ids[:1], lp[:1], 3)
    assert tok.tolist() == ids[0, :3].tolist() and par.tolist() == [-1, -1, -1]
    # N = 1: the argmax of position 0
    par, tok, dep, sc = oracle.tree(ids, lp, 1)
    assert tok.tolist() == [ids[0, 0]] and sc.tolist() == [lp[0, 0]]
    # N above the size of the tree is rejected
    with pytest.raises(oracle.OracleError):
        oracle.tree(ids[:2, :2], lp[:2, :2], 7)


# ----------------------------------------------------------------------------- whole step

def _small_workload(rng, B=2, K=5, H=24, V=64, Ds=16, R=8, biases=True):
    w = {
        "w_lm": rand_bf16(rng, (V, H), 0.3), "emb": rand_bf16(rng, (V, H), 0.5),
        "w_ih": rand_bf16(rng, (3 * Ds, H), 0.3), "w_hh": rand_bf16(rng, (3 * Ds, Ds), 0.3),
        "w1": rand_bf16(rng, (R, H + Ds), 0.3), "w2": rand_bf16(rng, (V, R), 0.5),
        "b_ih": None, "b_hh": None, "b1": None, "b2": None,
    }
    if biases:
        w["b_ih"] = rand_bf16(rng, (3 * Ds,), 0.2)
        w["b_hh"] = rand_bf16(rng, (3 * Ds,), 0.2)
        w["b1"] = rand_bf16(rng, (R,), 0.2)
        w["b2"] = rand_bf16(rng, (V,), 0.2)
    hidden = rand_bf16(rng, (B, K, H), 1.0)
    ids = rng.integers(0, V, size=(B, K)).astype(np.int32)
    return w, hidden, ids


def test_causality_position_j_sees_ids_0_to_j_only():
    """Section 4.1.2: S_{i-1} summarises the tokens before position i (anchor first)."""
    rng = np.random.default_rng(3)
    w, hidden, ids = _small_workload(rng, B=1)
    K = ids.shape[1]
    base = oracle.draft_step(w, hidden, ids, 4, 6, want_logp_full=True)["logp_full"][0]
    for jp in range(K):
        ids2 = ids.copy()
        ids2[0, jp] = (ids2[0, jp] + 17) % w["w_lm"].shape[0]
        lp = oracle.draft_step(w, hidden, ids2, 4, 6, want_logp_full=True)["logp_full"][0]
        assert np.array_equal(lp[:jp], base[:jp])           # earlier positions untouched
        assert np.abs(lp[jp] - base[jp]).max() > 1e-6        # position jp sees id jp
        if jp + 1 < K:
            assert np.abs(lp[jp + 1:] - base[jp + 1:]).max() > 1e-6


def test_correction_off_gives_base_distribution():
    """Table 4 'w/o Domino head': with W2 = 0 the refined distribution is the base one."""
    rng = np.random.default_rng(4)
    w, hidden, ids = _small_workload(rng)
    w_off = dict(w, w2=np.zeros_like(w["w2"]))
    on0 = oracle.draft_step(w_off, hidden, ids, 4, 6, want_logp_full=True)
    off = oracle.draft_step(dict(w, w2=None), hidden, ids, 4, 6, want_logp_full=True)
    np.testing.assert_array_equal(on0["logp_full"], off["logp_full"])
    # base logits: hidden . W_lm^T + b2 (library matmul as the special-case reference)
    from scipy.special import log_softmax as sp_lsm
    z = to_f64(hidden).reshape(-1, hidden.shape[-1]) @ to_f64(w["w_lm"]).T + to_f64(w["b2"])
    np.testing.assert_allclose(off["logp_full"].reshape(z.shape), sp_lsm(z, axis=1), atol=1e-12)


def test_uniform_bias_shift_leaves_distribution_unchanged():
    rng = np.random.default_rng(5)
    w, hidden, ids = _small_workload(rng, biases=False)
    a = oracle.draft_step(w, hidden, ids, 4, 6, want_logp_full=True)
    b2 = np.full(w["w_lm"].shape[0], bf16([2.5])[0], np.uint16)
    b = oracle.draft_step(dict(w, b2=b2), hidden, ids, 4, 6, want_logp_full=True)
    np.testing.assert_allclose(a["logp_full"], b["logp_full"], atol=1e-12)
    assert a["topk_ids"].tolist() == b["topk_ids"].tolist()


def test_step_equals_composition_and_sequence_selection():
    rng = np.random.default_rng(6)
    w, hidden, ids = _small_workload(rng, B=3)
    k, N = 4, 9
    full = oracle.draft_step(w, hidden, ids, k, N, want_logp_full=True)
    sel = oracle.draft_step(w, hidden, ids, k, N, seqs=[2, 0], want_logp_full=True)
    for si, b in enumerate([2, 0]):
        for key in ("logp_full", "topk_ids", "topk_logp", "tree_parent", "tree_token", "tree_score"):
            np.testing.assert_array_equal(sel[key][si], full[key][b])
    b = 1
    E = oracle.embed(w["emb"], ids[b])
    S = oracle.gru(E, w["w_ih"], w["w_hh"], w["b_ih"], w["b_hh"])
    u = oracle.lowrank(to_f64(hidden[b]), S, w["w1"], w["b1"])
    z = oracle.logits(to_f64(hidden[b]), u, w["w_lm"], w["w2"], w["b2"])
    lp, lse = oracle.log_softmax(z)
    np.testing.assert_array_equal(lp, full["logp_full"][b])
    tid, tlp = oracle.topk(lp, k)
    np.testing.assert_array_equal(tid, full["topk_ids"][b])
    par, tok, dep, sc = oracle.tree(tid, tlp, N)
    np.testing.assert_array_equal(tok, full["tree_token"][b])


def test_lowrank_concat_order_hidden_then_state():
    """W1 acts on [H_i; S_{i-1}]: the first H columns see hidden, the rest the state."""
    H, Ds = 3, 2
    hidden = np.array([[1.0, 2.0, 3.0]])
    S = np.array([[10.0, 20.0]])
    w1 = bf16([[1, 0, 0, 0, 0], [0, 0, 0, 1, 0], [0, 0, 0, 0, 0.5]])
    u = oracle.lowrank(hidden, S, w1)
    silu = lambda x: x / (1 + math.exp(-x))
    assert u[0].tolist() == pytest.approx([silu(1.0), silu(10.0), silu(10.0)], abs=1e-14)


def test_bad_token_and_bad_args():
    rng = np.random.default_rng(8)
    w, hidden, ids = _small_workload(rng, B=1)
    bad = ids.copy(); bad[0, 2] = w["w_lm"].shape[0]
    with pytest.raises(oracle.OracleError) as e:
        oracle.draft_step(w, hidden, bad, 4, 6)
    assert e.value.rc == oracle.ERR_TOKEN
    bad[0, 2] = -1
    with pytest.raises(oracle.OracleError):
        oracle.draft_step(w, hidden, bad, 4, 6)
    with pytest.raises(oracle.OracleError):
        oracle.draft_step(w, hidden, ids, 0, 6)


def test_parameter_count_matches_paper_56M():
    """The head adds 'only 56M parameters' for Qwen3-8B (d_s = 1024, r = 256, H = 4096,
    V = 151936).  The shapes the oracle takes must add up to that figure."""
    H, V, Ds, R = 4096, 151936, 1024, 256
    gru = 3 * Ds * H + 3 * Ds * Ds + 2 * 3 * Ds   # w_ih, w_hh, b_ih, b_hh
    w1 = R * (H + Ds)                              # W1 over [H_i; S_{i-1}]
    w2 = V * R                                     # W2 to the full vocabulary
    total = gru + w1 + w2
    assert total == 55_941_120
    assert round(total / 1e6) == 56
    # the oracle accepts exactly these shapes (tiny V to keep it fast)
    rng = np.random.default_rng(9)
    Vs = 8
    w = {"w_lm": rand_bf16(rng, (Vs, H), 0.02), "emb": rand_bf16(rng, (Vs, H), 0.02),
         "w_ih": rand_bf16(rng, (3 * Ds, H), 0.02), "w_hh": rand_bf16(rng, (3 * Ds, Ds), 0.02),
         "b_ih": None, "b_hh": None, "w1": rand_bf16(rng, (R, H + Ds), 0.02), "b1": None,
         "w2": rand_bf16(rng, (Vs, R), 0.02), "b2": None}
    hidden = rand_bf16(rng, (1, 2, H), 1.0)
    out = oracle.draft_step(w, hidden, np.array([[1, 2]], np.int32), 2, 3)
    assert out["topk_ids"].shape == (1, 2, 2)


# ---------------------------------------------------------------------------- O8 tree verification
def _golden(name):
    with open(os.path.join(os.path.dirname(__file__), "golden", name)) as f:
        return json.load(f)


def test_verify_hand_case_a():
    """Hand-worked greedy verification (section 3.1): tie at the anchor, a negative row, a leaf stop."""
    g = _golden("verify_case_a.json")
    ra, nodes, bonus = oracle.verify_greedy(np.array(g["target"], np.float32), g["parent"], g["token"])
    assert ra.tolist() == g["expect_row_argmax"]
    assert nodes.tolist() == g["expect_nodes"]
    assert bonus == g["expect_bonus"]
    assert len(nodes) + 1 == g["expect_tau"]


def _brute_force_accepted(target, parent, token):
    """Every path from the anchor whose tokens all equal numpy's argmax (first occurrence) of the
    parent's row; the accepted path is the longest such path (each step has one candidate)."""
    N = len(parent)
    am = np.argmax(target, axis=1)
    best = []
    for end in range(N):
        path, c = [], end
        while c != -1:
            path.append(c)
            c = int(parent[c])
        path.reverse()
        ok = all(token[n] == am[(parent[n] + 1)] for n in path)
        if ok and len(path) > len(best):
            best = path
    last = best[-1] if best else -1
    return am, best, int(am[last + 1])


@pytest.mark.parametrize("seed,N,V,chain,p", [(1, 12, 300, False, 0.7), (2, 20, 50, False, 0.9),
                                               (3, 16, 1000, True, 0.8), (4, 1, 7, False, 1.0),
                                               (5, 30, 64, False, 0.5)])
def test_verify_matches_brute_force(seed, N, V, chain, p):
    from paper_2605_29707_gb300 import inputs
    c = inputs.make_verify_case(2, N, V, seed, p_plant=p, chain=chain)
    for b in range(2):
        ra, nodes, bonus = oracle.verify_greedy(c.target[b], c.parent[b], c.token[b])
        am, best, bb = _brute_force_accepted(c.target[b], c.parent[b], c.token[b])
        assert ra.tolist() == am.tolist()
        assert nodes.tolist() == best
        assert bonus == bb
        # stop rule: no child of the last accepted node carries the bonus token
        last = nodes[-1] if len(nodes) else -1
        assert not any(c.parent[b, i] == last and c.token[b, i] == bonus for i in range(N))


def test_verify_special_cases():
    # no nodes: tau = 1, bonus = argmax after the anchor
    t = np.array([[0.0, 3.0, 3.0, -1.0]], np.float32)
    ra, nodes, bonus = oracle.verify_greedy(t, np.zeros(0, np.int32), np.zeros(0, np.int32))
    assert ra.tolist() == [1] and len(nodes) == 0 and bonus == 1
    # a chain whose every row points at the next token: all N accepted, tau = N + 1
    N, V = 6, 10
    parent = np.arange(-1, N - 1, dtype=np.int32)
    token = np.array([(3 * i + 1) % V for i in range(N)], np.int32)
    t = np.zeros((N + 1, V), np.float32)
    for r in range(N):
        t[r, token[r]] = 1.0
    t[N, 9] = 2.0
    ra, nodes, bonus = oracle.verify_greedy(t, parent, token)
    assert nodes.tolist() == list(range(N)) and bonus == 9
    # invalid parent (not an earlier node)
    with pytest.raises(oracle.OracleError):
        oracle.verify_greedy(np.zeros((3, 4), np.float32), np.array([-1, 1], np.int32), np.array([0, 1], np.int32))
    with pytest.raises(oracle.OracleError):
        oracle.verify_greedy(np.zeros((2, 4), np.float32), np.array([-1, 0], np.int32), np.array([0, 1], np.int32))


# ---------------------------------------------------------------------------- O11/O12 verification at T > 0
def _fixture_logits(rows):
    return np.array([[float(x) if x == "-inf" else _ev(x) for x in r] for r in rows], np.float32)


@pytest.mark.parametrize("case", [0, 1, 2])
def test_verify_sample_hand_case_a(case):
    """Hand-worked verification at T = 1, 0.5, 2 (section 3.1): draws by the id-order inverse CDF,
    a zero-mass id skipped at u = 0, accepted and rejected children."""
    g = _golden("verify_sample_case_a.json")
    c = g["cases"][case]
    rs, nodes, bonus = oracle.verify_sample(_fixture_logits(g["target"]), g["parent"], g["token"], c["T"],
                                            np.array(g["uniforms"], np.float32))
    assert rs.tolist() == c["expect_row_sample"]
    assert nodes.tolist() == c["expect_nodes"]
    assert bonus == c["expect_bonus"]
    assert len(nodes) + 1 == c["expect_tau"]


@pytest.mark.parametrize("T", [0.6, 1.0, 1.7])
def test_row_sample_is_the_inverse_cdf_of_the_tempered_softmax(T):
    """Stratified uniforms (i + 1/2) / M: each id is drawn for M p(id) +- 1 of them, p from scipy's
    softmax of logits / T, and the draw never decreases as u grows (cumulative in id order)."""
    from scipy.special import softmax
    rng = np.random.default_rng(11)
    V, M = 37, 20000
    row = (rng.standard_normal(V) * 2.0).astype(np.float32)
    row[5] = -np.inf
    p = softmax(row.astype(np.float64) / T)
    draws = np.array([oracle.row_sample(row, T, (i + 0.5) / M) for i in range(M)])
    assert np.all(np.diff(draws) >= 0)
    counts = np.bincount(draws, minlength=V)
    assert counts[5] == 0
    assert np.all(np.abs(counts - M * p) <= 1.0 + 1e-9)


def test_verify_sample_first_emitted_token_follows_the_target():
    """Lossless: whatever the tree, the first token the verification emits (the accepted child's or
    the bonus) is distributed as the target's own draw after the anchor; stratified over row 0's
    uniform, the other rows' uniforms fixed."""
    from scipy.special import softmax
    from paper_2605_29707_gb300 import inputs
    c = inputs.make_verify_case(1, 8, 6, 21, p_plant=1.0)
    T, M = 1.3, 6000
    tgt, par, tok = c.target[0], c.parent[0], c.token[0]
    p0 = softmax(tgt[0].astype(np.float64) / T)
    rest = inputs.uniform01(9, (21, "verify-sample-rest")).astype(np.float32)
    first = []
    for i in range(M):
        u = rest.copy()
        u[0] = (i + 0.5) / M
        rs, nodes, bonus = oracle.verify_sample(tgt, par, tok, T, u)
        first.append(int(tok[nodes[0]]) if len(nodes) else bonus)
        assert (int(tok[nodes[0]]) if len(nodes) else bonus) == rs[0]
    counts = np.bincount(first, minlength=6)
    assert np.all(np.abs(counts - M * p0) <= 1.0 + 1e-9)


@pytest.mark.parametrize("seed,N,V,chain", [(1, 12, 300, False), (3, 16, 1000, True), (5, 30, 64, False)])
def test_verify_sample_at_low_temperature_is_greedy(seed, N, V, chain):
    """With every row's maximum at least 1 above the rest and T = 0.01, the tempered softmax puts all
    but e^-100 of its mass on the argmax: every draw is the argmax and the walk is the greedy one."""
    from paper_2605_29707_gb300 import inputs
    c = inputs.make_verify_case(2, N, V, seed, p_plant=0.8, chain=chain)
    for b in range(2):
        t = c.target[b].copy()
        for r in range(N + 1):
            a = int(np.argmax(t[r]))
            t[r, a] = np.float32(np.max(np.delete(t[r], a)) + 1.0)
        u = inputs.uniform01(N + 1, (seed, "verify-sample-u", b)).astype(np.float32) * np.float32(0.999)
        rs, nodes, bonus = oracle.verify_sample(t, c.parent[b], c.token[b], 0.01, u)
        ra, gnodes, gbonus = oracle.verify_greedy(t, c.parent[b], c.token[b])
        assert rs.tolist() == ra.tolist()
        assert nodes.tolist() == gnodes.tolist() and bonus == gbonus


def test_verify_sample_special_cases():
    below_one = float(np.nextafter(np.float32(1.0), np.float32(0.0)))
    # u = 0: the first id of non-zero mass; u just below 1: the last one
    row = np.array([-np.inf, 0.0, 0.0, -np.inf], np.float32)
    assert oracle.row_sample(row, 1.0, 0.0) == 1
    assert oracle.row_sample(row, 1.0, below_one) == 2
    # a row with no finite value: id 0
    assert oracle.row_sample(np.full(4, -np.inf, np.float32), 1.0, 0.5) == 0
    # no nodes: the draw after the anchor is the bonus, tau = 1
    rs, nodes, bonus = oracle.verify_sample(np.array([[0.0, 0.0, 0.0, 0.0]], np.float32), np.zeros(0, np.int32),
                                            np.zeros(0, np.int32), 1.0, np.array([0.6], np.float32))
    assert rs.tolist() == [2] and len(nodes) == 0 and bonus == 2
    # bad temperature, bad uniforms, bad tree
    for T in (0.0, -1.0, float("inf"), float("nan")):
        with pytest.raises(oracle.OracleError):
            oracle.row_sample(row, T, 0.5)
    for u in (1.0, -0.1, float("nan")):
        with pytest.raises(oracle.OracleError):
            oracle.row_sample(row, 1.0, u)
    with pytest.raises(oracle.OracleError):
        oracle.verify_sample(np.zeros((3, 4), np.float32), np.array([-1, 1], np.int32), np.array([0, 1], np.int32),
                             1.0, np.zeros(3, np.float32))


# ---------------------------------------------------------------------------- O9 greedy rollout
def test_rollout_hand_case_c():
    """Hand-worked greedy rollout (section 4.1.2 / Fig. 3) from hand case C's numbers."""
    g = load("hand_case_c.json")
    r = load("rollout_case_c.json")
    w = {n: bf16(g[n]) for n in ("w_lm", "emb", "w_ih", "w_hh", "b_ih", "b_hh", "w1", "b1", "w2", "b2")}
    hidden = bf16(g["hidden"]).reshape(1, g["K"], g["H"])
    tokens, logp = oracle.rollout_greedy(w, hidden, np.array([r["anchor"]], np.int32))
    assert tokens[0].tolist() == r["expect_tokens"]
    assert logp[0] == pytest.approx(r["expect_logp"], abs=r["tolerance"])


def test_rollout_sample_hand_case_c():
    """Hand-worked sampled rollout (section 4.1.2 / Fig. 3) from hand case C's distributions:
    inverse-CDF choices in id order for given uniforms."""
    g = load("hand_case_c.json")
    r = load("rollout_sample_case_c.json")
    w = {n: bf16(g[n]) for n in ("w_lm", "emb", "w_ih", "w_hh", "b_ih", "b_hh", "w1", "b1", "w2", "b2")}
    hidden = bf16(g["hidden"]).reshape(1, g["K"], g["H"])
    for case in r["cases"]:
        uni = np.array([case["uniforms"]], np.float32)
        tokens, logp = oracle.rollout_sample(w, hidden, np.array([r["anchor"]], np.int32), uni)
        if "expect_tokens" in case:
            assert tokens[0].tolist() == case["expect_tokens"]
            assert logp[0] == pytest.approx(case["expect_logp"], abs=r["tolerance"])
        else:
            assert int(tokens[0, 0]) == case["expect_first"]
            assert logp[0, 0] == pytest.approx(case["expect_first_logp"], abs=r["tolerance"])


def test_rollout_sample_rejects_uniforms_outside_unit_interval():
    g = load("hand_case_c.json")
    w = {n: bf16(g[n]) for n in ("w_lm", "emb", "w_ih", "w_hh", "b_ih", "b_hh", "w1", "b1", "w2", "b2")}
    hidden = bf16(g["hidden"]).reshape(1, g["K"], g["H"])
    for bad in (1.0, -0.25, np.nan):
        with pytest.raises(RuntimeError):
            oracle.rollout_sample(w, hidden, np.array([2], np.int32), np.array([[0.5, bad]], np.float32))


def _small_weights(rng, V, H, Ds, R, biases):
    w = {"w_lm": rand_bf16(rng, (V, H), 0.3), "emb": rand_bf16(rng, (V, H), 0.5),
         "w_ih": rand_bf16(rng, (3 * Ds, H), 0.3), "w_hh": rand_bf16(rng, (3 * Ds, Ds), 0.3),
         "w1": rand_bf16(rng, (R, H + Ds), 0.3), "w2": rand_bf16(rng, (V, R), 0.8)}
    if biases:
        for n, m in (("b_ih", 3 * Ds), ("b_hh", 3 * Ds), ("b1", R), ("b2", V)):
            w[n] = rand_bf16(rng, (m,), 0.2)
    return w


@pytest.mark.parametrize("B,K,V,H,Ds,R,biases", [(2, 5, 40, 16, 6, 4, False), (3, 7, 13, 8, 3, 2, True),
                                                 (1, 6, 200, 24, 8, 8, True)])
def test_rollout_is_the_fixed_point_of_the_teacher_forced_step(B, K, V, H, Ds, R, biases):
    """The draft step fed the rollout's own tokens as its prefix has, at every position, the
    rollout's token as its argmax and the rollout's log-probability for it."""
    rng = np.random.default_rng(B * 100 + K)
    w = _small_weights(rng, V, H, Ds, R, biases)
    hidden = rand_bf16(rng, (B, K, H), 1.0)
    anchors = rng.integers(0, V, B).astype(np.int32)
    tokens, logp = oracle.rollout_greedy(w, hidden, anchors)
    prefix = np.concatenate([anchors[:, None], tokens[:, :-1]], axis=1).astype(np.int32)
    ref = oracle.draft_step(w, hidden, prefix, 1, 1, want_logp_full=True)
    for b in range(B):
        for j in range(K):
            row = ref["logp_full"][b, j]
            assert int(np.argmax(row)) == tokens[b, j]
            assert logp[b, j] == pytest.approx(row[tokens[b, j]], abs=1e-12)


@pytest.mark.parametrize("B,K,V,H,Ds,R,biases", [(2, 5, 40, 16, 6, 4, False), (3, 7, 13, 8, 3, 2, True)])
def test_rollout_sample_follows_the_teacher_forced_step(B, K, V, H, Ds, R, biases):
    """Fed the sampled tokens as its prefix, the (pinned) draft step gives, at every position, a
    distribution whose cumulative interval of the sampled token holds that step's uniform, and
    the sampled token's log-probability; uniforms near 0 and near 1 pick the first and the last
    id of non-zero probability."""
    rng = np.random.default_rng(B * 1000 + K)
    w = _small_weights(rng, V, H, Ds, R, biases)
    hidden = rand_bf16(rng, (B, K, H), 1.0)
    anchors = rng.integers(0, V, B).astype(np.int32)
    uni = rng.random((B, K), dtype=np.float32)
    uni[0, 0] = 0.0
    uni[-1, -1] = np.float32(1.0) - np.float32(2 ** -24)
    tokens, logp = oracle.rollout_sample(w, hidden, anchors, uni)
    prefix = np.concatenate([anchors[:, None], tokens[:, :-1]], axis=1).astype(np.int32)
    ref = oracle.draft_step(w, hidden, prefix, 1, 1, want_logp_full=True)
    for b in range(B):
        for j in range(K):
            p = np.exp(ref["logp_full"][b, j])
            t = int(tokens[b, j])
            lo, hi = float(np.sum(p[:t])), float(np.sum(p[: t + 1]))
            assert lo - 1e-12 <= uni[b, j] < hi + 1e-12, (b, j, t, lo, float(uni[b, j]), hi)
            assert logp[b, j] == pytest.approx(ref["logp_full"][b, j, t], abs=1e-12)
    assert int(tokens[0, 0]) == 0
    assert int(tokens[-1, -1]) == int(np.nonzero(np.exp(ref["logp_full"][B - 1, K - 1]) > 0)[0][-1])


def test_rollout_head_off_is_the_base_argmax_and_rejects_bad_anchors():
    rng = np.random.default_rng(7)
    V, H, K = 30, 12, 4
    w = {"w_lm": rand_bf16(rng, (V, H), 0.4)}
    hidden = rand_bf16(rng, (2, K, H), 1.0)
    tokens, logp = oracle.rollout_greedy(w, hidden, np.array([3, 4], np.int32))
    z = np.einsum("bkh,vh->bkv", to_f64(hidden), to_f64(w["w_lm"]))
    assert tokens.tolist() == np.argmax(z, axis=2).tolist()
    with pytest.raises(oracle.OracleError):
        oracle.rollout_greedy(w, hidden, np.array([3, V], np.int32))


# ---------------------------------------------------------------------------- O13-O15 exponential race
def test_philox_known_answer_vectors():
    """O13 against the generator's published known-answer vectors."""
    g = load("philox4x32_10_kat.json")
    for v in g["vectors"]:
        ctr = [int(x, 16) for x in v["ctr"]]
        key = [int(x, 16) for x in v["key"]]
        assert [int(x) for x in oracle.philox4x32_10(ctr, key)] == [int(x, 16) for x in v["out"]]


def test_gumbel_rows_have_the_standard_gumbel_law():
    """O14: 2^20 perturbations of one row follow the standard Gumbel law (mean = the
    Euler-Mascheroni constant, variance pi^2 / 6, P(g <= 0) = 1/e, every value inside the range the
    23-bit uniform allows), and rows of other sequences and steps are uncorrelated with it."""
    n = 1 << 20
    g = oracle.gumbel_row(0x0123456789ABCDEF, 5, 3, n)
    assert np.isfinite(g).all()
    lo, hi = -math.log(-math.log(2.0 ** -24)), -math.log(-math.log(1.0 - 2.0 ** -24))
    assert lo - 1e-12 <= g.min() and g.max() <= hi + 1e-12
    assert abs(g.mean() - 0.5772156649015329) < 5 * math.sqrt(math.pi ** 2 / 6 / n)
    assert abs(g.var() - math.pi ** 2 / 6) < 0.02
    assert abs(np.mean(g <= 0.0) - math.exp(-1.0)) < 5 * math.sqrt(math.exp(-1) * (1 - math.exp(-1)) / n)
    for b, j in ((4, 3), (6, 3), (5, 2), (5, 4)):  # same word of another group; another word; other steps
        other = oracle.gumbel_row(0x0123456789ABCDEF, b, j, n)
        assert abs(np.corrcoef(g, other)[0, 1]) < 5 / math.sqrt(n)
    assert abs(np.corrcoef(g, oracle.gumbel_row(0x0123456789ABCDF0, 5, 3, n))[0, 1]) < 5 / math.sqrt(n)


def test_rollout_sample_gumbel_draws_follow_the_softmax():
    """O15 with the correction branch off (the logits of a position do not depend on the tokens
    drawn before it): over 6000 sequences with the same hidden rows, the tokens drawn at each
    position have the softmax's frequencies (chi-square, 5 categories), and logp is the
    log-softmax of the drawn token."""
    rng = np.random.default_rng(11)
    V, H, K, B = 5, 8, 2, 6000
    w = {"w_lm": rand_bf16(rng, (V, H), 0.6)}
    one = rand_bf16(rng, (1, K, H), 1.0)
    hidden = np.repeat(one, B, axis=0)
    anchors = np.zeros(B, np.int32)
    tokens, logp = oracle.rollout_sample_gumbel(w, hidden, anchors, 77)
    z = np.einsum("kh,vh->kv", to_f64(one[0]), to_f64(w["w_lm"]))
    lp = z - np.log(np.exp(z - z.max(axis=1, keepdims=True)).sum(axis=1, keepdims=True)) - z.max(axis=1, keepdims=True)
    for j in range(K):
        p = np.exp(lp[j])
        counts = np.bincount(tokens[:, j], minlength=V)
        chi2 = float(np.sum((counts - B * p) ** 2 / (B * p)))
        assert chi2 < 35.0, (j, counts.tolist(), (B * p).round(1).tolist())  # df 4: p < 1e-6 by chance
        assert np.allclose(logp[:, j], lp[j][tokens[:, j]], atol=1e-12)


@pytest.mark.parametrize("B,K,V,H,Ds,R,biases", [(2, 5, 40, 16, 6, 4, False), (5, 7, 13, 8, 3, 2, True)])
def test_rollout_sample_gumbel_follows_the_teacher_forced_step(B, K, V, H, Ds, R, biases):
    """Fed the drawn tokens as its prefix, the (pinned) draft step gives, at every position, a
    distribution whose log-probabilities plus the (pinned) perturbations of that sequence and step
    are largest at the drawn token, and the drawn token's log-probability; another seed draws
    other tokens."""
    rng = np.random.default_rng(B * 10000 + K)
    w = _small_weights(rng, V, H, Ds, R, biases)
    hidden = rand_bf16(rng, (B, K, H), 1.0)
    anchors = rng.integers(0, V, B).astype(np.int32)
    seed = 0xFEEDFACE12345678
    tokens, logp = oracle.rollout_sample_gumbel(w, hidden, anchors, seed)
    prefix = np.concatenate([anchors[:, None], tokens[:, :-1]], axis=1).astype(np.int32)
    ref = oracle.draft_step(w, hidden, prefix, 1, 1, want_logp_full=True)
    for b in range(B):
        for j in range(K):
            key = ref["logp_full"][b, j] + oracle.gumbel_row(seed, b, j, V)
            t = int(tokens[b, j])
            assert t == int(np.argmax(key)), (b, j)
            assert logp[b, j] == pytest.approx(ref["logp_full"][b, j, t], abs=1e-12)
    other, _ = oracle.rollout_sample_gumbel(w, hidden, anchors, seed + 1)
    assert (other != tokens).any()


def test_rollout_sample_gumbel_exact_tie_takes_the_lower_id():
    """O15's tie rule: two ids whose perturbations coincide exactly (the 23-bit uniform repeats
    about once per 2^23 pairs, so a row of 2^16 perturbations holds a few such pairs) and whose
    logits are equal and far above the rest tie exactly; the lower id is drawn."""
    seed = 99
    g = oracle.gumbel_row(seed, 0, 0, 1 << 16)
    order = np.argsort(g, kind="stable")
    same = np.nonzero(g[order[1:]] == g[order[:-1]])[0]
    assert same.size > 0
    v1, v2 = sorted((int(order[same[0]]), int(order[same[0] + 1])))
    V, H = v2 + 1, 8
    w_lm = np.zeros((V, H), np.float32)
    w_lm[v1, 0] = w_lm[v2, 0] = 30.0  # 30 + g > 27 beats 0 + g < 17 for every other id
    hidden = np.zeros((1, 1, H), np.float32)
    hidden[0, 0, 0] = 1.0
    tokens, logp = oracle.rollout_sample_gumbel({"w_lm": bf16(w_lm)}, bf16(hidden), np.array([0], np.int32), seed)
    assert int(tokens[0, 0]) == v1
    z = np.zeros(V)
    z[[v1, v2]] = 30.0
    assert logp[0, 0] == pytest.approx(30.0 - (z.max() + np.log(np.exp(z - z.max()).sum())), abs=1e-9)


def test_gumbel_row_reaches_both_ends_of_the_uniform_finitely():
    """O14's uniform never reaches 0 or 1: the words whose top 23 bits are all zero or all one
    (one in 2^23 each) give the smallest and largest perturbations, -log(-log(2^-24)) and
    -log(-log(1 - 2^-24)), both finite; scanning rows of 2^22 perturbations finds both."""
    lo, hi = -math.log(-math.log(2.0 ** -24)), -math.log(-math.log(1.0 - 2.0 ** -24))
    found_lo = found_hi = False
    for j in range(24):
        g = oracle.gumbel_row(7, 1, j, 1 << 22)
        assert np.isfinite(g).all(), j
        assert g.min() >= lo - 1e-12 and g.max() <= hi + 1e-12
        found_lo |= abs(float(g.min()) - lo) < 1e-12
        found_hi |= abs(float(g.max()) - hi) < 1e-12
        if found_lo and found_hi:
            break
    assert found_lo and found_hi
