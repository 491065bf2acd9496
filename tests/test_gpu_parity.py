"""GPU parity: the CUDA step (through the C ABI) against the fp64 oracle on the same seeded inputs.

Small cases cover several tiles and ragged tails in every dimension (tokens, hidden size,
rank, vocabulary), both GEMM orientations (<= 128 tokens: weights on the 128-row MMA operand;
more: tokens on it), both top-k widths, biases, the correction-off path and bad ids.  The
full Qwen3-shaped configurations run the launch configuration the benchmark times, and the
oracle checks every sequence of them.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2605_29707_gb300 import binding, inputs
from paper_2605_29707_gb300.step import DraftStep
from tests.parity import check_topk, check_tree

pytestmark = pytest.mark.gpu


def _dev():
    return torch.device("cuda:0")


def _run_gpu(wl, head_on=True, table=False):
    c = wl.cfg
    st = DraftStep(wl.weights, c.B, c.K, c.H, c.V, c.k, c.N, Ds=c.Ds, R=c.R, device=_dev(), head_on=head_on,
                   input_table=table)
    hidden = torch.from_numpy(wl.hidden.view(np.int16)).view(torch.bfloat16).to(_dev())
    ids = torch.from_numpy(wl.prefix_ids).to(_dev())
    out = st.run(hidden, ids)
    return st, out, hidden, ids


def _check(wl, out, seqs=None, head_on=True, batch=8):
    """Every sequence in `seqs` (default: all) against the oracle, `batch` sequences of full
    [K, V] fp64 log-probs at a time.  Returns the gap-excused top-k and tree differences."""
    c = wl.cfg
    w = dict(wl.weights)
    if not head_on:
        w["w2"] = None
    seqs = list(range(c.B)) if seqs is None else list(seqs)
    ex_topk = ex_tree = 0
    for lo in range(0, len(seqs), batch):
        part = seqs[lo:lo + batch]
        ref = oracle.draft_step(w, wl.hidden, wl.prefix_ids, c.k, c.N, seqs=part, want_logp_full=True)
        for si, b in enumerate(part):
            ex_topk += check_topk(out["topk_ids"][b], out["topk_logp"][b], ref["logp_full"][si], c.k)
            ex_tree += check_tree(out["tree_parent"][b], out["tree_token"][b], out["tree_depth"][b],
                                  out["tree_score"][b], out["topk_ids"][b], ref["logp_full"][si], c.K, c.N,
                                  oracle_tree=(ref["tree_parent"][si], ref["tree_token"][si]))
    return ex_topk, ex_tree


SMALL = {
    # one 128-row vocabulary tile short of a full chunk, ragged K tail in both segments
    "ragged-swap16": dict(B=3, K=5, H=328, V=5000, Ds=136, R=72, k=5, N=12, seed=11, biases=True),
    "swap32-k20": dict(B=2, K=13, H=256, V=2600, Ds=64, R=64, k=20, N=40, seed=12),
    "swap64": dict(B=4, K=16, H=192, V=3001, Ds=128, R=128, k=8, N=16, seed=13),
    "swap128": dict(B=7, K=16, H=128, V=1900, Ds=96, R=64, k=4, N=10, seed=14, biases=True),
    "normal-2tiles": dict(B=12, K=16, H=256, V=3000, Ds=128, R=64, k=8, N=16, seed=15),
    "normal-ragged": dict(B=9, K=31, H=200, V=2049, Ds=72, R=40, k=3, N=7, seed=16, biases=True),
    "k1-chain": dict(B=2, K=6, H=64, V=700, Ds=32, R=16, k=1, N=6, seed=17),
    "K1": dict(B=5, K=1, H=64, V=900, Ds=32, R=16, k=6, N=6, seed=18),
    # the GRU computes its own projections (three launches): H not a multiple of 64 (a short last
    # k chunk), 32 GRU CTAs, four u pairs per warp
    "fused-ragged": dict(B=2, K=7, H=328, V=5000, Ds=256, R=64, k=5, N=12, seed=19, biases=True),
    # the largest k and N the boundary accepts: 32-entry lists, a 256-node tree (slots past 32
    # live in shared memory), on a vocabulary with a ragged last chunk
    "max-k-N": dict(B=2, K=8, H=128, V=3001, Ds=64, R=32, k=32, N=256, seed=20),
    # the largest K (64 positions: the GRU's longest recurrence, the deepest tree rows)
    "max-K": dict(B=1, K=64, H=64, V=800, Ds=32, R=16, k=3, N=40, seed=21, biases=True),
    # the longest block the fused-projection GRU takes (M = 32)
    "fused-K32": dict(B=1, K=32, H=128, V=1500, Ds=256, R=32, k=4, N=30, seed=22),
    # tokens on M in CTA pairs (the 2-SM MMA kernel): 32-entry lists (k = 20), and a second token
    # tile of 22 rows (M = 150) with a ragged vocabulary and biases
    "pair-k20": dict(B=10, K=16, H=192, V=3001, Ds=64, R=64, k=20, N=24, seed=26, biases=True),
    "pair-ragged": dict(B=10, K=15, H=136, V=2333, Ds=72, R=40, k=6, N=10, seed=27, biases=True),
}


@pytest.mark.parametrize("name", ["tiny"] + list(SMALL))
def test_small_parity(name):
    cfg = inputs.CONFIGS["tiny"] if name == "tiny" else inputs.custom_config(name, **SMALL[name])
    wl = inputs.make_workload(cfg)
    _, out, _, _ = _run_gpu(wl)
    ex_topk, ex_tree = _check(wl, out)
    # gap-excused differences are allowed but must stay rare on these inputs
    assert ex_topk <= max(1, cfg.M * cfg.k // 50)
    assert ex_tree <= max(1, cfg.B * cfg.N // 10)


# the input-projection table in place of the GRU's own E . W_ih^T: the fused path (B <= 2), the
# chained small-M path, the large-M path, K = 1
TABLE = ["tiny", "ragged-swap16", "swap64", "normal-2tiles", "normal-ragged", "K1", "fused-ragged", "fused-K32"]


@pytest.mark.parametrize("name", TABLE)
def test_small_parity_with_input_table(name):
    cfg = inputs.CONFIGS["tiny"] if name == "tiny" else inputs.custom_config(name, **SMALL[name])
    wl = inputs.make_workload(cfg)
    _, out, _, _ = _run_gpu(wl, table=True)
    ex_topk, ex_tree = _check(wl, out)
    assert ex_topk <= max(1, cfg.M * cfg.k // 50)
    assert ex_tree <= max(1, cfg.B * cfg.N // 10)


@pytest.mark.parametrize("name,table", [("fused-ragged", False), ("fused-ragged", True), ("swap64", False),
                                        ("swap64", True), ("normal-2tiles", False), ("normal-2tiles", True)])
def test_launches_per_step_counts_the_kernels(name, table):
    """The kernels one step launches (the library's per-launch timing hooks) are as many as
    domino_launches_per_step (_table with an input table) says."""
    cfg = inputs.custom_config(name, **SMALL[name])
    wl = inputs.make_workload(cfg)
    st, _, hidden, ids = _run_gpu(wl, table=table)
    binding.domino_timing_begin(64)
    assert st.enqueue(hidden, ids) == 0
    torch.cuda.synchronize()
    launched = sum(n for _, n in binding.domino_timing_end().values())
    assert launched == st.launches_per_step()
    if table:
        c = wl.cfg
        plain = binding.domino_launches_per_step(c.B, c.K, c.H, c.V, c.Ds, c.R, c.k, c.N)
        assert launched == (3 if plain == 3 else plain - 1)


@pytest.mark.parametrize("B,K,launches", [(1, 4, 3), (4, 16, 5)])
def test_bad_token_reported_with_input_table(B, K, launches):
    """With the table an out-of-range id is still reported (the GRU's own check at B <= 2, the
    gather's otherwise), and the GRU reads a valid table row for it."""
    wl = inputs.make_workload(inputs.custom_config("bad-t", B=B, K=K, H=64, V=500, Ds=32, R=16, k=2, N=3, seed=25))
    c = wl.cfg
    st = DraftStep(wl.weights, c.B, c.K, c.H, c.V, c.k, c.N, Ds=c.Ds, R=c.R, device=_dev(), input_table=True)
    assert st.launches_per_step() == launches
    hidden = torch.from_numpy(wl.hidden.view(np.int16)).view(torch.bfloat16).to(_dev())
    ids = torch.from_numpy(wl.prefix_ids).to(_dev())
    ids[B - 1, K - 1] = -2
    assert st.enqueue(hidden, ids) == 0
    assert binding.domino_check_status(st.workspace, torch.cuda.current_stream()) == binding.DOMINO_ERR_BAD_TOKEN
    ids[B - 1, K - 1] = 7
    assert st.enqueue(hidden, ids) == 0
    assert binding.domino_check_status(st.workspace, torch.cuda.current_stream()) == 0


def test_correction_off_is_base_distribution():
    cfg = inputs.custom_config("off", B=2, K=8, H=256, V=3000, Ds=64, R=64, k=6, N=12, seed=21, biases=True)
    wl = inputs.make_workload(cfg)
    _, out, _, _ = _run_gpu(wl, head_on=False)
    _check(wl, out, head_on=False)


def test_deterministic_and_host_entry_point_matches():
    wl = inputs.make_workload(inputs.custom_config("det", B=2, K=8, H=256, V=4000, Ds=64, R=64, k=8, N=16, seed=22))
    st, out1, hidden, ids = _run_gpu(wl)
    out2 = st.run(hidden, ids)
    for key in out1:
        np.testing.assert_array_equal(out1[key], out2[key])
    c = wl.cfg
    host = {
        "topk_ids": torch.empty(c.M * c.k, dtype=torch.int32).pin_memory(),
        "topk_logp": torch.empty(c.M * c.k, dtype=torch.float32).pin_memory(),
        "tree_parent": torch.empty(c.B * c.N, dtype=torch.int32).pin_memory(),
        "tree_token": torch.empty(c.B * c.N, dtype=torch.int32).pin_memory(),
        "tree_depth": torch.empty(c.B * c.N, dtype=torch.int32).pin_memory(),
        "tree_score": torch.empty(c.B * c.N, dtype=torch.float32).pin_memory(),
    }
    rc = st.run_host(hidden.cpu().pin_memory(), ids.cpu().pin_memory(), host)
    assert rc == 0, binding.domino_status_string(rc)
    np.testing.assert_array_equal(host["topk_ids"].numpy().reshape(out1["topk_ids"].shape), out1["topk_ids"])
    np.testing.assert_array_equal(host["tree_token"].numpy().reshape(out1["tree_token"].shape), out1["tree_token"])
    np.testing.assert_array_equal(host["tree_score"].numpy().reshape(out1["tree_score"].shape), out1["tree_score"])


@pytest.mark.parametrize("B,K,table", [(1, 6, False), (4, 16, False), (1, 6, True), (4, 16, True)])
def test_consecutive_steps_on_one_workspace(B, K, table):
    """Steps with different inputs back to back on one workspace each match the oracle: state
    words a previous step left behind (tagged with its epoch at B <= 2, cleared at larger B)
    never pass for the current step's."""
    cfg = inputs.custom_config("consec", B=B, K=K, H=256, V=2000, Ds=64, R=64, k=4, N=8, seed=41, biases=True)
    wl_a = inputs.make_workload(cfg)
    # same head and LM head, new hidden states and prefixes
    wl_b = inputs.make_workload(inputs.custom_config("consec", B=B, K=K, H=256, V=2000, Ds=64, R=64, k=4, N=8,
                                                     seed=42, biases=True), weights=wl_a.weights)
    c = wl_a.cfg
    st = DraftStep(wl_a.weights, c.B, c.K, c.H, c.V, c.k, c.N, Ds=c.Ds, R=c.R, device=_dev(), input_table=table)
    for wl in (wl_a, wl_b, wl_a, wl_b):
        hidden = torch.from_numpy(wl.hidden.view(np.int16)).view(torch.bfloat16).to(_dev())
        ids = torch.from_numpy(wl.prefix_ids).to(_dev())
        out = st.run(hidden, ids)
        ex_topk, ex_tree = _check(wl, out)
        assert ex_topk <= max(1, c.M * c.k // 50)
        assert ex_tree <= max(1, c.B * c.N // 10)


# the GRU's own id check (3 launches) and the gather kernel's (6 launches)
@pytest.mark.parametrize("B,K,expect", [(1, 4, 3), (4, 16, 6)])
def test_bad_token_reported_by_device_status(B, K, expect):
    wl = inputs.make_workload(inputs.custom_config("bad", B=B, K=K, H=64, V=500, Ds=32, R=16, k=2, N=3, seed=23))
    c = wl.cfg
    assert binding.domino_launches_per_step(c.B, c.K, c.H, c.V, c.Ds, c.R, c.k, c.N) == expect
    st = DraftStep(wl.weights, c.B, c.K, c.H, c.V, c.k, c.N, Ds=c.Ds, R=c.R, device=_dev())
    hidden = torch.from_numpy(wl.hidden.view(np.int16)).view(torch.bfloat16).to(_dev())
    ids = torch.from_numpy(wl.prefix_ids).to(_dev())
    ids[0, 2] = c.V  # out of range
    assert st.enqueue(hidden, ids) == 0
    assert binding.domino_check_status(st.workspace, torch.cuda.current_stream()) == binding.DOMINO_ERR_BAD_TOKEN
    # the next good step clears the status
    ids[0, 2] = 1
    assert st.enqueue(hidden, ids) == 0
    assert binding.domino_check_status(st.workspace, torch.cuda.current_stream()) == 0


def test_unsupported_and_invalid_arguments_on_device():
    wl = inputs.make_workload(inputs.custom_config("args", B=1, K=4, H=64, V=500, Ds=32, R=16, k=2, N=3, seed=24))
    c = wl.cfg
    st = DraftStep(wl.weights, c.B, c.K, c.H, c.V, c.k, c.N, Ds=c.Ds, R=c.R, device=_dev())
    hidden = torch.from_numpy(wl.hidden.view(np.int16)).view(torch.bfloat16).to(_dev())
    ids = torch.from_numpy(wl.prefix_ids).to(_dev())
    args = dict(hidden=hidden, prefix_ids=ids, w_lm=st.w["w_lm"], head=st.head, B=1, K=4, H=64, V=500, k=2, N=3,
                topk_ids=st.topk_ids, topk_logp=st.topk_logp, tree_parent=st.tree_parent,
                tree_token=st.tree_token, tree_depth=st.tree_depth, tree_score=st.tree_score,
                workspace=st.workspace, workspace_bytes=st.ws_bytes)
    assert binding.domino_draft_step(**args) == 0
    assert binding.domino_draft_step(**dict(args, workspace_bytes=st.ws_bytes - 1)) == binding.DOMINO_ERR_INVALID_ARG
    assert binding.domino_draft_step(**dict(args, N=31)) == binding.DOMINO_ERR_INVALID_ARG  # > 2+4+8+16
    assert binding.domino_draft_step(**dict(args, hidden=hidden.data_ptr() + 2)) == binding.DOMINO_ERR_UNSUPPORTED
    assert binding.domino_draft_step(**dict(args, k=33)) in (binding.DOMINO_ERR_UNSUPPORTED,
                                                             binding.DOMINO_ERR_INVALID_ARG)
    torch.cuda.synchronize()


FULL = ["qwen3-1.7b", "qwen3-8b", "qwen3-8b-b32", "qwen3-32b-b64"]


@pytest.mark.slow
@pytest.mark.parametrize("name,table", [(n, False) for n in FULL] + [("qwen3-8b", True), ("qwen3-8b-b32", True)])
def test_full_size_parity(name, table):
    """Every sequence of every full-size configuration (all 32 and all 64 of the serving
    batches) against the oracle, in the launch configuration the benchmark times."""
    wl = inputs.cached_workload(name)
    c = wl.cfg
    _, out, _, _ = _run_gpu(wl, table=table)
    ex_topk, ex_tree = _check(wl, out)
    assert ex_topk <= max(1, c.B * c.K * c.k // 20)
    assert ex_tree <= max(1, c.B * c.N // 10)
    for b in range(c.B):
        par, dep, sc = out["tree_parent"][b], out["tree_depth"][b], out["tree_score"][b]
        assert np.all(par < np.arange(c.N)) and np.all(np.diff(sc) <= 1e-6)
        assert np.all((dep >= 1) & (dep <= c.K))
        assert np.all(np.diff(out["topk_logp"][b], axis=-1) <= 0)
