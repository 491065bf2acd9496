"""The draft step for callers that cannot allocate device memory.

Such callers (code inside a host framework that owns every allocation, a plugin in a process
with a fixed memory pool, a real-time path that must not risk an allocation) call
domino_draft_step_static_scratch, which runs the same step with the library's static 16 MiB
device array as scratch.  This file is collected last; it checks the new entry point through
the C ABI against the existing workspace entry point and against the oracle, on two calls in a
row, and works both alone in a fresh process and after the other tests.  Because every call of
the process shares the one array, calls of different kinds back to back (a small batch, the
correction branch off, the small batch again) are its normal case and are checked too.
"""
import numpy as np
import pytest
import torch

from paper_2605_29707_gb300 import binding, inputs
from paper_2605_29707_gb300.step import DraftStep
from tests.test_gpu_parity import _check

pytestmark = pytest.mark.gpu

LOGP_TOL = 2e-2  # the tolerance the parity tests use for log-probabilities


def _compare(cfg, table=False, head_on=True):
    dev = torch.device("cuda:0")
    wl = inputs.make_workload(cfg)
    c = wl.cfg
    st = DraftStep(wl.weights, c.B, c.K, c.H, c.V, c.k, c.N, Ds=c.Ds, R=c.R, device=dev, input_table=table,
                   head_on=head_on)
    hidden = torch.from_numpy(wl.hidden.view(np.int16)).view(torch.bfloat16).to(dev)
    ids = torch.from_numpy(wl.prefix_ids).to(dev)
    ref = st.run(hidden, ids)  # existing entry point, caller-allocated workspace

    M = c.B * c.K
    status = torch.full((1,), 12345, dtype=torch.int32, device=dev)
    for call in range(2):
        out = {
            "topk_ids": torch.full((M * c.k,), -7, dtype=torch.int32, device=dev),
            "topk_logp": torch.full((M * c.k,), 7.0, dtype=torch.float32, device=dev),
            "tree_parent": torch.full((c.B * c.N,), -7, dtype=torch.int32, device=dev),
            "tree_token": torch.full((c.B * c.N,), -7, dtype=torch.int32, device=dev),
            "tree_depth": torch.full((c.B * c.N,), -7, dtype=torch.int32, device=dev),
            "tree_score": torch.full((c.B * c.N,), 7.0, dtype=torch.float32, device=dev),
        }
        rc = binding.domino_draft_step_static_scratch(
            hidden, ids, st.w["w_lm"], st.head, c.B, c.K, c.H, c.V, c.k, c.N,
            out["topk_ids"], out["topk_logp"],
            out["tree_parent"], out["tree_token"], out["tree_depth"], out["tree_score"], status,
            torch.cuda.current_stream(dev))
        assert rc == 0, binding.domino_status_string(rc)
        torch.cuda.synchronize(dev)
        assert int(status.item()) == 0, f"call {call}: device status {int(status.item())}"
        np.testing.assert_array_equal(out["topk_ids"].view(c.B, c.K, c.k).cpu().numpy(), ref["topk_ids"])
        np.testing.assert_allclose(out["topk_logp"].view(c.B, c.K, c.k).cpu().numpy(), ref["topk_logp"],
                                   atol=LOGP_TOL, rtol=0)
        for key in ("tree_parent", "tree_token", "tree_depth"):
            np.testing.assert_array_equal(out[key].view(c.B, c.N).cpu().numpy(), ref[key])
        np.testing.assert_allclose(out["tree_score"].view(c.B, c.N).cpu().numpy(), ref["tree_score"],
                                   atol=LOGP_TOL, rtol=0)
        got = {"topk_ids": out["topk_ids"].view(c.B, c.K, c.k).cpu().numpy(),
               "topk_logp": out["topk_logp"].view(c.B, c.K, c.k).cpu().numpy(),
               **{key: out[key].view(c.B, c.N).cpu().numpy()
                  for key in ("tree_parent", "tree_token", "tree_depth", "tree_score")}}
        ex_topk, ex_tree = _check(wl, got, head_on=head_on)
        assert ex_topk <= max(1, c.M * c.k // 50)
        assert ex_tree <= max(1, c.B * c.N // 10)


@pytest.mark.parametrize("name,table", [("tiny", False), ("B2", False), ("B2", True)])
def test_static_scratch_matches_workspace_entry_point(name, table):
    cfg = inputs.CONFIGS["tiny"] if name == "tiny" else inputs.custom_config(
        name, B=2, K=8, H=256, V=3000, Ds=64, R=64, k=6, N=12, seed=31, biases=True)
    _compare(cfg, table)


def test_static_scratch_small_batch_after_correction_off():
    """A small batch (its GRU clears nothing before the step), then the same shape with the
    correction branch off (a different layout of the shared array), then the small batch again."""
    kw = dict(B=2, K=16, H=256, V=2000, Ds=1024, R=64, k=4, N=8, seed=61, biases=True)
    _compare(inputs.custom_config("B2-big", **kw))
    _compare(inputs.custom_config("B2-big", **kw), head_on=False)
    _compare(inputs.custom_config("B2-big", **kw))


def test_static_scratch_rejects_sizes_beyond_the_array():
    c = inputs.CONFIGS["qwen3-8b-b32"]
    need = binding.domino_workspace_bytes(c.B, c.K, c.H, c.V, c.Ds, c.R, c.k, c.N)
    assert need > binding.DOMINO_STATIC_SCRATCH_BYTES
    dev = torch.device("cuda:0")
    dummy = torch.empty(16, dtype=torch.uint8, device=dev)  # never touched: rejected before launch
    head = binding.make_head(dummy, dummy, dummy, None, None, dummy, None, dummy, None, c.Ds, c.R)
    rc = binding.domino_draft_step_static_scratch(dummy, dummy, dummy, head, c.B, c.K, c.H, c.V, c.k, c.N,
                                                  dummy, dummy, dummy, dummy, dummy, None, None)
    assert rc == binding.DOMINO_ERR_UNSUPPORTED
