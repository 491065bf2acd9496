"""One workspace reused by steps of different shapes and kinds, every step against the oracle.

Small batches (B <= 2 at K = 16) clear nothing before a step: their GRU state words carry the
step's tag and are trusted only where the workspace's control words record that the last step
left nothing but state words there.  A step of another shape or kind (a larger batch, the
correction branch off, a smaller fused step) leaves other data (embedding rows, projection
partial sums, softmax records) where the next fused step keeps its states, and some of those
words could carry the right tag by chance; these sequences make the fused step's state region
grow over such data, and check that every step still matches the oracle.
"""
import numpy as np
import pytest
import torch

from paper_2605_29707_gb300 import binding, inputs
from paper_2605_29707_gb300.step import DraftStep
from tests.test_gpu_parity import _check

pytestmark = pytest.mark.gpu

# shapes: a non-fused chained batch (gather + projection GEMMs), a large fused step (M . d_s =
# 32 x 1024 state words), a small fused step (its state range lies inside the large one's)
SHAPES = {
    "chained-B4": dict(B=4, K=16, H=256, V=2000, Ds=64, R=64, k=4, N=8, seed=51, biases=True),
    "fused-big": dict(B=2, K=16, H=256, V=2000, Ds=1024, R=64, k=4, N=8, seed=52, biases=True),
    "fused-small": dict(B=1, K=4, H=256, V=2000, Ds=256, R=32, k=4, N=8, seed=53),
    "large-M": dict(B=12, K=16, H=256, V=3000, Ds=128, R=64, k=8, N=16, seed=54),
}


def _dev():
    return torch.device("cuda:0")


class _Case:
    """Device weights and inputs of one shape; outputs written into fresh buffers per call."""

    def __init__(self, name, head_on=True):
        self.wl = inputs.make_workload(inputs.custom_config(name, **SHAPES[name]))
        c = self.c = self.wl.cfg
        self.head_on = head_on
        self.st = DraftStep(self.wl.weights, c.B, c.K, c.H, c.V, c.k, c.N, Ds=c.Ds, R=c.R, device=_dev(),
                            head_on=head_on)
        self.hidden = torch.from_numpy(self.wl.hidden.view(np.int16)).view(torch.bfloat16).to(_dev())
        self.ids = torch.from_numpy(self.wl.prefix_ids).to(_dev())

    def ws_bytes(self):
        return self.st.ws_bytes

    def _outs(self):
        c = self.c
        M = c.B * c.K
        return {"topk_ids": torch.full((M * c.k,), -7, dtype=torch.int32, device=_dev()),
                "topk_logp": torch.full((M * c.k,), 7.0, dtype=torch.float32, device=_dev()),
                "tree_parent": torch.full((c.B * c.N,), -7, dtype=torch.int32, device=_dev()),
                "tree_token": torch.full((c.B * c.N,), -7, dtype=torch.int32, device=_dev()),
                "tree_depth": torch.full((c.B * c.N,), -7, dtype=torch.int32, device=_dev()),
                "tree_score": torch.full((c.B * c.N,), 7.0, dtype=torch.float32, device=_dev())}

    def _numpy(self, o):
        c = self.c
        return {"topk_ids": o["topk_ids"].view(c.B, c.K, c.k).cpu().numpy(),
                "topk_logp": o["topk_logp"].view(c.B, c.K, c.k).cpu().numpy(),
                **{key: o[key].view(c.B, c.N).cpu().numpy()
                   for key in ("tree_parent", "tree_token", "tree_depth", "tree_score")}}

    def run_on(self, workspace, nbytes):
        c, o = self.c, self._outs()
        head = self.st.head  # head off: w2 NULL (the correction branch off), b2 still applied
        rc = binding.domino_draft_step(self.hidden, self.ids, self.st.w["w_lm"], head, c.B, c.K, c.H, c.V, c.k,
                                       c.N, o["topk_ids"], o["topk_logp"], o["tree_parent"], o["tree_token"],
                                       o["tree_depth"], o["tree_score"], workspace, nbytes,
                                       torch.cuda.current_stream())
        assert rc == 0, binding.domino_status_string(rc)
        st = binding.domino_check_status(workspace, torch.cuda.current_stream())
        assert st == 0, binding.domino_status_string(st)
        return self._numpy(o)

    def run_static(self):
        c, o = self.c, self._outs()
        head = self.st.head  # head off: w2 NULL (the correction branch off), b2 still applied
        status = torch.full((1,), 12345, dtype=torch.int32, device=_dev())
        rc = binding.domino_draft_step_static_scratch(
            self.hidden, self.ids, self.st.w["w_lm"], head, c.B, c.K, c.H, c.V, c.k, c.N, o["topk_ids"],
            o["topk_logp"], o["tree_parent"], o["tree_token"], o["tree_depth"], o["tree_score"], status,
            torch.cuda.current_stream())
        assert rc == 0, binding.domino_status_string(rc)
        torch.cuda.synchronize()
        assert int(status.item()) == 0, binding.domino_status_string(int(status.item()))
        return self._numpy(o)

    def check(self, out):
        ex_topk, ex_tree = _check(self.wl, out, head_on=self.head_on)
        c = self.c
        assert ex_topk <= max(1, c.M * c.k // 50)
        assert ex_tree <= max(1, c.B * c.N // 10)


# Each sequence grows the fused step's state range over another step's data at least once.
SEQUENCES = {
    "fused-after-chained": ["chained-B4", "fused-big", "fused-big", "chained-B4", "fused-big"],
    "fused-after-head-off": ["fused-big", "fused-big:off", "fused-big", "fused-big"],
    "fused-shrink-then-grow": ["fused-big", "fused-small", "fused-big", "fused-small", "fused-small",
                               "fused-big"],
    "fused-after-large-M": ["large-M", "fused-small", "large-M", "fused-big", "large-M:off", "fused-big"],
}


def _run_sequence(names, run):
    """Runs the steps in order; a failure names the step and its shape."""
    for i, (name, cs) in enumerate(zip(names, _cases(names))):
        try:
            cs.check(run(cs))
        except AssertionError as e:
            raise AssertionError(f"step {i} ({name}) of {names}: {e}") from e


def _cases(names):
    cache = {}
    out = []
    for n in names:
        if n not in cache:
            base, _, mode = n.partition(":")
            cache[n] = _Case(base, head_on=(mode != "off"))
        out.append(cache[n])
    return out


@pytest.mark.parametrize("seq", list(SEQUENCES))
def test_one_workspace_across_shapes(seq):
    nbytes = max(cs.ws_bytes() for cs in _cases(SEQUENCES[seq]))
    ws = torch.zeros(nbytes, dtype=torch.uint8, device=_dev())  # zeroed once, before the first use
    _run_sequence(SEQUENCES[seq], lambda cs: cs.run_on(ws, nbytes))


@pytest.mark.parametrize("seq", ["fused-after-head-off", "fused-shrink-then-grow", "fused-after-chained"])
def test_static_scratch_across_shapes(seq):
    """The static-scratch entry point shares one array among every call of the process, so a
    change of shape between calls is its normal case."""
    _run_sequence(SEQUENCES[seq], lambda cs: cs.run_static())
