"""Failure detection on the GPU without a fault: a wait that can never be satisfied runs out.

The library's test hook (domino_debug_hold) makes one GRU CTA withhold what its peers wait for:
its hidden states of one position, or its arrival at the barrier of the state clear.  The
peers' bounded waits then expire (about a second each), every kernel of the step completes, the
device status reads DOMINO_ERR_TIMEOUT, and the next step on the same workspace is correct.
Nothing traps, asserts or hangs.
"""
import time

import pytest
import torch

from paper_2605_29707_gb300 import binding
from tests.test_gpu_workspace_reuse import _Case

pytestmark = pytest.mark.gpu


def _enqueue(cs, ws, nbytes):
    c = cs.c
    o = cs._outs()
    rc = binding.domino_draft_step(cs.hidden, cs.ids, cs.st.w["w_lm"], cs.st.head, c.B, c.K, c.H, c.V, c.k, c.N,
                                   o["topk_ids"], o["topk_logp"], o["tree_parent"], o["tree_token"],
                                   o["tree_depth"], o["tree_score"], ws, nbytes, torch.cuda.current_stream())
    assert rc == 0, binding.domino_status_string(rc)


@pytest.fixture
def disarm():
    yield
    assert binding.domino_debug_hold(binding.DOMINO_HOLD_OFF) == 0


# the fused small-batch GRU (no clear before the step), the chained one (cleared by the gather)
# and the large-M one (its own launch order)
@pytest.mark.parametrize("name,cta,pos", [("fused-big", 3, 2), ("fused-big", 0, 15), ("chained-B4", 1, 0),
                                          ("large-M", 2, 7)])
def test_withheld_state_times_out_then_next_step_is_correct(name, cta, pos, disarm):
    cs = _Case(name)
    nbytes = cs.ws_bytes()
    ws = torch.zeros(nbytes, dtype=torch.uint8, device=torch.device("cuda:0"))
    cs.check(cs.run_on(ws, nbytes))
    assert binding.domino_debug_hold(binding.DOMINO_HOLD_STATE, cta, pos) == 0
    t0 = time.perf_counter()
    _enqueue(cs, ws, nbytes)
    status = binding.domino_check_status(ws, torch.cuda.current_stream())
    elapsed = time.perf_counter() - t0
    assert status == binding.DOMINO_ERR_TIMEOUT, binding.domino_status_string(status)
    assert elapsed < 30.0
    # the hook held one launch only; the workspace serves the next steps unchanged
    cs.check(cs.run_on(ws, nbytes))
    cs.check(cs.run_on(ws, nbytes))


def test_withheld_clear_barrier_arrival_times_out(disarm):
    """A fresh workspace makes the fused step clear its state words behind a grid barrier; one CTA
    that never arrives makes every CTA give up, and the next step clears again and is correct."""
    cs = _Case("fused-big")
    nbytes = cs.ws_bytes()
    ws = torch.zeros(nbytes, dtype=torch.uint8, device=torch.device("cuda:0"))
    assert binding.domino_debug_hold(binding.DOMINO_HOLD_CLEAR_BARRIER, 5) == 0
    _enqueue(cs, ws, nbytes)
    status = binding.domino_check_status(ws, torch.cuda.current_stream())
    assert status == binding.DOMINO_ERR_TIMEOUT, binding.domino_status_string(status)
    cs.check(cs.run_on(ws, nbytes))
    cs.check(cs.run_on(ws, nbytes))


def test_hold_on_a_step_without_the_event_withholds_nothing(disarm):
    """A step that needs no clear (its workspace already holds its state range) has no barrier to
    withhold: it completes normally, and the hook, held for one launch, is gone after it."""
    cs = _Case("fused-big")
    nbytes = cs.ws_bytes()
    ws = torch.zeros(nbytes, dtype=torch.uint8, device=torch.device("cuda:0"))
    cs.check(cs.run_on(ws, nbytes))
    assert binding.domino_debug_hold(binding.DOMINO_HOLD_CLEAR_BARRIER, 5) == 0
    cs.check(cs.run_on(ws, nbytes))
    fresh = torch.zeros(nbytes, dtype=torch.uint8, device=torch.device("cuda:0"))
    cs.check(cs.run_on(fresh, nbytes))  # this one clears: the hook is no longer armed
