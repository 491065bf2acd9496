"""The host-buffer entry point (domino_draft_step_host) over consecutive calls on one set of buffers.

A call copies its inputs in, runs the step and copies every output back before it returns.
From the second call with the same buffers on, it replays a CUDA graph of the whole call (the
input copies, the step's kernels, the output copy).  These tests rewrite the inputs in place
between calls, so that a replay that did not read them afresh would show, and compare every
call with the device entry point on the same inputs and the first and last calls with the
oracle.  Pinned inputs take the graph; pageable ones may not be captured and run directly.
"""
import dataclasses

import numpy as np
import pytest
import torch

from paper_2605_29707_gb300 import binding, inputs
from paper_2605_29707_gb300.step import DraftStep
from tests.test_gpu_parity import _check

pytestmark = pytest.mark.gpu

INT_KEYS = ("topk_ids", "tree_parent", "tree_token", "tree_depth")
FLOAT_KEYS = ("topk_logp", "tree_score")
CONFIGS = {
    "tiny": inputs.CONFIGS["tiny"],
    # more than 128 tokens: the non-fused launch sequence (clear, gather, projections, GRU, ...)
    "host-m160": inputs.custom_config("host-m160", B=10, K=16, H=192, V=3001, Ds=64, R=64, k=8, N=16, seed=71,
                                      biases=True),
}


def _variant(wl, i):
    """Call i's inputs: the workload's hidden states rolled by i positions and its prefix ids
    shifted by 37 i (mod V); the same shapes with other values on every call."""
    c = wl.cfg
    hidden = np.ascontiguousarray(np.roll(wl.hidden, i, axis=1))
    ids = np.ascontiguousarray(((wl.prefix_ids.astype(np.int64) + 37 * i) % c.V).astype(np.int32))
    return dataclasses.replace(wl, hidden=hidden, prefix_ids=ids)


def _host_buffers(c, pinned):
    def empty(shape, dt):
        return torch.empty(shape, dtype=dt, pin_memory=pinned)
    h_hidden = empty((c.B, c.K, c.H), torch.int16)  # bf16 bit patterns
    h_ids = empty((c.B, c.K), torch.int32)
    out = {"topk_ids": empty((c.B, c.K, c.k), torch.int32), "topk_logp": empty((c.B, c.K, c.k), torch.float32),
           "tree_parent": empty((c.B, c.N), torch.int32), "tree_token": empty((c.B, c.N), torch.int32),
           "tree_depth": empty((c.B, c.N), torch.int32), "tree_score": empty((c.B, c.N), torch.float32)}
    return h_hidden, h_ids, out


def _device_ref(ref_st, wl_i):
    dev = torch.device("cuda:0")
    hidden = torch.from_numpy(wl_i.hidden.view(np.int16)).view(torch.bfloat16).to(dev)
    ids = torch.from_numpy(wl_i.prefix_ids).to(dev)
    return ref_st.run(hidden, ids)


def _same(out, ref):
    for key in INT_KEYS:
        np.testing.assert_array_equal(out[key].numpy(), ref[key], err_msg=key)
    for key in FLOAT_KEYS:
        np.testing.assert_allclose(out[key].numpy(), ref[key], atol=1e-6, rtol=0, err_msg=key)


@pytest.mark.parametrize("name,pinned", [("tiny", True), ("host-m160", True), ("tiny", False)])
def test_host_entry_consecutive_calls(name, pinned):
    wl = inputs.make_workload(CONFIGS[name])
    c = wl.cfg
    dev = torch.device("cuda:0")
    st = DraftStep(wl.weights, c.B, c.K, c.H, c.V, c.k, c.N, Ds=c.Ds, R=c.R, device=dev)
    ref_st = DraftStep(wl.weights, c.B, c.K, c.H, c.V, c.k, c.N, Ds=c.Ds, R=c.R, device=dev)
    h_hidden, h_ids, out = _host_buffers(c, pinned)
    calls = 4
    for i in range(calls):
        wl_i = _variant(wl, i)
        h_hidden.copy_(torch.from_numpy(wl_i.hidden.view(np.int16)))
        h_ids.copy_(torch.from_numpy(wl_i.prefix_ids))
        for v in out.values():
            v.fill_(-7)
        rc = st.run_host(h_hidden, h_ids, out)
        assert rc == 0, (i, binding.domino_status_string(rc))
        _same(out, _device_ref(ref_st, wl_i))
        if i in (0, calls - 1):
            got = {k: v.numpy() for k, v in out.items()}
            ex_topk, ex_tree = _check(wl_i, got)
            assert ex_topk <= max(1, c.M * c.k // 50)
            assert ex_tree <= max(1, c.B * c.N // 10)


@pytest.mark.parametrize("name", ["tiny", "host-m160"])
def test_host_entry_bad_token_on_a_replayed_call(name):
    """A bad prefix id on a call that replays the graph comes back as DOMINO_ERR_BAD_TOKEN, and
    the next call (good ids again) is correct."""
    wl = inputs.make_workload(CONFIGS[name])
    c = wl.cfg
    dev = torch.device("cuda:0")
    st = DraftStep(wl.weights, c.B, c.K, c.H, c.V, c.k, c.N, Ds=c.Ds, R=c.R, device=dev)
    ref_st = DraftStep(wl.weights, c.B, c.K, c.H, c.V, c.k, c.N, Ds=c.Ds, R=c.R, device=dev)
    h_hidden, h_ids, out = _host_buffers(c, True)
    h_hidden.copy_(torch.from_numpy(wl.hidden.view(np.int16)))
    for i in range(4):
        ids = wl.prefix_ids.copy()
        if i == 2:
            ids[c.B - 1, c.K - 1] = c.V
        h_ids.copy_(torch.from_numpy(ids))
        rc = st.run_host(h_hidden, h_ids, out)
        if i == 2:
            assert rc == binding.DOMINO_ERR_BAD_TOKEN
        else:
            assert rc == 0, (i, binding.domino_status_string(rc))
    _same(out, _device_ref(ref_st, wl))
