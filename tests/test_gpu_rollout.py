"""The greedy sequential draft loop on the GPU (domino_rollout_greedy) against the oracle.

Section 4.1.2 / Fig. 3: at inference each draft token is chosen from the final logits and fed
back to the causal encoder.  The argmax decisions are taken in fp32 on the GPU and in fp64 in the
oracle, so where the oracle's two best log-probabilities are within the parity tolerance either
choice is correct (and the rest of the rollout then follows that choice).  The check therefore
runs the oracle's draft step teacher-forced on the GPU's own tokens: every GPU token must be a
valid greedy choice there (within 4e-2 of the position's best log-probability) with the GPU's
log-probability within 2e-2; and up to the first such near-tie the GPU tokens must equal the
oracle rollout's exactly.
"""
import ctypes
import dataclasses
import functools

import numpy as np
import pytest
import torch

import oracle
from paper_2605_29707_gb300 import binding, inputs

pytestmark = pytest.mark.gpu

LOGP_TOL = 2e-2
GAP = 4e-2


def _full_emb(wl):
    """The workload with every embedding row drawn.  The generator leaves the rows no prefix id
    names at zero, but a rollout feeds back tokens of its own choosing, so here every row is
    live and every step's GRU input is a real embedding."""
    c = wl.cfg
    w = dict(wl.weights)
    w["emb"] = inputs.normal_bf16((c.V, c.H), (c.seed, "emb-all"))
    return dataclasses.replace(wl, weights=w)


@functools.lru_cache(maxsize=2)
def _full_size(name):
    return _full_emb(inputs.cached_workload(name))


def _device_weights(wl, dev, head_on=True, table=False):
    """Device weights and the head struct; table=True also builds the input-projection table
    (kept alive in w["x_table"]) and points the head at it."""
    w = {n: torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16).to(dev)
         for n, a in wl.weights.items() if a is not None}
    c = wl.cfg
    x_table = None
    if table:
        x_table = torch.empty(binding.domino_input_table_bytes(c.V, c.Ds) // 4, dtype=torch.float32, device=dev)
        rc = binding.domino_build_input_table(w["emb"], w["w_ih"], c.V, c.H, c.Ds, x_table,
                                              torch.cuda.current_stream(dev))
        assert rc == 0, binding.domino_status_string(rc)
        w["x_table"] = x_table
    head = binding.make_head(w.get("emb"), w.get("w_ih"), w.get("w_hh"), w.get("b_ih"), w.get("b_hh"), w.get("w1"),
                             w.get("b1"), w.get("w2") if head_on else None, w.get("b2"), c.Ds if head_on else 0,
                             c.R if head_on else 0, x_table)
    return w, head


def _run_gpu(wl, head_on=True, table=False):
    c = wl.cfg
    dev = torch.device("cuda:0")
    w, head = _device_weights(wl, dev, head_on, table)
    hidden = torch.from_numpy(wl.hidden.view(np.int16)).view(torch.bfloat16).to(dev)
    anchors = torch.from_numpy(np.ascontiguousarray(wl.prefix_ids[:, 0])).to(dev)
    nbytes = binding.domino_rollout_workspace_bytes(c.B, c.K, c.H, c.V, c.Ds if head_on else 0, c.R if head_on else 0)
    assert nbytes > 0
    ws = torch.empty(nbytes, dtype=torch.uint8, device=dev)
    tokens = torch.full((c.B, c.K), -7, dtype=torch.int32, device=dev)
    logp = torch.full((c.B, c.K), 7.0, dtype=torch.float32, device=dev)
    s = torch.cuda.current_stream(dev)
    rc = binding.domino_rollout_greedy(hidden, anchors, w["w_lm"], head, c.B, c.K, c.H, c.V, tokens, logp,
                                       ws, nbytes, s)
    assert rc == 0, binding.domino_status_string(rc)
    assert binding.domino_check_status(ws, s) == 0
    return tokens.cpu().numpy(), logp.cpu().numpy()


def _check(wl, head_on=True, table=False):
    c = wl.cfg
    w = wl.weights if head_on else {"w_lm": wl.weights["w_lm"], "b2": wl.weights.get("b2")}
    tokens, logp = _run_gpu(wl, head_on, table)
    anchors = np.ascontiguousarray(wl.prefix_ids[:, 0]).astype(np.int32)
    o_tok, _ = oracle.rollout_greedy(w, wl.hidden, anchors)
    excused = 0
    for b in range(c.B):
        prefix = np.concatenate([[anchors[b]], tokens[b, :-1]]).astype(np.int32)[None, :]
        ref = oracle.draft_step(w, wl.hidden[b:b + 1], prefix, 1, 1, want_logp_full=True)
        lp = ref["logp_full"][0]
        same = True
        for j in range(c.K):
            t = int(tokens[b, j])
            assert 0 <= t < c.V
            best = float(lp[j].max())
            assert lp[j, t] >= best - GAP, (b, j, t, lp[j, t], best)
            assert abs(float(logp[b, j]) - lp[j, t]) <= LOGP_TOL, (b, j, logp[b, j], lp[j, t])
            if same:
                top2 = np.partition(lp[j], -2)[-2:]
                if abs(top2[1] - top2[0]) > GAP:
                    assert t == int(o_tok[b, j]), (b, j, t, o_tok[b, j])
                elif t != int(o_tok[b, j]):
                    excused += 1
                    same = False  # the rollouts follow different, equally valid tokens from here
    return excused


@pytest.mark.parametrize("cfg", [
    inputs.CONFIGS["tiny"],
    inputs.custom_config("roll-b3", B=3, K=8, H=512, V=3000, Ds=64, R=64, seed=21, biases=True),
    inputs.custom_config("roll-b8", B=8, K=5, H=256, V=1000, Ds=32, R=16, seed=22),
    inputs.custom_config("roll-k1", B=2, K=1, H=128, V=777, Ds=16, R=8, seed=23),
    # r > 256: W2 streamed through the shared-memory ring every step
    inputs.custom_config("roll-wide", B=2, K=4, H=256, V=2500, Ds=32, R=512, seed=26, biases=True),
    # r = 256 at a vocabulary past 152 x 1024 rows: every CTA's slice spans tensor memory, shared
    # memory and rows read through L2, with a ragged last slice
    inputs.custom_config("roll-tiers", B=8, K=3, H=256, V=167001, Ds=32, R=256, seed=27),
    inputs.custom_config("roll-tiers-b1", B=1, K=4, H=256, V=160003, Ds=32, R=256, seed=28, biases=True),
])
def test_rollout_matches_oracle(cfg):
    _check(_full_emb(inputs.make_workload(cfg)))


@pytest.mark.parametrize("cfg", [
    inputs.CONFIGS["tiny"],
    inputs.custom_config("roll-b3", B=3, K=8, H=512, V=3000, Ds=64, R=64, seed=21, biases=True),
    inputs.custom_config("roll-wide", B=2, K=4, H=256, V=2500, Ds=32, R=512, seed=26, biases=True),
    inputs.custom_config("roll-tiers-b1", B=1, K=4, H=256, V=160003, Ds=32, R=256, seed=28, biases=True),
])
def test_rollout_with_input_table_matches_oracle(cfg):
    """Phase A's input-gate sums read from the table emb . W_ih^T: the same rollout."""
    _check(_full_emb(inputs.make_workload(cfg)), table=True)


# Phase C on the tensor cores (the table's two-barrier step, B <= 2, r a multiple of 64 up to 256):
# W2 blocks of 128 rows in tensor memory only (small vocabularies), in tensor and shared memory
# (r = 128 and 256), and with the rows past those blocks read through L2 (V past 152 x 768).
MMA_CASES = [
    inputs.custom_config("mma-r64", B=1, K=6, H=256, V=5000, Ds=64, R=64, seed=51, biases=True),
    inputs.custom_config("mma-r128-b2", B=2, K=4, H=256, V=160003, Ds=64, R=128, seed=52),
    inputs.custom_config("mma-r256-b2", B=2, K=4, H=256, V=160003, Ds=32, R=256, seed=53, biases=True),
    inputs.custom_config("mma-r192-b1", B=1, K=3, H=128, V=120007, Ds=32, R=192, seed=54),
]


@pytest.mark.parametrize("cfg", MMA_CASES)
def test_rollout_tensor_core_phase_c_matches_oracle(cfg):
    _check(_full_emb(inputs.make_workload(cfg)), table=True)


def test_rollout_head_off():
    _check(inputs.make_workload(inputs.custom_config("roll-off", B=2, K=6, H=256, V=2000, seed=24)), head_on=False)


def test_rollout_rejects_bad_anchor_and_sizes():
    wl = inputs.make_workload(inputs.custom_config("roll-bad", B=1, K=3, H=128, V=500, Ds=16, R=8, seed=25))
    c = wl.cfg
    dev = torch.device("cuda:0")
    w, head = _device_weights(wl, dev)
    hidden = torch.from_numpy(wl.hidden.view(np.int16)).view(torch.bfloat16).to(dev)
    nbytes = binding.domino_rollout_workspace_bytes(c.B, c.K, c.H, c.V, c.Ds, c.R)
    ws = torch.empty(nbytes, dtype=torch.uint8, device=dev)
    tokens = torch.empty((1, 3), dtype=torch.int32, device=dev)
    logp = torch.empty((1, 3), dtype=torch.float32, device=dev)
    bad = torch.tensor([c.V], dtype=torch.int32, device=dev)
    s = torch.cuda.current_stream(dev)
    assert binding.domino_rollout_greedy(hidden, bad, w["w_lm"], head, 1, 3, c.H, c.V, tokens, logp, ws,
                                         nbytes, s) == 0
    assert binding.domino_check_status(ws, s) == binding.DOMINO_ERR_BAD_TOKEN
    assert binding.domino_rollout_greedy(hidden, bad, w["w_lm"], head, 1, 3, c.H, c.V, tokens, logp, ws,
                                         nbytes - 256, s) == binding.DOMINO_ERR_INVALID_ARG
    assert binding.domino_rollout_workspace_bytes(9, 3, c.H, c.V, c.Ds, c.R) == 0
    # token ids must fit the greedy argmax key's 22 bits
    assert binding.domino_rollout_workspace_bytes(1, 3, c.H, 1 << 22, c.Ds, c.R) == 0


@pytest.mark.parametrize("name", ["qwen3-8b", "qwen3-1.7b"])
def test_rollout_full_size(name):
    _check(_full_size(name))


def test_rollout_full_size_with_input_table():
    _check(_full_size("qwen3-8b"), table=True)


# ---------------------------------------------------------------------------- input table
def _table_case(wl, rows):
    """GPU table rows against the fp64 product of the same bf16 values, within the fp32
    summation bound gamma_H = H u / (1 - H u) (u = 2^-24) times sum_h |emb[t, h] W_ih[g, h]|
    (bf16 x bf16 products are exact in fp32)."""
    c = wl.cfg
    dev = torch.device("cuda:0")
    w, _ = _device_weights(wl, dev, True, table=True)
    tab = w["x_table"].view(c.V, 3 * c.Ds)
    got = tab[torch.from_numpy(rows).to(dev).long()].cpu().numpy().astype(np.float64)
    emb = inputs.bf16_bits_to_f32(wl.weights["emb"][rows]).numpy().astype(np.float64)
    wih = inputs.bf16_bits_to_f32(wl.weights["w_ih"]).numpy().astype(np.float64)
    ref = emb @ wih.T
    mag = np.abs(emb) @ np.abs(wih).T
    u = 2.0 ** -24
    gamma = c.H * u / (1 - c.H * u)
    err = np.abs(got - ref)
    assert (err <= gamma * mag + 1e-30).all(), float((err - gamma * mag).max())


@pytest.mark.parametrize("cfg", [
    # a ragged last 128-token tile and 3 Ds = 72 gate rows (a ragged 256-row tile)
    inputs.custom_config("tab-ragged", B=1, K=2, H=256, V=1000, Ds=24, R=8, seed=41),
    inputs.custom_config("tab-mid", B=1, K=2, H=512, V=3001, Ds=64, R=16, seed=42, biases=True),
])
def test_input_table_matches_product(cfg):
    wl = _full_emb(inputs.make_workload(cfg))
    _table_case(wl, np.arange(cfg.V, dtype=np.int64))


def test_input_table_full_size_sampled_rows():
    wl = _full_size("qwen3-8b")
    rows = np.unique(np.concatenate([[0, 1, wl.cfg.V - 1],
                                     np.random.default_rng(3).integers(0, wl.cfg.V, 61)])).astype(np.int64)
    _table_case(wl, rows)


# ---------------------------------------------------------------------------- sampled loop
CDF_TOL = 5e-3  # fp32 logits and sums on the GPU against fp64: how far u may sit past a boundary


def _run_gpu_sample(wl, uniforms, head_on=True, table=False):
    c = wl.cfg
    dev = torch.device("cuda:0")
    w, head = _device_weights(wl, dev, head_on, table)
    hidden = torch.from_numpy(wl.hidden.view(np.int16)).view(torch.bfloat16).to(dev)
    anchors = torch.from_numpy(np.ascontiguousarray(wl.prefix_ids[:, 0])).to(dev)
    uni = torch.from_numpy(uniforms).to(dev)
    nbytes = binding.domino_rollout_workspace_bytes(c.B, c.K, c.H, c.V, c.Ds if head_on else 0, c.R if head_on else 0)
    ws = torch.empty(nbytes, dtype=torch.uint8, device=dev)
    tokens = torch.full((c.B, c.K), -7, dtype=torch.int32, device=dev)
    logp = torch.full((c.B, c.K), 7.0, dtype=torch.float32, device=dev)
    s = torch.cuda.current_stream(dev)
    rc = binding.domino_rollout_sample(hidden, anchors, uni, w["w_lm"], head, c.B, c.K, c.H, c.V, tokens, logp, ws,
                                       nbytes, s)
    assert rc == 0, binding.domino_status_string(rc)
    assert binding.domino_check_status(ws, s) == 0
    return tokens.cpu().numpy(), logp.cpu().numpy()


def _check_sample(wl, head_on=True, seed=5, table=False):
    """Teacher-forced: every GPU token's cumulative-probability interval (under the oracle's step
    fed the GPU's own tokens) holds its uniform within CDF_TOL, with logp within LOGP_TOL; up to
    the first uniform within CDF_TOL of one of the oracle rollout's boundaries, the tokens equal
    the oracle rollout's."""
    c = wl.cfg
    w = wl.weights if head_on else {"w_lm": wl.weights["w_lm"], "b2": wl.weights.get("b2")}
    uni = np.random.default_rng(seed).random((c.B, c.K), dtype=np.float32)
    tokens, logp = _run_gpu_sample(wl, uni, head_on, table)
    anchors = np.ascontiguousarray(wl.prefix_ids[:, 0]).astype(np.int32)
    o_tok, _ = oracle.rollout_sample(w, wl.hidden, anchors, uni)
    excused = 0
    for b in range(c.B):
        prefix = np.concatenate([[anchors[b]], tokens[b, :-1]]).astype(np.int32)[None, :]
        ref = oracle.draft_step(w, wl.hidden[b:b + 1], prefix, 1, 1, want_logp_full=True)
        same = True
        for j in range(c.K):
            lp = ref["logp_full"][0, j]
            cdf = np.cumsum(np.exp(lp))
            t = int(tokens[b, j])
            assert 0 <= t < c.V
            lo = cdf[t - 1] if t > 0 else 0.0
            u = float(uni[b, j])
            assert lo - CDF_TOL <= u <= cdf[t] + CDF_TOL, (b, j, t, lo, u, cdf[t])
            assert abs(float(logp[b, j]) - lp[t]) <= LOGP_TOL, (b, j, logp[b, j], lp[t])
            if same:
                ot = int(o_tok[b, j])
                olo = cdf[ot - 1] if ot > 0 else 0.0
                if min(u - olo, cdf[ot] - u) > CDF_TOL:
                    assert t == ot, (b, j, t, ot)
                elif t != ot:
                    excused += 1
                    same = False
    return excused


@pytest.mark.parametrize("cfg", [
    inputs.CONFIGS["tiny"],
    inputs.custom_config("samp-b3", B=3, K=8, H=512, V=3000, Ds=64, R=64, seed=31, biases=True),
    inputs.custom_config("samp-b8", B=8, K=5, H=256, V=1000, Ds=32, R=16, seed=32),
    inputs.custom_config("samp-wide", B=2, K=4, H=256, V=2500, Ds=32, R=512, seed=33, biases=True),
    inputs.custom_config("samp-tiers", B=8, K=3, H=256, V=167001, Ds=32, R=256, seed=34),
])
def test_rollout_sample_matches_oracle(cfg):
    _check_sample(_full_emb(inputs.make_workload(cfg)))


@pytest.mark.parametrize("cfg", [
    inputs.custom_config("samp-b3", B=3, K=8, H=512, V=3000, Ds=64, R=64, seed=31, biases=True),
    inputs.custom_config("samp-tiers", B=8, K=3, H=256, V=167001, Ds=32, R=256, seed=34),
])
def test_rollout_sample_with_input_table_matches_oracle(cfg):
    _check_sample(_full_emb(inputs.make_workload(cfg)), table=True)


@pytest.mark.parametrize("cfg", [MMA_CASES[0], MMA_CASES[1], MMA_CASES[2]])
def test_rollout_sample_tensor_core_phase_c_matches_oracle(cfg):
    _check_sample(_full_emb(inputs.make_workload(cfg)), seed=9, table=True)


def test_rollout_sample_head_off():
    _check_sample(inputs.make_workload(inputs.custom_config("samp-off", B=2, K=6, H=256, V=2000, seed=35)),
                  head_on=False)


@pytest.mark.parametrize("name", ["qwen3-8b"])
def test_rollout_sample_full_size(name):
    _check_sample(_full_size(name), seed=7)


def test_rollout_sample_full_size_with_input_table():
    _check_sample(_full_size("qwen3-8b"), seed=8, table=True)


def test_rollout_sample_uniform_ends_and_bad_pointer():
    """u = 0 takes the first id of non-zero probability (id 0 here), and a misaligned uniforms
    pointer is refused before anything is enqueued."""
    wl = inputs.make_workload(inputs.custom_config("samp-ends", B=2, K=3, H=128, V=700, Ds=16, R=8, seed=36))
    c = wl.cfg
    uni = np.zeros((c.B, c.K), np.float32)
    tokens, _ = _run_gpu_sample(wl, uni)
    assert (tokens == 0).all()
    dev = torch.device("cuda:0")
    w, head = _device_weights(wl, dev)
    hidden = torch.from_numpy(wl.hidden.view(np.int16)).view(torch.bfloat16).to(dev)
    anchors = torch.from_numpy(np.ascontiguousarray(wl.prefix_ids[:, 0])).to(dev)
    raw = torch.zeros(c.B * c.K + 1, dtype=torch.float32, device=dev)
    nbytes = binding.domino_rollout_workspace_bytes(c.B, c.K, c.H, c.V, c.Ds, c.R)
    ws = torch.empty(nbytes, dtype=torch.uint8, device=dev)
    out_t = torch.empty((c.B, c.K), dtype=torch.int32, device=dev)
    out_l = torch.empty((c.B, c.K), dtype=torch.float32, device=dev)
    bad = raw.data_ptr() + 2  # not 4-byte aligned
    f = binding.load().domino_rollout_sample
    h = ctypes.byref(head)
    assert f(hidden.data_ptr(), anchors.data_ptr(), bad, w["w_lm"].data_ptr(), h, c.B, c.K, c.H, c.V,
             out_t.data_ptr(), out_l.data_ptr(), ws.data_ptr(), nbytes, None) == binding.DOMINO_ERR_INVALID_ARG


# ---------------------------------------------------------------------------- exponential race
def _run_gpu_gumbel(wl, seed, head_on=True, table=False):
    c = wl.cfg
    dev = torch.device("cuda:0")
    w, head = _device_weights(wl, dev, head_on, table)
    hidden = torch.from_numpy(wl.hidden.view(np.int16)).view(torch.bfloat16).to(dev)
    anchors = torch.from_numpy(np.ascontiguousarray(wl.prefix_ids[:, 0])).to(dev)
    nbytes = binding.domino_rollout_workspace_bytes(c.B, c.K, c.H, c.V, c.Ds if head_on else 0, c.R if head_on else 0)
    ws = torch.empty(nbytes, dtype=torch.uint8, device=dev)
    tokens = torch.full((c.B, c.K), -7, dtype=torch.int32, device=dev)
    logp = torch.full((c.B, c.K), 7.0, dtype=torch.float32, device=dev)
    s = torch.cuda.current_stream(dev)
    rc = binding.domino_rollout_sample_gumbel(hidden, anchors, seed, w["w_lm"], head, c.B, c.K, c.H, c.V, tokens,
                                              logp, ws, nbytes, s)
    assert rc == 0, binding.domino_status_string(rc)
    assert binding.domino_check_status(ws, s) == 0
    return tokens.cpu().numpy(), logp.cpu().numpy()


def _check_gumbel(wl, seed, head_on=True, table=False):
    """Teacher-forced, as _check with the perturbed log-probabilities: at every position, under
    the oracle's step fed the GPU's own tokens, the GPU token's log-probability plus the oracle's
    perturbation of that sequence, step and token is within GAP of the largest such sum, the
    GPU's logp within LOGP_TOL of the token's log-probability; up to the first position whose two
    largest sums are within GAP the tokens equal the oracle rollout's.  (The perturbations are a
    function of (seed, sequence, step, token) alone, so a rollout that took another, equally
    valid token keeps the same perturbations for the steps after it.)"""
    c = wl.cfg
    w = wl.weights if head_on else {"w_lm": wl.weights["w_lm"], "b2": wl.weights.get("b2")}
    tokens, logp = _run_gpu_gumbel(wl, seed, head_on, table)
    anchors = np.ascontiguousarray(wl.prefix_ids[:, 0]).astype(np.int32)
    o_tok, _ = oracle.rollout_sample_gumbel(w, wl.hidden, anchors, seed)
    excused = 0
    for b in range(c.B):
        prefix = np.concatenate([[anchors[b]], tokens[b, :-1]]).astype(np.int32)[None, :]
        ref = oracle.draft_step(w, wl.hidden[b:b + 1], prefix, 1, 1, want_logp_full=True)
        lp = ref["logp_full"][0]
        same = True
        for j in range(c.K):
            t = int(tokens[b, j])
            assert 0 <= t < c.V
            key = lp[j] + oracle.gumbel_row(seed, b, j, c.V)
            best = float(key.max())
            assert key[t] >= best - GAP, (b, j, t, key[t], best)
            assert abs(float(logp[b, j]) - lp[j, t]) <= LOGP_TOL, (b, j, logp[b, j], lp[j, t])
            if same:
                top2 = np.partition(key, -2)[-2:]
                if abs(top2[1] - top2[0]) > GAP:
                    assert t == int(o_tok[b, j]), (b, j, t, o_tok[b, j])
                elif t != int(o_tok[b, j]):
                    excused += 1
                    same = False
    return excused


@pytest.mark.parametrize("cfg", [
    inputs.CONFIGS["tiny"],
    inputs.custom_config("race-b3", B=3, K=8, H=512, V=3000, Ds=64, R=64, seed=61, biases=True),
    inputs.custom_config("race-b8", B=8, K=5, H=256, V=1000, Ds=32, R=16, seed=62),
    inputs.custom_config("race-b5", B=5, K=4, H=256, V=2000, Ds=32, R=32, seed=63),
    # r > 256: the streamed kernel
    inputs.custom_config("race-wide", B=6, K=4, H=256, V=2500, Ds=32, R=512, seed=64, biases=True),
    # tensor-memory, shared-memory and L2 rows of W2 in every CTA, a ragged last slice
    inputs.custom_config("race-tiers", B=8, K=3, H=256, V=167001, Ds=32, R=256, seed=65),
])
def test_rollout_sample_gumbel_matches_oracle(cfg):
    _check_gumbel(_full_emb(inputs.make_workload(cfg)), seed=0x9E3779B97F4A7C15)


@pytest.mark.parametrize("cfg", [MMA_CASES[0], MMA_CASES[1], MMA_CASES[2], MMA_CASES[3]])
def test_rollout_sample_gumbel_tensor_core_phase_c_matches_oracle(cfg):
    _check_gumbel(_full_emb(inputs.make_workload(cfg)), seed=12345, table=True)


def test_rollout_sample_gumbel_head_off():
    _check_gumbel(inputs.make_workload(inputs.custom_config("race-off", B=6, K=6, H=256, V=2000, seed=66)), seed=3,
                  head_on=False)


def test_rollout_sample_gumbel_full_size():
    _check_gumbel(_full_size("qwen3-8b"), seed=2026)


def test_rollout_sample_gumbel_full_size_with_input_table():
    _check_gumbel(_full_size("qwen3-8b"), seed=2027, table=True)


def test_rollout_sample_gumbel_seed_is_the_draw():
    """The same seed draws the same tokens and log-probabilities; a seed that differs in its high
    word only draws other tokens."""
    wl = _full_emb(inputs.make_workload(inputs.custom_config("race-seed", B=2, K=6, H=128, V=700, Ds=16, R=8,
                                                             seed=67)))
    a, la = _run_gpu_gumbel(wl, 1 << 40)
    b, lb = _run_gpu_gumbel(wl, 1 << 40)
    assert (a == b).all() and np.array_equal(la, lb)
    c, _ = _run_gpu_gumbel(wl, (1 << 40) + (1 << 33))
    assert (a != c).any()
