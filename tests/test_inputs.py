"""The seeded input generator (CPU): the same seed gives the same bytes, whatever the machine's
thread count; named streams are independent; bf16 rounding is to nearest even; the recipe's
properties (RMS-1 rows, ids in range, embedding rows only where a prefix id names them)."""
import numpy as np
import torch

from paper_2605_29707_gb300 import inputs


def test_same_seed_same_bytes():
    a = inputs.make_workload(inputs.CONFIGS["tiny"])
    b = inputs.make_workload(inputs.CONFIGS["tiny"])
    for name, w in a.weights.items():
        if w is None:
            assert b.weights[name] is None
        else:
            np.testing.assert_array_equal(w, b.weights[name])
    np.testing.assert_array_equal(a.hidden, b.hidden)
    np.testing.assert_array_equal(a.prefix_ids, b.prefix_ids)


def test_chunks_are_seeded_by_key_and_index_not_by_thread_count(monkeypatch):
    """A tensor of two chunks (the chunk size shrunk from 2^24 to 4096 for the test): chunk 0
    equals a one-chunk draw with the same key and chunk 1 the first values of the generator keyed
    (key, 1), with one thread or many."""
    monkeypatch.setattr(inputs, "_CHUNK", 4096)
    key = (7, "chunk-test")
    n_tail = 1000
    old = torch.get_num_threads()
    try:
        torch.set_num_threads(1)
        one = inputs.normal_bf16((inputs._CHUNK + n_tail,), key)
        torch.set_num_threads(max(2, old))
        many = inputs.normal_bf16((inputs._CHUNK + n_tail,), key)
    finally:
        torch.set_num_threads(old)
    np.testing.assert_array_equal(one, many)
    head = inputs.normal_bf16((inputs._CHUNK,), key)
    np.testing.assert_array_equal(one[:inputs._CHUNK], head)
    g = torch.Generator().manual_seed(inputs._key_seed(*key, 1))
    tail = inputs.f32_to_bf16_bits(torch.randn(n_tail, generator=g, dtype=torch.float32).mul_(inputs.WSTD))
    np.testing.assert_array_equal(one[inputs._CHUNK:], tail)


def test_named_streams_are_independent():
    a = inputs.normal_bf16((4096,), (0, "w_lm"))
    b = inputs.normal_bf16((4096,), (0, "w2"))
    c = inputs.normal_bf16((4096,), (1, "w_lm"))
    assert (a != b).mean() > 0.9 and (a != c).mean() > 0.9


def test_bf16_rounding_is_to_nearest_even():
    x = torch.tensor([1.0 + 2.0 ** -8, 1.0 + 3 * 2.0 ** -8, -(1.0 + 2.0 ** -8), 1.0 + 2.0 ** -8 + 2.0 ** -20])
    bits = inputs.f32_to_bf16_bits(x)
    # halfway cases go to the even mantissa; just above halfway rounds up
    assert list(bits) == [0x3F80, 0x3F82, 0xBF80, 0x3F81]
    back = inputs.bf16_bits_to_f32(bits)
    assert back.tolist() == [1.0, 1.015625, -1.0, 1.0078125]


def test_recipe_properties():
    cfg = inputs.custom_config("recipe", B=3, K=5, H=512, V=3000, Ds=32, R=16, seed=9, hidden_kind="rms1",
                               prefix_kind="sampled")
    wl = inputs.make_workload(cfg)
    h = inputs.bf16_bits_to_f32(wl.hidden.reshape(-1, cfg.H)).double()
    rms = h.pow(2).mean(dim=1).sqrt()
    assert torch.allclose(rms, torch.ones_like(rms), atol=1e-2)
    ids = wl.prefix_ids
    assert ids.dtype == np.int32 and ids.shape == (3, 5) and ids.min() >= 0 and ids.max() < cfg.V
    emb = wl.weights["emb"]
    used = np.unique(ids)
    assert (emb[used] != 0).any(axis=1).all()
    unused = np.setdiff1d(np.arange(cfg.V), used)
    assert not emb[unused].any()
