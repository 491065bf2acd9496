"""Seeded synthetic inputs for the Domino draft-side block step.

This module only draws numbers: Gaussian weights and hidden states rounded to
bf16, prefix token ids, and (for the serving-batch shape) a scale for the hidden
states.  It is shared by the tests, the smoke check and the benchmark so that the
CUDA path and the CPU oracle see the same bytes; it computes none of the step
itself and imports neither the CUDA binding nor the oracle.

Recipe (Qwen3-shaped, random-init; no checkpoint or dataset is used):
  * every weight ~ N(0, 0.02) drawn in fp32 and rounded to bf16 (round to nearest even);
  * each tensor has its own seeded generator keyed by (config seed, tensor name), drawn
    in fixed 2^24-element chunks so the bytes do not depend on the machine's thread count;
  * embedding row r is drawn from its own key (seed, "emb", r); rows that no prefix id
    references are left zero because neither side ever reads them;
  * biases are absent (zero) unless a test asks for them;
  * hidden states ~ N(0, 1); "rms1" rescales each row to RMS 1 before rounding;
    "entropy" multiplies by alpha, bisected so the mean entropy of the base
    distribution softmax(hidden . W_lm^T) over 8 rows is 3 nats;
  * prefix_ids[b, 0] (the anchor) is uniform in [0, V); for "sampled" configs
    prefix_ids[b, j >= 1] is drawn by inverse CDF from softmax of the base logits of
    position j - 1 (hidden . W_lm^T in fp32, normalised in fp64), standing in for the
    tokens an upstream sampler would have drafted.
"""
from __future__ import annotations

import concurrent.futures as _cf
import dataclasses
import functools
import hashlib
import math
import os

import numpy as np
import torch

DS_DEFAULT = 1024   # GRU hidden size d_s (paper, implementation details)
R_DEFAULT = 256     # correction rank r (paper, implementation details)
WSTD = 0.02
_CHUNK = 1 << 24


@dataclasses.dataclass(frozen=True)
class Config:
    name: str
    B: int
    K: int
    H: int
    V: int
    k: int
    N: int
    seed: int
    hidden_kind: str = "normal"      # normal | rms1 | entropy
    prefix_kind: str = "uniform"     # uniform | sampled
    seq_seed_base: int | None = None  # per-sequence seeds for hidden / prefix ids
    Ds: int = DS_DEFAULT
    R: int = R_DEFAULT
    biases: bool = False
    entropy_target: float = 3.0

    @property
    def M(self) -> int:
        return self.B * self.K


CONFIGS = {
    "tiny": Config("tiny", B=1, K=4, H=256, V=4096, k=4, N=8, seed=0),
    "qwen3-1.7b": Config("qwen3-1.7b", B=1, K=16, H=2048, V=151936, k=8, N=16, seed=1,
                         prefix_kind="sampled"),
    "qwen3-8b": Config("qwen3-8b", B=1, K=16, H=4096, V=151936, k=8, N=16, seed=2,
                       hidden_kind="rms1", prefix_kind="sampled"),
    "qwen3-8b-b32": Config("qwen3-8b-b32", B=32, K=16, H=4096, V=151936, k=8, N=16, seed=2,
                           hidden_kind="rms1", prefix_kind="sampled", seq_seed_base=2000),
    "qwen3-32b-b64": Config("qwen3-32b-b64", B=64, K=16, H=5120, V=151936, k=10, N=32, seed=3,
                            hidden_kind="entropy", prefix_kind="sampled"),
}


def _key_seed(*key) -> int:
    h = hashlib.blake2b(repr(key).encode(), digest_size=8).digest()
    return int.from_bytes(h, "little") & ((1 << 63) - 1)


def f32_to_bf16_bits(x: torch.Tensor) -> np.ndarray:
    """Round fp32 to bf16 (nearest even) and return the raw uint16 bit patterns."""
    return x.to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> torch.Tensor:
    t = torch.from_numpy(np.ascontiguousarray(b).view(np.int16))
    return t.view(torch.bfloat16).to(torch.float32)


def _normal_into(out: np.ndarray, key: tuple, std: float) -> None:
    flat = out.reshape(-1)
    n = flat.size
    nchunks = (n + _CHUNK - 1) // _CHUNK

    def work(c):
        lo = c * _CHUNK
        hi = min(n, lo + _CHUNK)
        g = torch.Generator().manual_seed(_key_seed(*key, c))
        x = torch.randn(hi - lo, generator=g, dtype=torch.float32)
        if std != 1.0:
            x.mul_(std)
        flat[lo:hi] = f32_to_bf16_bits(x)

    threads = max(1, min(nchunks, os.cpu_count() or 1))
    if nchunks == 1:
        work(0)
    else:
        with _cf.ThreadPoolExecutor(threads) as ex:
            list(ex.map(work, range(nchunks)))


def normal_bf16(shape, key: tuple, std: float = WSTD) -> np.ndarray:
    out = np.empty(shape, np.uint16)
    _normal_into(out, key, std)
    return out


def normal_f32(shape, key: tuple) -> torch.Tensor:
    g = torch.Generator().manual_seed(_key_seed(*key))
    return torch.randn(*shape, generator=g, dtype=torch.float32)


def uniform01(n: int, key: tuple) -> np.ndarray:
    g = torch.Generator().manual_seed(_key_seed(*key))
    return torch.rand(n, generator=g, dtype=torch.float64).numpy()


def randint(n: int, high: int, key: tuple) -> np.ndarray:
    g = torch.Generator().manual_seed(_key_seed(*key))
    return torch.randint(0, high, (n,), generator=g, dtype=torch.int64).numpy().astype(np.int32)


def emb_rows(cfg: Config, rows) -> np.ndarray:
    out = np.empty((len(rows), cfg.H), np.uint16)
    for i, r in enumerate(rows):
        out[i] = normal_bf16((cfg.H,), (cfg.seed, "emb", int(r)))
    return out


def _base_logits_f32(hid_bf16: np.ndarray, w_lm: np.ndarray, rows_per_block: int = 256,
                     vchunk: int = 16384) -> torch.Tensor:
    """hidden . W_lm^T in fp32, used only to shape the synthetic prefix ids."""
    x = bf16_bits_to_f32(hid_bf16.reshape(-1, hid_bf16.shape[-1]))
    V = w_lm.shape[0]
    z = torch.empty(x.shape[0], V, dtype=torch.float32)
    for v0 in range(0, V, vchunk):
        w = bf16_bits_to_f32(w_lm[v0:v0 + vchunk])
        for r0 in range(0, x.shape[0], rows_per_block):
            z[r0:r0 + rows_per_block, v0:v0 + vchunk] = x[r0:r0 + rows_per_block] @ w.T
    return z


def _sample_inverse_cdf(z_row: torch.Tensor, u: float) -> int:
    p = torch.softmax(z_row.to(torch.float64), dim=0)
    c = torch.cumsum(p, dim=0)
    idx = int(torch.searchsorted(c, torch.tensor([u * float(c[-1])], dtype=torch.float64)).item())
    return min(idx, z_row.numel() - 1)


def _entropy_nats(z: torch.Tensor) -> float:
    lp = torch.log_softmax(z.to(torch.float64), dim=-1)
    return float(-(lp.exp() * lp).sum(-1).mean())


@dataclasses.dataclass
class Workload:
    cfg: Config
    weights: dict          # name -> uint16 array or None
    hidden: np.ndarray     # uint16 [B, K, H]
    prefix_ids: np.ndarray  # int32 [B, K]
    alpha: float = 1.0

    @property
    def dims(self):
        c = self.cfg
        return dict(B=c.B, K=c.K, H=c.H, V=c.V, Ds=c.Ds, R=c.R, k=c.k, N=c.N)


def make_weights(cfg: Config) -> dict:
    H, V, Ds, R, s = cfg.H, cfg.V, cfg.Ds, cfg.R, cfg.seed
    w = {
        "w_lm": normal_bf16((V, H), (s, "w_lm")),
        "emb": None,  # filled once the prefix ids are known (rows by key)
        "w_ih": normal_bf16((3 * Ds, H), (s, "w_ih")) if R > 0 else None,
        "w_hh": normal_bf16((3 * Ds, Ds), (s, "w_hh")) if R > 0 else None,
        "b_ih": None, "b_hh": None, "b1": None, "b2": None,
        "w1": normal_bf16((R, H + Ds), (s, "w1")) if R > 0 else None,
        "w2": normal_bf16((V, R), (s, "w2")) if R > 0 else None,
    }
    if cfg.biases:
        w["b_ih"] = normal_bf16((3 * Ds,), (s, "b_ih"), 0.1) if R > 0 else None
        w["b_hh"] = normal_bf16((3 * Ds,), (s, "b_hh"), 0.1) if R > 0 else None
        w["b1"] = normal_bf16((R,), (s, "b1"), 0.1) if R > 0 else None
        w["b2"] = normal_bf16((V,), (s, "b2"), 0.1)
    return w


def _hidden_for(cfg: Config, key: tuple, rows: int, alpha: float) -> np.ndarray:
    x = normal_f32((rows, cfg.H), key)
    if cfg.hidden_kind == "rms1":
        x = x / torch.sqrt((x * x).mean(dim=1, keepdim=True))
    elif cfg.hidden_kind == "entropy":
        x = x * alpha
    return f32_to_bf16_bits(x)


def _calibrate_alpha(cfg: Config, w_lm: np.ndarray) -> float:
    x = normal_f32((8, cfg.H), (cfg.seed, "alpha-probe"))
    z1 = _base_logits_f32(f32_to_bf16_bits(x), w_lm).to(torch.float64)
    lo, hi = 0.05, 50.0
    for _ in range(40):
        mid = math.sqrt(lo * hi)
        if _entropy_nats(z1 * mid) > cfg.entropy_target:
            lo = mid
        else:
            hi = mid
    return math.sqrt(lo * hi)


def make_workload(cfg: Config | str, weights: dict | None = None) -> Workload:
    if isinstance(cfg, str):
        cfg = CONFIGS[cfg]
    w = dict(weights) if weights is not None else make_weights(cfg)
    B, K, V = cfg.B, cfg.K, cfg.V
    alpha = _calibrate_alpha(cfg, w["w_lm"]) if cfg.hidden_kind == "entropy" else 1.0

    hidden = np.empty((B, K, cfg.H), np.uint16)
    ids = np.empty((B, K), np.int32)
    if cfg.seq_seed_base is not None:
        for b in range(B):
            hidden[b] = _hidden_for(cfg, (cfg.seq_seed_base + b, "hidden"), K, alpha)
    else:
        hidden[:] = _hidden_for(cfg, (cfg.seed, "hidden"), B * K, alpha).reshape(B, K, cfg.H)

    def seq_key(b):
        return (cfg.seq_seed_base + b,) if cfg.seq_seed_base is not None else (cfg.seed, b)

    if cfg.prefix_kind == "uniform":
        for b in range(B):
            ids[b] = randint(K, V, (*seq_key(b), "prefix"))
    else:
        z = _base_logits_f32(hidden[:, :K - 1], w["w_lm"]).reshape(B, K - 1, V) if K > 1 else None
        for b in range(B):
            ids[b, 0] = randint(1, V, (*seq_key(b), "anchor"))[0]
            u = uniform01(K, (*seq_key(b), "prefix-u"))
            for j in range(1, K):
                ids[b, j] = _sample_inverse_cdf(z[b, j - 1], float(u[j]))

    if w.get("emb") is None and cfg.R > 0:
        emb = np.zeros((V, cfg.H), np.uint16)
        used = np.unique(ids)
        emb[used] = emb_rows(cfg, used)
        w["emb"] = emb
    return Workload(cfg, w, hidden, ids, alpha)


@functools.lru_cache(maxsize=2)
def cached_workload(name: str) -> Workload:
    return make_workload(CONFIGS[name])


def custom_config(name="custom", **kw) -> Config:
    base = dict(B=1, K=4, H=256, V=4096, k=4, N=8, seed=0)
    base.update(kw)
    return Config(name, **base)


# ---------------------------------------------------------------------------- verification inputs
@dataclasses.dataclass
class VerifyCase:
    """Synthetic inputs of greedy tree verification: a draft tree per sequence and the target's
    next-token logits after the anchor (row 0) and after each node (row i + 1)."""
    parent: np.ndarray  # int32 [B, N]
    token: np.ndarray   # int32 [B, N]
    target: np.ndarray  # float32 [B, N + 1, V]


def random_tree(N: int, V: int, key: tuple, chain: bool = False):
    """A valid draft tree of N nodes: parent[i] in [-1, i) (the previous node for a chain),
    tokens in [0, V) distinct among the children of one node."""
    g = torch.Generator().manual_seed(_key_seed(*key))
    parent = np.empty(N, np.int32)
    token = np.empty(N, np.int32)
    used = {}
    for i in range(N):
        p = i - 1 if chain else int(torch.randint(-1, i, (1,), generator=g)) if i > 0 else -1
        parent[i] = p
        taken = used.setdefault(p, set())
        while True:
            t = int(torch.randint(0, V, (1,), generator=g))
            if t not in taken:
                break
        taken.add(t)
        token[i] = t
    return parent, token


def make_verify_case(B: int, N: int, V: int, seed: int, p_plant: float = 0.7, chain: bool = False,
                     trees=None, margin: float = 1.0) -> VerifyCase:
    """Target logits ~ N(0, 1) fp32; with probability p_plant the row after a node (or after the
    anchor) gets one of that node's children's tokens raised to the row maximum + margin, so that
    accepted paths of every length occur (greedy: any margin > 0; sampled at T = 1 over 151936
    ids, margin 9 gives the planted token about two thirds of the mass).  `trees` ([B] pairs of
    parent/token) replaces the random trees, e.g. with trees a draft step produced."""
    parent = np.empty((B, N), np.int32)
    token = np.empty((B, N), np.int32)
    target = np.empty((B, N + 1, V), np.float32)
    for b in range(B):
        if trees is not None:
            parent[b], token[b] = trees[b]
        else:
            parent[b], token[b] = random_tree(N, V, (seed, "verify-tree", b), chain=chain)
        t = normal_f32((N + 1, V), (seed, "verify-target", b)).numpy()
        u = uniform01(2 * (N + 1), (seed, "verify-plant", b))
        for r in range(N + 1):
            kids = [c for c in range(N) if parent[b, c] == r - 1]
            if kids and u[2 * r] < p_plant:
                c = kids[min(len(kids) - 1, int(u[2 * r + 1] * len(kids)))]
                t[r, token[b, c]] = t[r].max() + margin
        target[b] = t
    return VerifyCase(parent, token, target)
