"""Seeded synthetic inputs for the SPSA step: byte batches and parameters.

This module holds none of the method's arithmetic.  It only produces inputs
(numpy arrays on the host) that both the CUDA path and the fp64 oracle consume
unchanged, so it imports neither of them.

Byte batches stand in for the paper's clustered FineWeb-Edu shards (Sec. 4:
each expert trains on its own data cluster; bytes are the tokens, V = 256).
Each cluster is an order-k Markov chain over 256 byte values.  For every
context (the previous k bytes) the next byte is drawn by rank from a Zipf
law p(r) proportional to r^-s, r = 1..256 (s = 1.1 by default), and the rank
is mapped to a byte by a permutation of 0..255 that depends on the cluster and
the context.  The permutation is an 8-bit, 4-round Feistel network keyed by a
64-bit hash of (cluster key, context, round), so no 65,536 x 256 table is ever
materialised.  The first k bytes of a sequence are uniform.

A "mixture" of clusters (the monolithic control trained on two clusters)
draws the cluster of every sequence uniformly from the listed clusters.
"""
from __future__ import annotations

import numpy as np

V = 256
_MASK64 = np.uint64(0xFFFFFFFFFFFFFFFF)


def _splitmix64(x: np.ndarray) -> np.ndarray:
    """The splitmix64 finaliser (Steele, Lea, Flood, OOPSLA'14) on uint64."""
    with np.errstate(over="ignore"):
        z = (x + np.uint64(0x9E3779B97F4A7C15)) & _MASK64
        z = ((z ^ (z >> np.uint64(30))) * np.uint64(0xBF58476D1CE4E5B9)) & _MASK64
        z = ((z ^ (z >> np.uint64(27))) * np.uint64(0x94D049BB133111EB)) & _MASK64
        return z ^ (z >> np.uint64(31))


def cluster_key(base_seed: int, cluster: int) -> np.uint64:
    """64-bit key of one data cluster."""
    x = np.array([(base_seed * 0x100000001B3 + cluster * 0x9E3779B1 + 0x5A17) & 0xFFFFFFFFFFFFFFFF],
                 dtype=np.uint64)
    return _splitmix64(_splitmix64(x))[0]


def _feistel8(rank: np.ndarray, keys: np.ndarray, ctx: np.ndarray) -> np.ndarray:
    """Keyed bijection of 0..255 (per element key and context), 4 rounds."""
    left = (rank >> 4) & 0xF
    right = rank & 0xF
    with np.errstate(over="ignore"):
        mixed = (ctx.astype(np.uint64) * np.uint64(0xD6E8FEB86659FD93)) & _MASK64
    base = _splitmix64(keys ^ mixed)
    for rnd in range(4):
        with np.errstate(over="ignore"):
            h = _splitmix64(base + np.uint64(rnd * 0x632BE59BD9B4E019 & 0xFFFFFFFFFFFFFFFF)
                            + right.astype(np.uint64))
        f = (h & np.uint64(0xF)).astype(np.int64)
        left, right = right, left ^ f
    return ((left << 4) | right).astype(np.int64)


def zipf_cdf(s: float = 1.1) -> np.ndarray:
    """Cumulative Zipf(s) probabilities over ranks 1..256 (last entry 1)."""
    w = np.arange(1, V + 1, dtype=np.float64) ** (-s)
    c = np.cumsum(w / w.sum())
    c[-1] = 1.0
    return c


def markov_bytes(clusters: np.ndarray, length: int, order: int, base_seed: int,
                 rng: np.random.Generator, zipf_s: float = 1.1) -> np.ndarray:
    """[len(clusters), length] uint8: one sequence per entry of ``clusters``,
    each from the order-`order` Zipf Markov chain of its cluster."""
    cl = np.asarray(clusters, dtype=np.int64)
    n_seqs = cl.size
    uniq = np.unique(cl)
    key_of = {int(c): cluster_key(base_seed, int(c)) for c in uniq}
    keys = np.array([key_of[int(c)] for c in cl], dtype=np.uint64)
    cdf = zipf_cdf(zipf_s)
    out = np.zeros((n_seqs, length), dtype=np.int64)
    k0 = min(order, length)
    out[:, :k0] = rng.integers(0, V, size=(n_seqs, k0))
    for t in range(k0, length):
        ctx = np.zeros(n_seqs, dtype=np.int64)
        for j in range(1, order + 1):
            ctx = ctx * V + out[:, t - j]
        u = rng.random(n_seqs)
        rank = np.searchsorted(cdf, u, side="right").clip(0, V - 1)
        out[:, t] = _feistel8(rank, keys, ctx)
    return out.astype(np.uint8)


def expert_batch(n_experts: int, batch: int, seq_len: int, order: int, seed: int, step: int,
                 mixture=None, zipf_s: float = 1.1) -> np.ndarray:
    """One step's batch: uint8 [n_experts, batch, seq_len + 1].

    Expert e draws from its own cluster e, unless ``mixture`` lists the
    clusters that each sequence's cluster is drawn from uniformly."""
    rng = np.random.default_rng([seed & 0xFFFFFFFF, step & 0xFFFFFFFF, 0xB17E5])
    if mixture is None:
        clusters = np.repeat(np.arange(n_experts), batch)
    else:
        clusters = rng.choice(np.asarray(list(mixture), dtype=np.int64), size=n_experts * batch)
    seqs = markov_bytes(clusters, seq_len + 1, order, seed, rng, zipf_s)
    return seqs.reshape(n_experts, batch, seq_len + 1)


def param_count(E: int, H: int) -> int:
    """Parameters of one expert: Emb[V,E], W_ih[4H,E], W_hh[4H,H], b[4H],
    W_out[V,H], b_out[V]."""
    return V * E + 4 * H * E + 4 * H * H + 4 * H + V * H + V


def param_offsets(E: int, H: int) -> dict:
    """Offsets of the blocks inside one expert's flat parameter vector."""
    o = {"emb": 0}
    o["w_ih"] = o["emb"] + V * E
    o["w_hh"] = o["w_ih"] + 4 * H * E
    o["b"] = o["w_hh"] + 4 * H * H
    o["w_out"] = o["b"] + 4 * H
    o["b_out"] = o["w_out"] + V * H
    o["end"] = o["b_out"] + V
    return o


def init_params(n_experts: int, E: int, H: int, seed: int, std: float | None = None) -> np.ndarray:
    """fp32 [n_experts, P] initial parameters.

    std given: every parameter ~ N(0, std).  Otherwise the scaled scheme:
    Emb ~ N(0, 0.1); W_ih, W_hh ~ N(0, 1/sqrt(E+H)); W_out ~ N(0, 1/sqrt(H));
    biases 0."""
    P = param_count(E, H)
    o = param_offsets(E, H)
    rng = np.random.default_rng([seed & 0xFFFFFFFF, 0x1417])
    if std is not None:
        return (rng.standard_normal((n_experts, P)) * std).astype(np.float32)
    th = np.zeros((n_experts, P), dtype=np.float64)
    th[:, o["emb"]:o["w_ih"]] = rng.standard_normal((n_experts, o["w_ih"])) * 0.1
    sw = 1.0 / np.sqrt(E + H)
    th[:, o["w_ih"]:o["b"]] = rng.standard_normal((n_experts, o["b"] - o["w_ih"])) * sw
    th[:, o["w_out"]:o["b_out"]] = rng.standard_normal((n_experts, o["b_out"] - o["w_out"])) / np.sqrt(H)
    return th.astype(np.float32)


# The five workloads: sizes and hyper-parameters of one SPSA step.
CONFIGS = {
    "tiny": dict(n_experts=1, E=32, H=64, n_pert=8, eps=1e-3, lr=1e-2, batch=4, seq_len=64,
                 order=1, mixture=None, init_std=0.1),
    "soma_n2": dict(n_experts=2, E=64, H=960, n_pert=64, eps=1e-3, lr=1e-3, batch=32,
                    seq_len=256, order=2, mixture=None, init_std=None),
    "mono": dict(n_experts=1, E=64, H=1376, n_pert=1024, eps=1e-3, lr=1e-3, batch=32,
                 seq_len=256, order=2, mixture=(0, 1), init_std=None),
    "soma_n8": dict(n_experts=8, E=64, H=480, n_pert=64, eps=1e-3, lr=1e-3, batch=32,
                    seq_len=512, order=2, mixture=None, init_std=None),
    "soma_n256": dict(n_experts=256, E=32, H=48, n_pert=64, eps=1e-3, lr=1e-3, batch=16,
                      seq_len=512, order=2, mixture=None, init_std=None),
}


def config_batch(name: str, seed: int = 0, step: int = 0, **overrides) -> np.ndarray:
    c = dict(CONFIGS[name], **overrides)
    return expert_batch(c["n_experts"], c["batch"], c["seq_len"], c["order"], seed, step,
                        mixture=c["mixture"])


def config_params(name: str, seed: int = 0, **overrides) -> np.ndarray:
    c = dict(CONFIGS[name], **overrides)
    return init_params(c["n_experts"], c["E"], c["H"], seed, c["init_std"])


# ---------------------------------------------------------------------------
# The paper's expert body (Sec. "Model size"): D pre-norm residual blocks of
# width d, a bias-free LSTM and a GELU MLP of width 4d each, gain-only
# LayerNorm, and one frozen tied head E [V, d] shared by every expert.
# ---------------------------------------------------------------------------

def body_param_count(d: int, D: int = 2) -> int:
    """M_body = 16 D d^2 + (2D + 1) d body parameters of one expert."""
    return 16 * D * d * d + (2 * D + 1) * d


def body_offsets(d: int, D: int = 2) -> dict:
    """Offsets inside one body's flat vector: per block k, W_ih [4d, d],
    W_hh [4d, d], W_1 [4d, d], W_2 [d, 4d]; then per block the gains ga, gb
    [d]; then the final gain gf [d]."""
    q = d * d
    o = {}
    for k in range(D):
        base = 16 * q * k
        o[f"w_ih{k}"] = base
        o[f"w_hh{k}"] = base + 4 * q
        o[f"w1{k}"] = base + 8 * q
        o[f"w2{k}"] = base + 12 * q
    g0 = 16 * q * D
    for k in range(D):
        o[f"ga{k}"] = g0 + 2 * d * k
        o[f"gb{k}"] = g0 + 2 * d * k + d
    o["gf"] = g0 + 2 * d * D
    o["gains"] = g0
    o["end"] = o["gf"] + d
    return o


def init_body(n_experts: int, d: int, D: int, seed: int) -> np.ndarray:
    """fp32 [n_experts, M_body]: W_ih, W_hh, W_1 ~ N(0, 1/sqrt(d)),
    W_2 ~ N(0, 1/sqrt(4d)), gains 1."""
    o = body_offsets(d, D)
    rng = np.random.default_rng([seed & 0xFFFFFFFF, 0x2B0D])
    th = np.zeros((n_experts, o["end"]), dtype=np.float64)
    for k in range(D):
        th[:, o[f"w_ih{k}"]:o[f"w2{k}"]] = rng.standard_normal((n_experts, 12 * d * d)) / np.sqrt(d)
        th[:, o[f"w2{k}"]:o[f"w2{k}"] + 4 * d * d] = (rng.standard_normal((n_experts, 4 * d * d))
                                                     / np.sqrt(4 * d))
    th[:, o["gains"]:] = 1.0
    return th.astype(np.float32)


def init_head(d: int, seed: int) -> np.ndarray:
    """fp32 [V, d] frozen tied embedding/decode matrix E ~ N(0, 1/sqrt(d)),
    standing in for the seed run's learned E."""
    rng = np.random.default_rng([seed & 0xFFFFFFFF, 0x4EAD])
    return (rng.standard_normal((V, d)) / np.sqrt(d)).astype(np.float32)


# The body workloads: the paper's width-32 N = 256 ensemble at the SOMA
# N=256 batch shape, and its own training batch (B = 64, 1,024-byte windows).
BODY_CONFIGS = {
    "body_tiny": dict(n_experts=2, d=32, D=2, n_pert=4, eps=1e-3, lr=1e-3, batch=3, seq_len=20,
                      order=2),
    "body_n256": dict(n_experts=256, d=32, D=2, n_pert=64, eps=1e-3, lr=1e-3, batch=16,
                      seq_len=512, order=2),
    "body_n256_paper": dict(n_experts=256, d=32, D=2, n_pert=64, eps=1e-3, lr=1e-3, batch=64,
                            seq_len=1024, order=2),
}


def body_config_batch(name: str, seed: int = 0, step: int = 0, **overrides) -> np.ndarray:
    c = dict(BODY_CONFIGS[name], **overrides)
    return expert_batch(c["n_experts"], c["batch"], c["seq_len"], c["order"], seed, step)


def body_config_params(name: str, seed: int = 0, **overrides) -> np.ndarray:
    c = dict(BODY_CONFIGS[name], **overrides)
    return init_body(c["n_experts"], c["d"], c["D"], seed)
