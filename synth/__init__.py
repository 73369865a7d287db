"""Seeded synthetic inputs for the ReSS global-attention layer.

This module holds the workload shapes and the random input recipe only: it contains none
of the method's arithmetic (no pooling, softmax, drift or selection).  Both the CUDA path
(through tests and bench.py) and the CPU oracle receive the arrays it returns, so the two
sides always see the same bf16 bytes.

Token layout of one layer (the 3D-ViT global attention of Sec. 3 / Sec. 5.1): every view
contributes 37x37 = 1369 patch tokens and 5 special (camera/register) tokens.  All patch
tokens of all views come first (view-major, row-major inside a view), then all special
tokens; special tokens therefore sit in the trailing key blocks, which the method always
keeps (Sec. 4.1, "Blocks containing special tokens are always kept").

Recipe, per tensor X in {Q, K, V}, head h and token t of view v:

    X[t, h, :] = n + (sigma / sqrt(r)) * sum_k a[t, k] * U[h, v, k, :] + ramp[t] * w[X, h, :]
                 (+ (1 / sqrt(r0)) * sum_k b[t, k] * U0[h, k, :]  when a cross-view rank r0 > 0)

n ~ N(0, I) fresh per tensor; U[h, v] ~ N(0, I) shared by Q, K and V; a[t] ~ N(0, I_r)
shared by the three tensors of token t; ramp[t] = 2 p / 1368 - 1 for patch p of its view
and 0 for special tokens; w[X, h] ~ N(0, I).  W_o ~ N(0, 0.02^2) is the d_model x d_model
output projection (Linear.weight layout, out x in).  Everything is rounded to bf16
(round-to-nearest-even) and returned as uint16 bit patterns.

Determinism: numpy's PCG64 streams, one per (seed, tensor id); sums are accumulated with
separate elementwise multiplies and adds in float32, which are correctly rounded on every
platform.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np

PATCHES_PER_VIEW = 37 * 37          # 1369
SPECIAL_PER_VIEW = 5                # camera + register tokens
TOKENS_PER_VIEW = PATCHES_PER_VIEW + SPECIAL_PER_VIEW  # 1374
HEAD_DIM = 64
BLOCK = 64

# stream ids of the generator (one PCG64 stream per id)
_ID = {"Q": 0, "K": 1, "V": 2, "W_o": 3, "U": 4, "a": 5, "w": 6, "b": 7, "U0": 8}


@dataclass(frozen=True)
class Workload:
    """One synthetic global-attention layer and the ReSS settings applied to it."""
    name: str
    views: int
    heads: int
    d_model: int
    sparsity: float          # dropped fraction of candidate key blocks per row
    rounds: int              # restoration rounds R
    rank: int = 16           # per-view shared rank r
    sigma: float = 2.0       # scale of the per-view component
    cross_rank: int = 0      # cross-view shared rank (0 = none)
    cross_scale: float = 1.0
    rho: float = 0.5         # swap budget fraction, Eq. 17
    seed: int = 0

    # ---- derived shapes -------------------------------------------------------------
    @property
    def n_tokens(self) -> int:
        return self.views * TOKENS_PER_VIEW

    @property
    def n_special(self) -> int:
        return self.views * SPECIAL_PER_VIEW

    @property
    def n_blocks(self) -> int:
        return -(-self.n_tokens // BLOCK)

    @property
    def n_candidates(self) -> int:
        """|P|: key blocks made only of patch tokens."""
        return (self.n_tokens - self.n_special) // BLOCK

    def budgets(self) -> np.ndarray:
        """Uniform per-head keep budget c_h = max(2, round_half_even((1 - s) |P|))."""
        c = max(2, int(round((1.0 - self.sparsity) * self.n_candidates)))
        c = min(c, self.n_candidates)
        return np.full(self.heads, c, dtype=np.int32)

    def with_(self, **kw) -> "Workload":
        d = {f: getattr(self, f) for f in self.__dataclass_fields__}
        d.update(kw)
        return Workload(**d)


# The five workloads the benchmark and the parity tests use (2 to 100 views).
WORKLOADS = {
    "tiny_v2": Workload("tiny_v2", views=2, heads=4, d_model=256, sparsity=0.5, rounds=2, rank=8),
    "vggt_v8": Workload("vggt_v8", views=8, heads=16, d_model=1024, sparsity=0.75, rounds=3),
    "vggt_v32": Workload("vggt_v32", views=32, heads=16, d_model=1024, sparsity=0.9, rounds=3),
    "vggt_v100": Workload("vggt_v100", views=100, heads=16, d_model=1024, sparsity=0.9, rounds=3,
                          cross_rank=4, cross_scale=1.0),
    "vggt_v64": Workload("vggt_v64", views=64, heads=16, d_model=1024, sparsity=0.9, rounds=4),
}
SWEEP_V64 = [(s, r) for s in (0.5, 0.75, 0.9, 0.95) for r in (0, 1, 2, 4)]


def _rng(seed: int, name: str) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([seed, _ID[name]])))


def bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 values to bf16 (nearest, ties to even); return the uint16 bit patterns."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    lsb = (u >> np.uint32(16)) & np.uint32(1)       # inputs are finite: no uint32 overflow
    r = u + np.uint32(0x7FFF)
    r += lsb
    r >>= np.uint32(16)
    return r.astype(np.uint16)


def bf16_to_f32(bits: np.ndarray) -> np.ndarray:
    """Widen bf16 bit patterns to float32 (exact)."""
    return (bits.astype(np.uint32) << 16).view(np.float32)


def token_views(wl: Workload) -> tuple[np.ndarray, np.ndarray]:
    """Per-token view index and positional ramp (0 for special tokens)."""
    V = wl.views
    view = np.empty(wl.n_tokens, dtype=np.int64)
    ramp = np.zeros(wl.n_tokens, dtype=np.float32)
    p = np.arange(PATCHES_PER_VIEW, dtype=np.float32)
    npatch = V * PATCHES_PER_VIEW
    view[:npatch] = np.repeat(np.arange(V), PATCHES_PER_VIEW)
    ramp[:npatch] = np.tile(2.0 * p / np.float32(PATCHES_PER_VIEW - 1) - 1.0, V)
    view[npatch:] = np.repeat(np.arange(V), SPECIAL_PER_VIEW)
    return view, ramp


def make_inputs(wl: Workload) -> dict:
    """Q, K, V as bf16 bits [N, H, 64] and W_o as bf16 bits [d_model, d_model]."""
    N, H, r = wl.n_tokens, wl.heads, wl.rank
    view, ramp = token_views(wl)
    U = _rng(wl.seed, "U").standard_normal((H, wl.views, r, HEAD_DIM), dtype=np.float32)
    a = _rng(wl.seed, "a").standard_normal((N, r), dtype=np.float32)
    w = _rng(wl.seed, "w").standard_normal((3, H, HEAD_DIM), dtype=np.float32)
    coef = np.float32(wl.sigma / math.sqrt(r))
    if wl.cross_rank:
        U0 = _rng(wl.seed, "U0").standard_normal((H, wl.cross_rank, HEAD_DIM), dtype=np.float32)
        b = _rng(wl.seed, "b").standard_normal((N, wl.cross_rank), dtype=np.float32)
        ccoef = np.float32(wl.cross_scale / math.sqrt(wl.cross_rank))

    # shared (tensor-independent) structured part, one view and one rank term at a time
    shared = np.zeros((N, H, HEAD_DIM), dtype=np.float32)
    for v in range(wl.views):
        idx = np.nonzero(view == v)[0]
        acc = np.zeros((idx.size, H, HEAD_DIM), dtype=np.float32)
        for k in range(r):
            acc += a[idx, k][:, None, None] * U[None, :, v, k, :]
        shared[idx] = acc * coef
    if wl.cross_rank:
        cross = np.zeros((N, H, HEAD_DIM), dtype=np.float32)
        for k in range(wl.cross_rank):
            cross += b[:, k][:, None, None] * U0[None, :, k, :]
        shared += ccoef * cross
        del cross

    out = {}
    for xi, name in enumerate(("Q", "K", "V")):
        x = _rng(wl.seed, name).standard_normal((N, H, HEAD_DIM), dtype=np.float32)
        x += shared
        x += ramp[:, None, None] * w[xi][None, :, :]
        out[name] = bf16_bits(x)
        del x
    W = _rng(wl.seed, "W_o").standard_normal((wl.d_model, wl.d_model), dtype=np.float32)
    out["W_o"] = bf16_bits(W * np.float32(0.02))
    return out


def make_random_layer(n_tokens: int, heads: int, d_model: int, seed: int,
                      rank: int = 4, sigma: float = 2.0) -> dict:
    """A layer of arbitrary (ragged) length for unit and edge-case tests: Q, K, V = N(0, I)
    + a rank-`rank` component shared by the three tensors + a linear ramp over the token
    index.  Same return format as make_inputs."""
    g = np.random.Generator(np.random.PCG64(np.random.SeedSequence([seed, 100])))
    U = g.standard_normal((heads, rank, HEAD_DIM), dtype=np.float32)
    a = g.standard_normal((n_tokens, rank), dtype=np.float32)
    w = g.standard_normal((3, heads, HEAD_DIM), dtype=np.float32)
    ramp = np.linspace(-1.0, 1.0, n_tokens, dtype=np.float32)
    shared = np.zeros((n_tokens, heads, HEAD_DIM), dtype=np.float32)
    for k in range(rank):
        shared += a[:, k][:, None, None] * U[None, :, k, :]
    shared *= np.float32(sigma / math.sqrt(rank))
    out = {}
    for xi, name in enumerate(("Q", "K", "V")):
        x = g.standard_normal((n_tokens, heads, HEAD_DIM), dtype=np.float32)
        x += shared
        x += ramp[:, None, None] * w[xi][None, :, :]
        out[name] = bf16_bits(x)
    W = g.standard_normal((d_model, d_model), dtype=np.float32)
    out["W_o"] = bf16_bits(W * np.float32(0.02))
    return out
