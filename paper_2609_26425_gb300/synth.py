"""Seeded synthetic inputs shaped like the paper's video world-model workloads.

This module only draws random numbers (torch CPU generator, fixed call
order, rounded to bf16) and describes the workload shapes.  It holds none of
the quantization or attention arithmetic, so both the CUDA path and the CPU
oracle can take their inputs from it.

Recipe (per head h, channel c):
  * Queries  q = N(0,1) * s_hc with s_hc = exp(a_hc), a_hc ~ N(0, 0.5^2)
    (LogNormal(0, 0.5) channel scales).  With query drift rho, the log-scales
    follow an AR(1) chain across chunks:
    a^(t) = rho a^(t-1) + sqrt(1 - rho^2) * 0.5 * xi.
  * Keys     k = N(0,1) with 4 fixed outlier channels multiplied by 8; with
    ``key_tail='student_t3'`` those channels are Student-t(nu=3) draws times 8.
  * Values   v = N(0,1).
  * Sensitivity weights w and the principal Query basis U are given to the
    path as inputs.  ``population_w`` is the per-channel variance s_hc^2 of the
    query distribution normalised to mean one, ``population_U`` the unit
    vectors of the r highest-variance channels (the exact top-r eigenvectors
    of that distribution's diagonal second moment), ``random_orthonormal`` a
    general orthonormal basis for tests.
Seeds: workload seed ``s``; (layer, chunk) sub-seed ``s*10**6 + layer*10**3 +
chunk``.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field, replace

import numpy as np
import torch

HEAD_DIM = 128
NUM_OUTLIERS = 4
OUTLIER_GAIN = 8.0


@dataclass(frozen=True)
class Workload:
    """Shape of one synthetic workload (one attention layer unless ``layers``)."""
    name: str
    heads: int
    chunk_tokens: int          # tokens appended per chunk (= query tokens per chunk)
    past_chunks: int           # cached chunks attended by the new chunk
    centroids: int             # C
    group_size: int            # G
    psac_rank: int             # r
    candidates: int = 4        # M (top-M QSAC candidates)
    kmeans_iters: int = 10
    head_dim: int = HEAD_DIM
    layers: int = 1
    window: int = 0            # sliding window in chunks (0 = unbounded ring)
    key_tail: str = "gauss"    # or "student_t3"
    query_drift: float = 0.0   # AR(1) rho of the query log-scales across chunks
    seed: int = 0
    note: str = ""

    @property
    def cache_tokens(self) -> int:
        return self.past_chunks * self.chunk_tokens


WORKLOADS = {
    "single_layer_h4": Workload(
        "single_layer_h4", heads=4, chunk_tokens=880, past_chunks=2, centroids=64,
        group_size=32, psac_rank=16, kmeans_iters=10, seed=0,
        note="1 layer, 4 heads, 2 cached chunks of 880, new chunk 880"),
    "wan14b_layer": Workload(
        "wan14b_layer", heads=40, chunk_tokens=4680, past_chunks=6, centroids=256,
        group_size=32, psac_rank=16, kmeans_iters=10, query_drift=0.9, seed=1,
        note="Wan-14B-shaped DiT self-attention layer: 3 latent frames x 1560 tokens per "
             "chunk, 6 cached chunks (28080 tokens)"),
    "wan14b_stack": Workload(
        "wan14b_stack", heads=40, chunk_tokens=4680, past_chunks=8, centroids=256,
        group_size=32, psac_rank=16, kmeans_iters=10, layers=40, query_drift=0.9, seed=2,
        note="40 layers of the Wan-14B layer, cache grown to 37440 tokens"),
    "dit1p3b_window": Workload(
        "dit1p3b_window", heads=12, chunk_tokens=880, past_chunks=15, centroids=64,
        group_size=32, psac_rank=8, layers=30, window=15, key_tail="student_t3", seed=3,
        note="~1.3B causal video DiT: 1-frame chunks of 880, sliding window of 15 frames"),
}


def sub_seed(seed: int, layer: int, chunk: int) -> int:
    return seed * 10**6 + layer * 10**3 + chunk


def _gen(seed: int) -> torch.Generator:
    g = torch.Generator()
    g.manual_seed(int(seed))
    return g


class ChunkSource:
    """Seeded Q/K/V chunks of one layer of a workload."""

    def __init__(self, wl: Workload, layer: int = 0):
        self.wl = wl
        self.layer = layer
        H, d = wl.heads, wl.head_dim
        g = _gen(sub_seed(wl.seed, layer, 999))
        self.log_scale0 = torch.randn(H, d, generator=g, dtype=torch.float32) * 0.5
        self.outliers = torch.randperm(d, generator=g)[:NUM_OUTLIERS].sort().values
        self._ls_cache = {0: self.log_scale0}

    def query_log_scale(self, chunk: int) -> torch.Tensor:
        """Per-head channel log-scales a^(chunk) ([H][d] fp32)."""
        rho = self.wl.query_drift
        if rho == 0.0:
            return self.log_scale0
        if chunk in self._ls_cache:
            return self._ls_cache[chunk]
        prev = self.query_log_scale(chunk - 1)
        g = _gen(sub_seed(self.wl.seed, self.layer, 500 + chunk))
        xi = torch.randn(prev.shape, generator=g, dtype=torch.float32)
        a = rho * prev + math.sqrt(1.0 - rho * rho) * 0.5 * xi
        self._ls_cache[chunk] = a
        return a

    def chunk(self, chunk: int, tokens: int | None = None):
        """(q, k, v) bf16 CPU tensors [N][H][d] for chunk index ``chunk``."""
        wl = self.wl
        N = wl.chunk_tokens if tokens is None else tokens
        H, d = wl.heads, wl.head_dim
        g = _gen(sub_seed(wl.seed, self.layer, chunk))
        s = torch.exp(self.query_log_scale(chunk))
        q = torch.randn(N, H, d, generator=g, dtype=torch.float32) * s
        k = torch.randn(N, H, d, generator=g, dtype=torch.float32)
        if wl.key_tail == "student_t3":
            z = torch.randn(N, H, NUM_OUTLIERS, generator=g, dtype=torch.float32)
            chi = torch.randn(N, H, NUM_OUTLIERS, 3, generator=g, dtype=torch.float32).pow(2).sum(-1)
            k[:, :, self.outliers] = z / torch.sqrt(chi / 3.0) * OUTLIER_GAIN
        else:
            k[:, :, self.outliers] *= OUTLIER_GAIN
        v = torch.randn(N, H, d, generator=g, dtype=torch.float32)
        return q.to(torch.bfloat16), k.to(torch.bfloat16), v.to(torch.bfloat16)


def population_w(log_scale: torch.Tensor) -> torch.Tensor:
    """Per-channel query variance exp(2a) normalised to mean one ([H][d] fp32)."""
    var = torch.exp(2.0 * log_scale.double())
    return (var / var.mean(dim=-1, keepdim=True)).float()


def population_U(log_scale: torch.Tensor, r: int) -> torch.Tensor:
    """Unit vectors of the r highest-variance channels, [H][d][r] bf16."""
    H, d = log_scale.shape
    U = torch.zeros(H, d, r, dtype=torch.float32)
    if r > 0:
        idx = torch.argsort(log_scale, dim=-1, descending=True)[:, :r]
        for h in range(H):
            U[h, idx[h], torch.arange(r)] = 1.0
    return U.to(torch.bfloat16)


def random_orthonormal(seed: int, H: int, d: int, r: int) -> torch.Tensor:
    """Orthonormal columns from the QR factorisation of a Gaussian, [H][d][r] bf16."""
    g = _gen(seed)
    a = torch.randn(H, d, max(r, 1), generator=g, dtype=torch.float64)
    qm, _ = torch.linalg.qr(a)
    return qm[:, :, :r].to(torch.bfloat16)


def random_weights(seed: int, H: int, d: int) -> torch.Tensor:
    """Positive weights with mean one per head ([H][d] fp32), LogNormal(0, 1) shaped."""
    g = _gen(seed)
    a = torch.exp(torch.randn(H, d, generator=g, dtype=torch.float64))
    return (a / a.mean(dim=-1, keepdim=True)).float()


def gaussian_bf16(seed: int, *shape, scale: float = 1.0) -> torch.Tensor:
    g = _gen(seed)
    return (torch.randn(*shape, generator=g, dtype=torch.float32) * scale).to(torch.bfloat16)


def bits(t: torch.Tensor) -> np.ndarray:
    """bf16 tensor -> numpy uint16 bit pattern (same shape)."""
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


def from_bits(a: np.ndarray) -> torch.Tensor:
    """numpy uint16 bf16 bit pattern -> bf16 CPU tensor."""
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16)


def hadamard_queries(H: int, d: int = 128) -> torch.Tensor:
    """Queries along the rows of a Sylvester Hadamard matrix, [d][H][d] bf16.

    Query n of head h is s_h(n) * had[n], with had the d x d matrix of +-1
    built by repeated Kronecker doubling and s_h(n) = n + 1 for even heads,
    d - n for odd heads (integers <= 256, exact in bf16).  The rows are
    orthogonal, so the set's second moment has the rows as eigenvectors with
    eigenvalues s_h(n)^2 and a constant diagonal.
    """
    had = torch.ones(1, 1, dtype=torch.float32)
    while had.shape[0] < d:
        had = torch.cat([torch.cat([had, had], 1), torch.cat([had, -had], 1)], 0)
    n = torch.arange(d, dtype=torch.float32)
    q = torch.empty(d, H, d, dtype=torch.float32)
    for h in range(H):
        s = n + 1 if h % 2 == 0 else d - n
        q[:, h] = s[:, None] * had
    return q.to(torch.bfloat16)
