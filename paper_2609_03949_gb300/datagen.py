"""Seeded synthetic MLA decode workloads.

This module only draws inputs. It holds none of the method's arithmetic (no scoring, selection,
attention or trigger), so both the CUDA library and the CPU oracle consume its output.

Recipe (one decode step of one attention layer, B independent sequences):

* cache row u of sequence b is ``[L_u ; K_u]``: the 512-wide compressed latent followed by the 64-wide
  decoupled RoPE key (the paper's ``C_u = [c_u; r_u]``, Eq. 1, 576 values, 1152 bytes in bf16);
* latent entries ~ N(0,1)/sqrt(512);
* RoPE keys: N(0,1)^64 vectors rotated at their position u (interleaved pairs (2i, 2i+1), frequency
  10000^(-2i/64)); ``lognormal_keys`` rescales each key to norm 8*exp(0.5*xi), xi ~ N(0,1), before rotating;
* absorbed query latent part ~ N(0,1)^512 per head; RoPE part N(0,1)^64 rotated at position N;
* ``query_rank`` k > 0 makes the content queries low-rank plus noise, as a model's queries are: q = sqrt((1-nu) 512/k)
  U g + sqrt(nu) eps, U the first k rows of a seeded Haar 512x512 rotation, g ~ N(0,1)^k, eps ~ N(0,1)^512, nu =
  ``query_noise`` (E|q|^2 = 512 as in the isotropic case); ``prefix_queries`` draws the context's earlier queries
  from the same law (the sketch basis is computed from them);
* planted rows: ``n_planted`` distinct archive positions per sequence; planted row p targets head p mod H and
  stores the key 4 * q_rope[h] / |q_rope[h]| (a stored, already-rotated value);
* everything stored as bf16 by round-to-nearest-even from fp32, or kept fp32;
* a Haar-random 64x64 orthogonal matrix (QR of a seeded Gaussian, sign-fixed) for the width-r digest.
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np
import torch

D_LATENT = 512
D_ROPE = 64
D_ROW = D_LATENT + D_ROPE
ROPE_BASE = 10000.0


@dataclasses.dataclass
class Workload:
    """One synthetic decode step. ``cache`` is [B, N, 576]; latent = cache[..., :512], rope = cache[..., 512:]."""

    B: int
    H: int
    N: int
    dtype: str                    # "bf16" or "f32"
    cache: torch.Tensor           # [B, N, 576]
    q_latent: torch.Tensor        # [B, H, 512]
    q_rope: torch.Tensor          # [B, H, 64]
    rot: torch.Tensor             # [64, 64] float32, row-major orthogonal
    planted_pos: torch.Tensor     # [B, n_planted] int64 positions (may be empty)
    planted_head: torch.Tensor    # [n_planted] int64 target head of each planted row
    seed: int
    query_rank: int = 0           # > 0: content queries low-rank plus noise (see the module notes)
    query_noise: float = 0.0

    @property
    def latent(self) -> torch.Tensor:
        return self.cache[..., :D_LATENT]

    @property
    def rope(self) -> torch.Tensor:
        return self.cache[..., D_LATENT:]

    def to(self, device) -> "Workload":
        return dataclasses.replace(
            self, cache=self.cache.to(device), q_latent=self.q_latent.to(device),
            q_rope=self.q_rope.to(device), rot=self.rot.to(device))

    def slice_batch(self, bs) -> "Workload":
        """Sub-workload with the sequences ``bs`` (a list of batch indices)."""
        bs = list(bs)
        return dataclasses.replace(
            self, B=len(bs), cache=self.cache[bs].contiguous(), q_latent=self.q_latent[bs].contiguous(),
            q_rope=self.q_rope[bs].contiguous(), planted_pos=self.planted_pos[bs].contiguous())


def _slice_rows(self, n: int) -> "Workload":
    """The same sequences cut to their first ``n`` cached rows (an earlier point of the same stream)."""
    pp = self.planted_pos.clone()
    pp[pp >= n] = -1
    return dataclasses.replace(self, N=n, cache=self.cache[:, :n].contiguous(), planted_pos=pp)


Workload.slice_rows = _slice_rows


def _spiked_queries(n: int, query_rank: int, query_noise: float, basis_seed: int, gen: torch.Generator,
                    device) -> torch.Tensor:
    """n content queries [n, 512] (fp32): sqrt((1-nu) 512/k) U g + sqrt(nu) eps (see the module notes)."""
    U = torch.from_numpy(haar_orthogonal(basis_seed, D_LATENT)[:query_rank]).float().to(device)
    g = torch.randn(n, query_rank, generator=gen, device=device)
    eps = torch.randn(n, D_LATENT, generator=gen, device=device)
    return math.sqrt((1.0 - query_noise) * D_LATENT / query_rank) * (g @ U) + math.sqrt(query_noise) * eps


def prefix_queries(wl: "Workload", n: int, seed_offset: int = 1) -> torch.Tensor:
    """n earlier content queries of the same context [n, 512], in the workload's storage dtype: the same law as its
    decode queries (the same subspace U when ``query_rank`` > 0), independent draws."""
    gen = torch.Generator(device="cpu")
    gen.manual_seed(int(wl.seed) * 7 + 1_000_003 * int(seed_offset))
    if wl.query_rank > 0:
        q = _spiked_queries(n, wl.query_rank, wl.query_noise, wl.seed + 15485863, gen, "cpu")
    else:
        q = torch.randn(n, D_LATENT, generator=gen)
    return q.to(torch.bfloat16 if wl.dtype == "bf16" else torch.float32)


def haar_orthogonal(seed: int, n: int = D_ROPE) -> np.ndarray:
    """Haar-distributed n x n orthogonal matrix (default 64): QR of a seeded Gaussian with sign(diag R) > 0 (fp64)."""
    rng = np.random.default_rng(seed)
    g = rng.standard_normal((n, n))
    q, r = np.linalg.qr(g)
    q = q * np.sign(np.diag(r))[None, :]
    return q


def _rope_tables(positions: np.ndarray):
    """cos/sin of pos * 10000^(-2i/64) for the 32 interleaved pairs, computed in fp64."""
    inv = ROPE_BASE ** (-np.arange(0, D_ROPE, 2, dtype=np.float64) / D_ROPE)
    ang = positions.astype(np.float64)[:, None] * inv[None, :]
    return np.cos(ang), np.sin(ang)


def _rotate_pairs(x: torch.Tensor, cos: torch.Tensor, sin: torch.Tensor) -> torch.Tensor:
    """Rotate interleaved pairs (x[2i], x[2i+1]) by the angles whose cos/sin are given ([..., 32])."""
    xe, xo = x[..., 0::2], x[..., 1::2]
    out = torch.empty_like(x)
    out[..., 0::2] = xe * cos - xo * sin
    out[..., 1::2] = xe * sin + xo * cos
    return out


def make_workload(B: int, H: int, N: int, *, dtype: str = "bf16", seed: int = 0, n_planted: int = 0,
                  lognormal_keys: bool = False, planted_lo: int = 0, planted_hi: int | None = None,
                  query_rank: int = 0, query_noise: float = 0.05, device: str | torch.device = "cpu") -> Workload:
    """Draw one decode step's cache and queries.

    Planted rows go to distinct positions in [planted_lo, planted_hi) (the archive range of the caller's
    selection parameters; default the whole context).
    """
    if dtype not in ("bf16", "f32"):
        raise ValueError(f"dtype must be bf16 or f32, got {dtype}")
    device = torch.device(device)
    gen = torch.Generator(device=device)
    gen.manual_seed(int(seed))
    store = torch.bfloat16 if dtype == "bf16" else torch.float32
    cos_k, sin_k = _rope_tables(np.arange(N))
    cos_k = torch.from_numpy(cos_k).float().to(device)
    sin_k = torch.from_numpy(sin_k).float().to(device)
    cos_q, sin_q = _rope_tables(np.array([N]))
    cos_q = torch.from_numpy(cos_q).float().to(device)
    sin_q = torch.from_numpy(sin_q).float().to(device)

    q_latent = torch.randn(B, H, D_LATENT, generator=gen, device=device)
    if query_rank > 0:   # drawn from a generator of their own, so the cache is the same as with isotropic queries
        gq = torch.Generator(device=device)
        gq.manual_seed(int(seed) + 31337)
        q_latent = _spiked_queries(B * H, query_rank, query_noise, seed + 15485863, gq, device).view(B, H, D_LATENT)
    q_rope = _rotate_pairs(torch.randn(B, H, D_ROPE, generator=gen, device=device), cos_q, sin_q)

    hi = N if planted_hi is None else planted_hi
    n_planted = int(min(n_planted, max(0, hi - planted_lo)))
    planted_pos = torch.zeros(B, n_planted, dtype=torch.int64)
    planted_head = torch.arange(n_planted, dtype=torch.int64) % max(H, 1)

    cache = torch.empty(B, N, D_ROW, dtype=store, device=device)
    for b in range(B):  # one sequence at a time bounds the fp32 temporaries
        lat = torch.randn(N, D_LATENT, generator=gen, device=device) / math.sqrt(D_LATENT)
        key = torch.randn(N, D_ROPE, generator=gen, device=device)
        if lognormal_keys:
            xi = torch.randn(N, 1, generator=gen, device=device)
            key = key / key.norm(dim=1, keepdim=True) * (8.0 * torch.exp(0.5 * xi))
        key = _rotate_pairs(key, cos_k, sin_k)
        if n_planted:
            perm = torch.randperm(hi - planted_lo, generator=gen, device=device)[:n_planted] + planted_lo
            planted_pos[b] = perm.cpu()
            qd = q_rope[b, planted_head.to(device)]
            key[perm] = 4.0 * qd / qd.norm(dim=1, keepdim=True)
        cache[b, :, :D_LATENT] = lat.to(store)
        cache[b, :, D_LATENT:] = key.to(store)
        del lat, key

    rot = torch.from_numpy(haar_orthogonal(seed + 7919)).float().to(device)
    return Workload(B=B, H=H, N=N, dtype=dtype, cache=cache, q_latent=q_latent.to(store),
                    q_rope=q_rope.to(store), rot=rot, planted_pos=planted_pos, planted_head=planted_head,
                    seed=int(seed), query_rank=int(query_rank), query_noise=float(query_noise if query_rank else 0.0))


# The five evaluation workloads, named by what they are, with their sizes. ``CONFIG_PARAMS`` gives the selection
# parameters each one is run with, and each draws from its own seed unless a sweep point overrides it.
CONFIGS = {
    "fp32_h16_n1k": dict(B=1, H=16, N=1024, dtype="f32", n_planted=8, seed=0),
    "h128_n8k": dict(B=1, H=128, N=8192, dtype="bf16", n_planted=32, seed=1),
    "h64_n32k_lognormal": dict(B=16, H=64, N=32768, dtype="bf16", n_planted=0, lognormal_keys=True, seed=2),
    "h128_n64k_two_tier": dict(B=8, H=128, N=65536, dtype="bf16", n_planted=32, seed=3),
    "h64_n64k": dict(B=8, H=64, N=65536, dtype="bf16", n_planted=64, seed=1000),
}

CONFIG_PARAMS = {
    "fp32_h16_n1k": dict(rho=1 / 8, window=64, r=64),
    "h128_n8k": dict(rho=1 / 32, window=128, r=64),
    "h64_n32k_lognormal": dict(rho=1 / 32, window=256, r=64),
    "h128_n64k_two_tier": dict(rho=1 / 32, window=256, r=64, trigger=1, z_eff=1.0),
    "h64_n64k": dict(rho=1 / 32, window=256, r=64),
}


def config_workload(name: str, device="cpu", **overrides) -> Workload:
    kw = dict(CONFIGS[name])
    kw.update(overrides)
    window = CONFIG_PARAMS[name]["window"]
    return make_workload(device=device, planted_lo=0, planted_hi=max(0, kw["N"] - window), **kw)


def bf16_bits(t: torch.Tensor) -> np.ndarray:
    """The raw uint16 storage of a bf16 tensor (host copy)."""
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)
