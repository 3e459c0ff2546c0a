"""Helpers shared by the GPU parity tests: run a step through the C ABI and compare it with the oracle.

Comparison rules (the path's correctness criteria, written out):

* Selection: every head's set has exactly k + W + n_sink rows and contains the window and the sinks. Its
  archive part must equal the oracle's except for rows whose score lies within 1e-3 relative of the k-th
  threshold tau: |a - tau| <= 1e-3 * max(|tau|, 1e-3 * rms(a)). Rows inside that band may differ, but the
  GPU's choice must still be a valid top-k: every kept archive row scores >= tau - band and every dropped one
  <= tau + band.
* Outputs: the oracle is re-run on the GPU's own selected sets (so near-tie swaps do not leak into the output
  check); per (b, h), max|o_gpu - o_ref| / max|o_ref| <= 2e-2 and |lse_gpu - lse_ref| <= 2e-2.
* Trigger: fired rows must match the oracle's except where |T - s*| lies within the same relative band.
"""
from __future__ import annotations

import math

import numpy as np
import torch

import oracle
from paper_2609_03949_gb300 import datagen
from paper_2609_03949_gb300 import vk

OUT_RTOL = 2e-2
LSE_ATOL = 2e-2
TIE_REL = 1e-3


def band(tau: float, a: np.ndarray) -> float:
    rms = float(np.sqrt(np.mean(a * a))) if a.size else 1.0
    return TIE_REL * max(abs(tau), TIE_REL * rms, 1e-30)


class GpuStep:
    """Inputs on the GPU plus the C-ABI call of one decode step."""

    def __init__(self, wl: datagen.Workload, *, rho, r=64, window=0, n_sink=0, trigger=0, z_eff=1.0, top_j=0,
                 flags=0, digest_bf16: np.ndarray | None = None, cap=None, sketch=None):
        """sketch = (stored bf16 entries [B,N,r_sk] uint16, basis [r_sk,512], residual norms eta [B,N]): the rank-r_sk
        content sketch of the row-level trigger, taken from the oracle so that both sides score the same index."""
        self.wl = wl.to("cuda")
        self.view = vk.make_view(self.wl.cache, self.wl.q_latent, self.wl.q_rope)
        r_sk = 0 if sketch is None else sketch[1].shape[0]
        self.params = vk.make_params(rho, r=r, window=window, n_sink=n_sink, trigger=trigger, z_eff=z_eff,
                                     top_j=top_j, flags=flags, r_sk=r_sk)
        B, N = wl.B, wl.N
        P = (N + 63) // 64
        self.rot = self.wl.rot.contiguous()
        self.eta = torch.empty(B, N, dtype=torch.float32, device="cuda")
        self.page_res = torch.empty(B, P, dtype=torch.float32, device="cuda")
        self.page_knorm = torch.empty(B, P, dtype=torch.float32, device="cuda")
        self.page_eta = torch.empty(B, P, dtype=torch.float32, device="cuda")
        self.digest = None
        if r < 64:
            # the oracle's bf16 digest feeds both sides, so the scores are compared on identical inputs
            assert digest_bf16 is not None
            self.digest = torch.from_numpy(digest_bf16.astype(np.int16)).view(torch.bfloat16).cuda().contiguous()
        vk.vk_build_digest(self.view, self.params, self.rot, None, self.eta, self.page_res, self.page_knorm,
                           self.page_eta)
        self.sketch = self.basis = None
        if sketch is not None:
            self.sketch = torch.from_numpy(sketch[0].astype(np.int16)).view(torch.bfloat16).cuda().contiguous()
            self.basis = torch.as_tensor(sketch[1], dtype=torch.float32).cuda().contiguous()
            self.eta = torch.as_tensor(sketch[2], dtype=torch.float32).cuda().contiguous()
        self.index = vk.make_index(self.digest, self.eta, self.page_res, self.rot if r < 64 else None,
                                   self.page_knorm, self.page_eta, self.sketch, self.basis)
        self.buf = vk.DecodeBuffers(self.view, self.params, cap=cap)

    def run(self):
        self.buf.run(self.view, self.params, self.index)
        torch.cuda.synchronize()
        st = vk.vk_poll_status(self.buf.ws)
        return dict(out=self.buf.out.cpu().double().numpy(), lse=self.buf.lse.cpu().double().numpy(),
                    smax=self.buf.smax.cpu().double().numpy(), idx=self.buf.idx.cpu().numpy(),
                    count=self.buf.count.cpu().numpy(), status=st)


def check_selection(a: np.ndarray, idx: np.ndarray, count: np.ndarray, k: int, W: int, n_sink: int,
                    heads=None) -> dict:
    """a: oracle scores [B,H,N] (fp64); idx/count: the GPU's tier-1 lists. Returns mismatch statistics."""
    B, H, N = a.shape
    nS = k + W + n_sink
    stats = dict(near_tie_swaps=0, heads=0)
    must = set(range(n_sink)) | set(range(N - W, N))
    for b in range(B):
        for h in (range(H) if heads is None else heads):
            c = int(count[b, h])
            assert c >= nS, (b, h, c, nS)
            sel = idx[b, h, :nS]
            assert np.all(np.diff(sel) > 0), f"ids not strictly ascending at b={b} h={h}"
            assert sel.min() >= 0 and sel.max() < N
            S = set(sel.tolist())
            assert must <= S, f"window/sinks missing at b={b} h={h}"
            arch = np.arange(n_sink, N - W)
            G = np.array(sorted(S - must), dtype=np.int64)
            assert len(G) == k, (b, h, len(G), k)
            if k == 0:
                continue
            sa = a[b, h, arch]
            order = np.lexsort((arch, -sa))
            ref = set(arch[order[:k]].tolist())
            tau = float(sa[order[k - 1]])
            eps = band(tau, sa)
            gmask = np.zeros(N, bool)
            gmask[G] = True
            kept, dropped = a[b, h, G], a[b, h, arch[~gmask[arch]]]
            assert kept.min() >= tau - eps, f"b={b} h={h}: kept row below the threshold band"
            if dropped.size:
                assert dropped.max() <= tau + eps, f"b={b} h={h}: dropped row above the threshold band"
            diff = ref.symmetric_difference(set(G.tolist()))
            for u in diff:
                assert abs(a[b, h, u] - tau) <= eps, f"b={b} h={h} u={u}: differs outside the tie band"
            stats["near_tie_swaps"] += len(diff) // 2
            stats["heads"] += 1
    return stats


def check_outputs(hi: oracle.HostInputs, lam: float, g: dict, idx=None, count=None) -> dict:
    """Oracle attention over the GPU's sets; asserts the output and lse tolerances, returns the max errors."""
    idx = g["idx"] if idx is None else idx
    count = g["count"] if count is None else count
    out, lse, smax = oracle.attention(hi, lam, idx, count)
    num = np.abs(g["out"] - out).max(axis=-1)
    den = np.maximum(np.abs(out).max(axis=-1), 1e-30)
    rel = num / den
    finite = np.isfinite(lse)
    lse_err = np.abs(g["lse"][finite] - lse[finite])
    assert np.all(np.isneginf(g["lse"][~finite])), "an empty set must give lse = -inf"
    assert np.all(rel <= OUT_RTOL), f"max relative output error {rel.max():.3e}"
    assert lse_err.size == 0 or lse_err.max() <= LSE_ATOL, f"max lse error {lse_err.max():.3e}"
    return dict(out_rel=float(rel.max()), lse_abs=float(lse_err.max()) if lse_err.size else 0.0, smax=smax)


def check_fired(a, eta, pres, wl, lam, z_eff, r, smax_ref, S_idx, S_cnt, gF, W, n_sink, top_j=0):
    """Fired sets vs the oracle's trigger rule T = lam (a + |(O qr)[r:]| page_res + z_eff |qc| eta) > s*.

    Exact outside the tie band around s* (and, with top_j, around the top_j-th trigger score); inside a band
    the GPU's choice must still be valid. gF[b][h] is the GPU's fired list. Returns the number of band swaps.
    """
    B, H, N = a.shape
    qr = wl.q_rope.double().cpu().numpy()
    qc_norm = np.linalg.norm(wl.q_latent.double().cpu().numpy(), axis=-1)
    if r < 64:
        qres = np.linalg.norm((qr @ wl.rot.double().cpu().numpy().T)[..., r:], axis=-1)
    else:
        qres = np.zeros((B, H))
    swaps = 0
    for b in range(B):
        for h in range(H):
            inS = np.zeros(N, bool)
            inS[S_idx[b, h, :S_cnt[b, h]]] = True
            u = np.arange(n_sink, N - W)
            u = u[~inS[u]]
            T = lam * (a[b, h, u] + qres[b, h] * pres[b, u // 64] + z_eff * qc_norm[b, h] * eta[b, u])
            Tmap = dict(zip(u.tolist(), T.tolist()))
            s = float(smax_ref[b, h])
            eps_s = band(s, np.array([s]))
            got = list(gF[b][h])
            assert len(set(got)) == len(got), "duplicate fired ids"
            for x in got:
                assert x in Tmap, f"b={b} h={h}: fired row {x} is not an unselected archive row"
                assert Tmap[x] > s - eps_s, f"b={b} h={h} u={x}: fired below s* - band"
            fired = u[T > s]
            if top_j == 0 or len(fired) <= top_j:
                diff = set(fired.tolist()).symmetric_difference(got)
                for x in diff:
                    assert abs(Tmap[x] - s) <= eps_s, f"b={b} h={h} u={x}: T={Tmap[x]} s*={s} outside the band"
                swaps += len(diff)
                if top_j:
                    assert len(got) <= top_j
                continue
            assert len(got) == top_j, (b, h, len(got), top_j)
            Tf = np.sort(T[T > s])[::-1]
            thr = float(Tf[top_j - 1])
            eps_t = band(thr, Tf)
            gotset = set(got)
            for x in got:
                assert Tmap[x] >= thr - eps_t, f"b={b} h={h} u={x}: kept below the top_j cut"
            for x in fired.tolist():
                if x not in gotset:
                    assert Tmap[x] <= thr + eps_t, f"b={b} h={h} u={x}: dropped above the top_j cut"
    return swaps




def check_fired_page(hi, wl, lam, z_eff, smax_ref, S_idx, S_cnt, gF, W, n_sink, top_j=0):
    """Fired sets of the page-level trigger (reading B) vs the oracle's rule: the archived rows outside S_h of every
    page with lam (|qr| max|K| + z_eff |qc| max eta) > s*. Exact outside the tie band around s* (and, with top_j,
    around the top_j-th page bound); inside a band the GPU's choice must still be valid. Returns the band swaps."""
    pk, pe = oracle.page_norms(hi)
    B, H, N = wl.B, wl.H, wl.N
    qrn = np.linalg.norm(wl.q_rope.double().cpu().numpy(), axis=-1)
    qcn = np.linalg.norm(wl.q_latent.double().cpu().numpy(), axis=-1)
    swaps = 0
    for b in range(B):
        for h in range(H):
            inS = np.zeros(N, bool)
            inS[S_idx[b, h, :S_cnt[b, h]]] = True
            u = np.arange(n_sink, N - W)
            u = u[~inS[u]]
            Bp = lam * (qrn[b, h] * pk[b, u // 64] + z_eff * qcn[b, h] * pe[b, u // 64])
            Bmap = dict(zip(u.tolist(), Bp.tolist()))
            s = float(smax_ref[b, h])
            eps_s = band(s, np.array([s]))
            got = list(gF[b][h])
            assert got == sorted(set(got)), "fired ids must be ascending and distinct"
            for x in got:
                assert x in Bmap, f"b={b} h={h}: fired row {x} is not an unselected archive row"
                assert Bmap[x] > s - eps_s, f"b={b} h={h} u={x}: page bound below s* - band"
            fired = u[Bp > s]
            if top_j == 0 or len(fired) <= top_j:
                diff = set(fired.tolist()).symmetric_difference(got)
                for x in diff:
                    assert abs(Bmap[x] - s) <= eps_s, f"b={b} h={h} u={x}: bound {Bmap[x]} s*={s} outside the band"
                swaps += len(diff)
                continue
            assert len(got) == top_j, (b, h, len(got), top_j)
            Bf = np.sort(Bp[Bp > s])[::-1]
            thr = float(Bf[top_j - 1])
            eps_t = band(thr, Bf)
            gotset = set(got)
            for x in got:
                assert Bmap[x] >= thr - eps_t, f"b={b} h={h} u={x}: kept below the top_j cut"
            for x in fired.tolist():
                if x not in gotset:
                    assert Bmap[x] <= thr + eps_t, f"b={b} h={h} u={x}: dropped above the top_j cut"
            # among rows of equal page bound the smaller positions are kept
            strict = [x for x in got if Bmap[x] > thr + eps_t]
            assert len(strict) <= top_j
    return swaps
