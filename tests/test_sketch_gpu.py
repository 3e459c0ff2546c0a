"""GPU parity of the rank-r_sk content sketch (Sec. 4.2, Eq. 4, Lemma 1) through the C ABI against the oracle.

* vk_build_sketch: every stored entry within one bf16 ulp of the oracle's (plus the fp32 rounding of a 512-term sum
  that cancels), the residual norms within 1e-5 relative (plus the same cancellation term).
* vk_sketch_basis: the leading directions that the queries' spectrum separates (the query law's rank) as a subspace
  (projector distance 1e-3) with their eigenvalues within 1e-4; the whole basis orthonormal to 1e-5; its captured
  second-moment energy within 1e-4 of the oracle's optimum.
* The decode step's trigger with the sketch (tensor-core scan at r = 64 for H = 64 and 128, the dense scan with a
  digest width or VK_FLAG_FORCE_DENSE): fired rows equal to the oracle's rule T = lam (a + |(O Qr)[r:]| page_res +
  p . s + z_eff rho eta) > s* outside the 1e-3 band around s* (and around the top_j-th score), and outputs over S u F
  within the step's tolerances. Both sides score the oracle's stored sketch and residual norms.
"""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2609_03949_gb300 import datagen
from paper_2609_03949_gb300 import vk

from parity_util import GpuStep, band, check_outputs, check_selection

pytestmark = pytest.mark.gpu
LAM = vk.DEFAULT_SM_SCALE
ULP = 2.0 ** -8


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2609_03949_gb300 import _build
    _build.build()
    vk.lib()


def sketch_workload(B, H, N, seed, query_rank=8, planted_frac=3):
    """Low-rank-plus-noise queries and, for every planted_frac-th head, a row whose latent part points along the
    head's content query (its logit dominates, its RoPE score is ordinary: the trigger must bring it back)."""
    wl = datagen.make_workload(B, H, N, seed=seed, n_planted=0, query_rank=query_rank)
    rng = np.random.default_rng(seed)
    for b in range(B):
        for h in range(0, H, planted_frac):
            u = int(rng.integers(0, N - 512))
            qc = wl.q_latent[b, h].float()
            wl.cache[b, u, :512] = (3.0 * qc / qc.norm()).to(wl.cache.dtype)
    return wl


def bf16_value(bits: np.ndarray) -> np.ndarray:
    return (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


@pytest.mark.parametrize("r_sk", [16, 32, 64])
def test_build_sketch_matches_oracle(r_sk):
    wl = sketch_workload(2, 4, 1536, seed=40 + r_sk)
    hi = oracle.HostInputs(wl)
    V, _ = oracle.sketch_basis(datagen.prefix_queries(wl, 200).double().numpy(), r_sk)
    s, s16, eta = oracle.build_sketch(hi, V)
    d = wl.to("cuda")
    view = vk.make_view(d.cache, d.q_latent, d.q_rope)
    basis = torch.as_tensor(V, dtype=torch.float32).cuda()
    sk = torch.empty(2, 1536, r_sk, dtype=torch.bfloat16, device="cuda")
    eg = torch.empty(2, 1536, dtype=torch.float32, device="cuda")
    vk.vk_build_sketch(view, r_sk, basis, sk, eg)
    torch.cuda.synchronize()
    got = sk.float().double().cpu().numpy()
    L = wl.latent.double().numpy()
    # fp32 products and sums over 512 terms: the cancellation bound of |V_j| |L_u| (|V_j| = 1), then one bf16 rounding
    lnorm = np.linalg.norm(L, axis=-1)
    tol = ULP * np.abs(s) + 64 * 2.0 ** -24 * lnorm[..., None] * math.sqrt(512)
    assert np.all(np.abs(got - s) <= tol), float(np.max(np.abs(got - s) / tol))
    # on most entries the two roundings agree exactly
    assert np.mean(got == bf16_value(s16)) > 0.99
    e = eg.double().cpu().numpy()
    assert np.all(np.abs(e - eta) <= 1e-5 * eta + 64 * 2.0 ** -24 * lnorm), float(np.max(np.abs(e - eta)))


@pytest.mark.parametrize("r_sk,n", [(16, 300), (32, 400), (64, 300)])
def test_sketch_basis_matches_oracle(r_sk, n):
    k_true = 8                                        # the query law's rank: its directions stand out of the noise
    wl = datagen.make_workload(1, 4, 64, seed=50 + r_sk, query_rank=k_true)
    q = datagen.prefix_queries(wl, n)
    qd = q.double().numpy()
    M = qd.T @ qd
    w = np.linalg.eigvalsh(M)[::-1]
    Vo, eo = oracle.sketch_basis(qd, k_true)          # the separated directions
    basis = torch.empty(r_sk, 512, dtype=torch.float32, device="cuda")
    eig = torch.empty(r_sk, dtype=torch.float32, device="cuda")
    ws = vk.vk_sketch_basis(q.cuda().contiguous(), r_sk, basis, eig)
    torch.cuda.synchronize()
    assert vk.vk_poll_status(ws) == vk.VK_OK
    Vg = basis.double().cpu().numpy()
    eg = eig.double().cpu().numpy()
    assert np.abs(Vg @ Vg.T - np.eye(r_sk)).max() <= 1e-5
    np.testing.assert_allclose(eg[:k_true], eo, rtol=1e-4)
    Pg = Vg[:k_true].T @ Vg[:k_true]
    Po = Vo.T @ Vo
    assert np.abs(Pg - Po).max() <= 1e-3
    captured = np.trace(Vg @ M @ Vg.T)
    assert captured >= (1 - 1e-4) * w[:r_sk].sum()
    # the sign rule on every returned direction
    big = np.argmax(np.abs(Vg), axis=1)
    assert np.all(Vg[np.arange(r_sk), big] > 0)


def check_fired_sketch(sub, z_eff, r, a, pres, shat, p, rho, eta, smax, gF, S_idx, S_cnt, W, n_sink, top_j):
    """The GPU's fired lists gF[b][h] against the row-level rule with the sketch term; returns the band swaps."""
    B, H, N = a.shape
    qr = sub.q_rope.double().cpu().numpy()
    qres = (np.linalg.norm((qr @ sub.rot.double().cpu().numpy().T)[..., r:], axis=-1) if r < 64
            else np.zeros((B, H)))
    swaps = 0
    for b in range(B):
        for h in range(H):
            inS = np.zeros(N, bool)
            inS[S_idx[b, h, :S_cnt[b, h]]] = True
            u = np.arange(n_sink, N - W)
            u = u[~inS[u]]
            T = LAM * (a[b, h, u] + qres[b, h] * pres[b, u // 64] + shat[b, u] @ p[b, h] + z_eff * rho[b, h] * eta[b, u])
            Tm = dict(zip(u.tolist(), T.tolist()))
            s = float(smax[b, h])
            eps = band(s, np.array([s]))
            got = list(gF[b][h])
            assert len(set(got)) == len(got)
            for x in got:
                assert x in Tm and Tm[x] > s - eps, (b, h, x)
            fired = u[T > s]
            if top_j == 0 or len(fired) <= top_j:
                diff = set(fired.tolist()).symmetric_difference(got)
                for x in diff:
                    assert abs(Tm[x] - s) <= eps, (b, h, x, Tm[x], s)
                swaps += len(diff)
                continue
            assert len(got) == top_j
            Tf = np.sort(T[T > s])[::-1]
            thr = float(Tf[top_j - 1])
            eps_t = band(thr, Tf)
            for x in got:
                assert Tm[x] >= thr - eps_t
            for x in set(fired.tolist()) - set(got):
                assert Tm[x] <= thr + eps_t
    return swaps


def run_sketch_case(wl, *, r_sk, rho_keep=1 / 32, window=128, z_eff=1.0, top_j=0, r=64, flags=0, n_prefix=200):
    hi = oracle.HostInputs(wl)
    V, _ = oracle.sketch_basis(datagen.prefix_queries(wl, n_prefix).double().numpy(), r_sk)
    _, s16, eta = oracle.build_sketch(hi, V)
    p, rho = oracle.sketch_query(hi, V)
    dig16 = oracle.build_index(hi, r)[1] if r < 64 else None
    g = GpuStep(wl, rho=rho_keep, r=r, window=window, trigger=vk.VK_TRIG_CS, z_eff=z_eff, top_j=top_j, flags=flags,
                digest_bf16=dig16, sketch=(s16, V, eta)).run()
    assert g["status"] == vk.VK_OK
    a = oracle.scores(hi, r, dig16)
    k = oracle.keep_count(wl.N, rho_keep, window)
    nS = k + window
    check_selection(a, g["idx"], g["count"], k, window, 0)
    Sc = np.full_like(g["count"], nS)
    _, _, smax = oracle.attention(hi, LAM, g["idx"][..., :nS], Sc)
    np.testing.assert_allclose(g["smax"], smax, rtol=1e-4, atol=1e-4)
    pres = oracle.build_index(hi, r)[3]
    gF = [[g["idx"][b, h, nS:g["count"][b, h]].tolist() for h in range(wl.H)] for b in range(wl.B)]
    swaps = check_fired_sketch(wl, z_eff, r, a, pres, bf16_value(s16), p, rho, eta, smax, gF, g["idx"], Sc, window, 0,
                               top_j)
    check_outputs(hi, LAM, g)
    return int((g["count"] - nS).sum()), swaps


@pytest.mark.parametrize("H,r_sk,z_eff,top_j", [(64, 64, 1.0, 0), (128, 64, 1.0, 0), (64, 32, 0.3, 0),
                                                (128, 16, 0.3, 0), (64, 64, 1.0, 8)])
def test_sketch_trigger_tensor_cores(H, r_sk, z_eff, top_j):
    wl = sketch_workload(2, H, 8192, seed=60 + H + r_sk)
    fired, swaps = run_sketch_case(wl, r_sk=r_sk, z_eff=z_eff, top_j=top_j)
    assert fired > 0                                  # the planted rows come back
    assert swaps <= max(2, fired // 100)


@pytest.mark.parametrize("r,flags", [(16, 0), (64, vk.VK_FLAG_FORCE_DENSE)])
def test_sketch_trigger_dense_scan(r, flags):
    wl = sketch_workload(2, 32, 4096, seed=70 + r)
    fired, swaps = run_sketch_case(wl, r_sk=32, r=r, flags=flags, z_eff=0.5)
    assert fired > 0
    assert swaps <= max(2, fired // 100)


def test_sketch_tightens_the_gpu_trigger():
    """At the sound z_eff = 1 the sketch's certificate is far smaller than |qc| |L|: far fewer rows fire than at sketch
    rank 0, and the planted rows still do."""
    wl = sketch_workload(2, 64, 8192, seed=81)
    f_sk, _ = run_sketch_case(wl, r_sk=64)
    g0 = GpuStep(wl, rho=1 / 32, window=128, trigger=vk.VK_TRIG_CS, z_eff=1.0).run()
    nS = oracle.keep_count(8192, 1 / 32, 128) + 128
    f0 = int((g0["count"] - nS).sum())
    assert f_sk < 0.5 * f0, (f_sk, f0)


def test_sketch_fp32_cache():
    """fp32 caches: materialised scores, the dense trigger scan with the sketch term, the fp32 per-head fired pass."""
    wl = datagen.make_workload(1, 16, 2048, dtype="f32", seed=91, n_planted=0, query_rank=8)
    rng = np.random.default_rng(91)
    for h in range(0, 16, 3):
        u = int(rng.integers(0, 1400))
        qc = wl.q_latent[0, h].float()
        wl.cache[0, u, :512] = 3.0 * qc / qc.norm()
    fired, swaps = run_sketch_case(wl, r_sk=32, window=64, rho_keep=1 / 16, z_eff=0.5)
    assert fired > 0
    assert swaps <= max(2, fired // 100)


def test_sketch_256_heads_dense_scan():
    """More than 128 heads with a sketch: the step materialises the scores and the dense scan adds the sketch term."""
    wl = sketch_workload(1, 256, 4096, seed=93, planted_frac=5)
    fired, swaps = run_sketch_case(wl, r_sk=64, z_eff=0.5)
    assert fired > 0
    assert swaps <= max(2, fired // 100)


@pytest.mark.parametrize("r,top_j", [(16, 5), (64, 3)])
def test_sketch_top_j(r, top_j):
    wl = sketch_workload(2, 64, 4096, seed=95 + r)
    fired, _ = run_sketch_case(wl, r_sk=32, r=r, z_eff=0.3, top_j=top_j)
    assert 0 < fired <= 2 * 64 * top_j
