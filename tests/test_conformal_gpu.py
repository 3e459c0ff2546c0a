"""GPU parity of the conformal calibration of the trigger's z (Sec. 4.2; Sec. 5): vk_conformal_z through the C ABI
against the oracle's vko_calib_zq and vko_conformal_quantile, on the GPU's own tier-1 sets.

The workload plants, for a third of the (b, h) queries, a row whose latent part points along the head's content query:
its logit dominates, but its RoPE score is ordinary, so tier 1 leaves it out and the query is hard. Hardness must
match the oracle wherever the best in-set and best out-of-set logits are apart by more than 1e-3 relative; zq within
2e-3 + 1e-3 |zq| (fp32 logits, the difference s* - idx_t over the certificate); z is the order statistic of the GPU's
own zq exactly, and the oracle's within the same tolerance.
"""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2609_03949_gb300 import datagen
from paper_2609_03949_gb300 import vk

from parity_util import GpuStep

pytestmark = pytest.mark.gpu
LAM = vk.DEFAULT_SM_SCALE


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2609_03949_gb300 import _build
    _build.build()
    vk.lib()


def content_planted(B, H, N, seed):
    wl = datagen.make_workload(B, H, N, seed=seed, n_planted=0, device="cuda")
    rng = np.random.default_rng(seed)
    for b in range(B):
        for h in range(0, H, 3):
            u = int(rng.integers(0, N - 512))
            qc = wl.q_latent[b, h].float()
            wl.cache[b, u, :512] = (3.0 * qc / qc.norm()).to(wl.cache.dtype)
    return wl


@pytest.mark.parametrize("r,z_max", [(64, 100.0), (16, 100.0), (64, 8.0)])
def test_conformal_z_matches_oracle(r, z_max):
    B, H, N, W = 2, 64, 8192, 256
    wl = content_planted(B, H, N, seed=101 + r)
    hi = oracle.HostInputs(wl)
    dig16 = None
    if r < 64:
        _, dig16, _, _ = oracle.build_index(hi, r)
    step = GpuStep(wl, rho=1 / 32, r=r, window=W, digest_bf16=dig16)
    g = step.run()
    assert g["status"] == vk.VK_OK
    zq = torch.empty(B, H, device="cuda")
    z_out = torch.empty(3, device="cuda")
    ws = vk.vk_conformal_z(step.view, step.params, step.index, step.buf.idx, step.buf.count, zq, z_out, tau=0.9,
                           z_max=z_max)
    torch.cuda.synchronize()
    assert vk.vk_poll_status(ws) == vk.VK_OK
    gz = zq.cpu().double().numpy()
    zo = z_out.cpu().double().numpy()

    a = oracle.scores(hi, r, dig16)
    _, _, eta, pres = oracle.build_index(hi, r)
    rzq, ustar, n_ref = oracle.calib_zq(hi, r, LAM, a, eta, pres, g["idx"], g["count"])
    # the margin that decides hardness, from exact logits
    L, K = wl.latent.double().cpu().numpy(), wl.rope.double().cpu().numpy()
    s = LAM * (np.einsum("bhj,bnj->bhn", wl.q_latent.double().cpu().numpy(), L) +
               np.einsum("bhj,bnj->bhn", wl.q_rope.double().cpu().numpy(), K))
    checked = 0
    for b in range(B):
        for h in range(H):
            inS = np.zeros(N, bool)
            inS[g["idx"][b, h, :g["count"][b, h]]] = True
            best_in, best_out = s[b, h, inS].max(), s[b, h, ~inS].max()
            if abs(best_in - best_out) <= 1e-3 * max(abs(best_in), abs(best_out)):
                continue
            checked += 1
            assert np.isnan(gz[b, h]) == np.isnan(rzq[b, h]), (b, h)
            if not np.isnan(rzq[b, h]):
                assert abs(gz[b, h] - rzq[b, h]) <= 2e-3 + 1e-3 * abs(rzq[b, h]), (b, h, gz[b, h], rzq[b, h])
    assert checked >= B * H - 4
    hard = ~np.isnan(gz)
    assert zo[2] == hard.sum() >= oracle.min_hard(0.9)
    assert zo[0] == pytest.approx(oracle.conformal_quantile(gz[hard], 0.9, z_max), abs=1e-6)
    assert zo[0] == pytest.approx(oracle.conformal_quantile(rzq[~np.isnan(rzq)], 0.9, z_max), abs=2e-3 + 1e-3 * zo[0])
    assert zo[1] == pytest.approx(zo[0] / math.sqrt(512.0), rel=1e-6)


@pytest.mark.parametrize("r_sk", [16, 64])
def test_conformal_z_with_sketch(r_sk):
    """Calibration with the rank-r_sk sketch certificate: queries of rank 8 plus noise; for a third of the heads a row
    along the query's residual outside the basis span (only the certificate can bring it back), so those are hard."""
    B, H, N, W = 2, 64, 8192, 256
    wl = datagen.make_workload(B, H, N, seed=111 + r_sk, n_planted=0, query_rank=8)
    V, _ = oracle.sketch_basis(datagen.prefix_queries(wl, 200).double().numpy(), r_sk)
    rng = np.random.default_rng(r_sk)
    for b in range(B):
        for h in range(0, H, 3):
            qc = wl.q_latent[b, h].double().numpy()
            res = qc - V.T @ (V @ qc)
            u = int(rng.integers(0, N - 512))
            wl.cache[b, u, :512] = torch.as_tensor(12.0 * res / np.linalg.norm(res)).to(wl.cache.dtype)
    hi = oracle.HostInputs(wl)
    _, s16, eta = oracle.build_sketch(hi, V)
    p, rho = oracle.sketch_query(hi, V)
    # tier 1 without the trigger; the sketch index rides along for the calibration
    step = GpuStep(wl, rho=1 / 32, window=W)
    g = step.run()
    assert g["status"] == vk.VK_OK
    sk = torch.from_numpy(s16.astype(np.int16)).view(torch.bfloat16).cuda().contiguous()
    basis = torch.as_tensor(V, dtype=torch.float32).cuda().contiguous()
    eta_g = torch.as_tensor(eta, dtype=torch.float32).cuda().contiguous()
    index = vk.make_index(None, eta_g, step.page_res, None, None, None, sk, basis)
    params = vk.make_params(1 / 32, window=W, trigger=vk.VK_TRIG_CS, r_sk=r_sk)
    zq = torch.empty(B, H, device="cuda")
    z_out = torch.empty(3, device="cuda")
    ws = vk.vk_conformal_z(step.view, params, index, step.buf.idx, step.buf.count, zq, z_out, tau=0.9, z_max=100.0)
    torch.cuda.synchronize()
    assert vk.vk_poll_status(ws) == vk.VK_OK
    gz = zq.cpu().double().numpy()
    zo = z_out.cpu().double().numpy()
    a = oracle.scores(hi)
    pres = oracle.build_index(hi, 64)[3]
    rzq, _, n_ref = oracle.calib_zq(hi, 64, LAM, a, eta, pres, g["idx"], g["count"], sketch=(s16, p, rho))
    hard = ~np.isnan(rzq)
    assert hard.sum() >= oracle.min_hard(0.9)
    np.testing.assert_array_equal(np.isnan(gz), np.isnan(rzq))
    np.testing.assert_allclose(gz[hard], rzq[hard], rtol=1e-3, atol=2e-3)
    assert zo[2] == hard.sum()
    assert zo[0] == pytest.approx(oracle.conformal_quantile(rzq[hard], 0.9, 100.0), abs=2e-3 + 1e-3 * zo[0])
    assert zo[1] == pytest.approx(zo[0] / math.sqrt(512.0 - r_sk), rel=1e-6)
