"""GPU parity of the PCA digest basis (the appendix's branch-width ablation): vk_pca_basis through the C ABI against
the oracle's fp64 moment and Jacobi eigensolver, and the width-r digest built on that basis through the whole
decode step.

The GPU accumulates the moment from bf16 rows in fp32 per CTA (fp64 across CTAs). By Weyl's inequality a symmetric
perturbation moves every eigenvalue by at most its spectral norm, so eigenvalues are compared at 1e-5 of the largest
one; eigenvectors only where the spectrum separates them (|cos| to the oracle's >= 1 - 1e-4); the retained energy of
every width r at 1e-5 of the total.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_03949_gb300 import datagen
from paper_2609_03949_gb300 import vk

from parity_util import check_selection, GpuStep

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2609_03949_gb300 import _build
    _build.build()
    vk.lib()


def anisotropic_workload(B, N, seed):
    # RoPE keys with a decaying spectrum s_j = 2^(-j/12) in a random orthogonal frame: distinct principal directions
    wl = datagen.make_workload(B, 64, N, seed=seed, n_planted=8, planted_hi=N - 256, device="cuda")
    g = torch.Generator().manual_seed(seed)
    Q = torch.from_numpy(datagen.haar_orthogonal(seed + 1)).float()
    s = torch.pow(2.0, -torch.arange(64, dtype=torch.float32) / 12.0)
    z = torch.randn(B, N, 64, generator=g) * s * 4.0
    wl.cache[:, :, 512:] = (z @ Q.T).to(wl.cache.dtype).cuda()
    return wl


def gpu_basis(wl):
    view = vk.make_view(wl.cache, wl.q_latent, wl.q_rope)
    rot = torch.empty(64, 64, device="cuda")
    eig = torch.empty(64, device="cuda")
    vk.vk_pca_basis(view, rot, eig)
    torch.cuda.synchronize()
    return rot, eig


@pytest.mark.parametrize("B,N", [(1, 5000), (3, 70000)])
def test_pca_basis_matches_oracle(B, N):
    wl = anisotropic_workload(B, N, seed=81 + B)
    rot, eig = gpu_basis(wl)
    R, E = rot.cpu().double().numpy(), eig.cpu().double().numpy()
    hi = oracle.HostInputs(wl)
    ref_eig, ref_rot = oracle.pca_basis(hi)
    assert np.abs(E - ref_eig).max() <= 1e-5 * ref_eig[0], np.abs(E - ref_eig).max() / ref_eig[0]
    np.testing.assert_allclose(R @ R.T, np.eye(64), atol=1e-5)
    gap = np.minimum(np.abs(np.diff(ref_eig, prepend=np.inf)), np.abs(np.diff(ref_eig, append=-np.inf)))
    sep = gap > 1e-2 * ref_eig
    cos = np.abs(np.sum(R * ref_rot, axis=1))
    assert sep.sum() >= 32
    assert np.all(cos[sep] >= 1 - 1e-4), cos[sep].min()
    big = np.abs(R).argmax(axis=1)
    assert np.all(R[np.arange(64), big] > 0)
    K = wl.rope.double().cpu().numpy().reshape(-1, 64)
    for r in (4, 8, 16, 32):
        e = float(((K @ R.T)[:, :r] ** 2).sum())
        assert abs(e - ref_eig[:r].sum()) <= 1e-5 * ref_eig.sum()


@pytest.mark.parametrize("r", [8, 16])
def test_pca_digest_decode_step(r):
    # the PCA basis as the digest rotation, through vk_build_digest and the whole step: the selection meets the oracle
    # run on the same basis (the basis is an input of the digest, like the Haar rotation)
    wl = anisotropic_workload(2, 20000, seed=91 + r)
    rot, _ = gpu_basis(wl)
    wl.rot = rot.cpu()
    hi = oracle.HostInputs(wl)
    _, dig16, _, _ = oracle.build_index(hi, r)
    step = GpuStep(wl, rho=1 / 32, r=r, window=256, digest_bf16=dig16)
    g = step.run()
    assert g["status"] == vk.VK_OK
    a = oracle.scores(hi, r, dig16)
    k = oracle.keep_count(wl.N, 1 / 32, 256)
    check_selection(a, g["idx"], g["count"], k, 256, 0)
    # the GPU's own digest on this basis matches the oracle's to one bf16 ulp plus the fp32 error of its 64-term sum
    # (64 2^-24 sum_j |O_ij K_j|: where the terms nearly cancel, that error can exceed an ulp of the small result)
    dig = torch.empty(2, wl.N, r, dtype=torch.bfloat16, device="cuda")
    vk.vk_build_digest(step.view, step.params, rot, dig)
    d64, _, _, _ = oracle.build_index(hi, r)
    got = dig.float().cpu().double().numpy()
    ulp = np.exp2(np.floor(np.log2(np.maximum(np.abs(d64), 1e-30))) - 7)
    acc = 64 * 2.0 ** -24 * (np.abs(wl.rope.double().cpu().numpy()) @ np.abs(rot.cpu().double().numpy()[:r]).T)
    assert np.all(np.abs(got - d64) <= ulp * 1.0001 + acc)
