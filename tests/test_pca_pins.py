"""Pins for the oracle's PCA digest basis (the appendix's branch-width ablation: principal directions of the RoPE
branch instead of a random rotation): the Jacobi eigensolver against numpy's eigh, the second moment against a
numpy product, an exactly known spectrum, and the energy optimality that makes PCA the best width-r truncation.
A planted mistake (the basis ordered by increasing eigenvalue) must fail a pin."""
import numpy as np
import pytest
import scipy.linalg
import torch

import oracle
from paper_2609_03949_gb300 import datagen


def _hadamard64():
    return scipy.linalg.hadamard(64).astype(np.float64)


def _host(cache):
    t = torch.as_tensor(cache, dtype=torch.float64).to(torch.bfloat16)
    B, N, _ = t.shape
    wl = datagen.Workload(B=B, H=1, N=N, dtype="bf16", cache=t, q_latent=torch.zeros(B, 1, 512, dtype=torch.bfloat16),
                          q_rope=torch.zeros(B, 1, 64, dtype=torch.bfloat16), rot=torch.eye(64),
                          planted_pos=torch.zeros(B, 0, dtype=torch.int64), planted_head=torch.zeros(0, dtype=torch.int64),
                          seed=0)
    return oracle.HostInputs(wl), wl


def pin_sym_eig_matches_numpy():
    rng = np.random.default_rng(3)
    for _ in range(3):
        X = rng.standard_normal((200, 64))
        M = X.T @ X
        eig, vec = oracle.sym_eig(M)
        w, U = np.linalg.eigh(M)
        np.testing.assert_allclose(eig, w[::-1], rtol=1e-10)
        dots = np.abs(np.sum(vec * U[:, ::-1].T, axis=1))
        np.testing.assert_allclose(dots, 1.0, atol=1e-8)
        np.testing.assert_allclose(vec.T @ np.diag(eig) @ vec, M, atol=1e-9 * np.abs(M).max())
        np.testing.assert_allclose(vec @ vec.T, np.eye(64), atol=1e-12)
        big = np.abs(vec).argmax(axis=1)
        assert np.all(vec[np.arange(64), big] > 0)     # each eigenvector's largest entry is positive


def pin_second_moment_matmul():
    wl = datagen.make_workload(2, 4, 700, seed=5)
    hi = oracle.HostInputs(wl)
    K = wl.rope.double().numpy().reshape(-1, 64)
    np.testing.assert_allclose(oracle.second_moment(hi), K.T @ K, rtol=1e-12)


def pin_pca_known_axes():
    # rows s_i h_i / 8 (Hadamard rows, exact in bf16): M = sum s_i^2 h_i h_i^T / 64, eigenpairs (s_i^2, h_i / 8)
    H = _hadamard64()
    s = np.arange(1, 65, dtype=np.float64)
    perm = np.random.default_rng(0).permutation(64)
    cache = np.zeros((1, 64, 576))
    cache[0, :, 512:] = (s[perm, None] * H[perm]) / 8.0
    hi, _ = _host(cache)
    eig, rot = oracle.pca_basis(hi)
    np.testing.assert_allclose(eig, (s[::-1] ** 2), rtol=1e-12)
    for i in range(64):
        want = H[63 - i] / 8.0                         # up to sign: all its entries tie in magnitude
        np.testing.assert_allclose(abs(float(rot[i] @ want)), 1.0, atol=1e-12)
        np.testing.assert_allclose(np.abs(rot[i]), np.abs(want), atol=1e-12)


def pin_pca_energy_optimal():
    # the first r principal coordinates keep sum_{j<r} lambda_j of the branch energy, at least as much as the first
    # r coordinates after any other rotation (here Haar draws)
    wl = datagen.make_workload(1, 4, 3000, seed=9)
    hi = oracle.HostInputs(wl)
    eig, rot = oracle.pca_basis(hi)
    K = wl.rope.double().numpy().reshape(-1, 64)
    Y = K @ rot.T
    for r in (4, 8, 16, 32):
        e_pca = float((Y[:, :r] ** 2).sum())
        np.testing.assert_allclose(e_pca, eig[:r].sum(), rtol=1e-9)
        for seed in range(3):
            O = datagen.haar_orthogonal(seed)
            assert e_pca >= float(((K @ O.T)[:, :r] ** 2).sum())


def pin_sym_eig_spread_repeated_zero():
    # a spectrum over seven decades, a spectrum of three repeated values, and the zero matrix, each in a Haar frame:
    # eigenvalues to the rounding of the largest; for a repeated value only its eigenspace is fixed, so the
    # eigenvectors' projector is compared with the frame's
    Q = datagen.haar_orthogonal(11)
    spread = np.logspace(3, -4, 64)
    eig, vec = oracle.sym_eig((Q.T * spread) @ Q)
    np.testing.assert_allclose(eig, spread, rtol=1e-9, atol=1e-12 * spread[0])
    np.testing.assert_allclose(vec @ vec.T, np.eye(64), atol=1e-12)
    sep = np.abs(vec @ Q.T)                            # row i against the frame's row i: |cos| = 1 where separated
    np.testing.assert_allclose(np.diag(sep)[:40], 1.0, atol=1e-9)
    rep = np.repeat([5.0, 2.0, 1.0], [16, 16, 32])
    eig, vec = oracle.sym_eig((Q.T * rep) @ Q)
    np.testing.assert_allclose(eig, rep, rtol=1e-12)
    for lo, hi_ in ((0, 16), (16, 32), (32, 64)):
        P_got = vec[lo:hi_].T @ vec[lo:hi_]
        P_want = Q[lo:hi_].T @ Q[lo:hi_]
        np.testing.assert_allclose(P_got, P_want, atol=1e-10)
    eig, vec = oracle.sym_eig(np.zeros((64, 64)))
    assert np.all(eig == 0.0)
    np.testing.assert_allclose(vec @ vec.T, np.eye(64), atol=1e-12)
    big = np.abs(vec).argmax(axis=1)
    assert np.all(vec[np.arange(64), big] > 0)


PINS = [pin_sym_eig_matches_numpy, pin_sym_eig_spread_repeated_zero, pin_second_moment_matmul, pin_pca_known_axes,
        pin_pca_energy_optimal]


@pytest.mark.parametrize("pin", PINS, ids=lambda f: f.__name__)
def test_pin(pin):
    oracle.set_mutation(oracle.MUT_NONE)
    pin()


@pytest.mark.parametrize("pin", [pin_pca_known_axes, pin_pca_energy_optimal])
def test_planted_mistake_is_caught(pin):
    oracle.set_mutation(oracle.MUT_PCA_ASCENDING)
    try:
        with pytest.raises(AssertionError):
            pin()
    finally:
        oracle.set_mutation(oracle.MUT_NONE)
