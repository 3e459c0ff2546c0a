"""Pins for the oracle's sigma selector (Sec. 4.1, Eq. 3; Corollary 1), independent of the oracle itself.

sigma_u is the norm of row u's RoPE branch minus its low-pass reconstruction over a fixed block of T rows
(sequence-axis DFT kept on bins [0, kappa)). The oracle writes the DFT's defining sums out; these pins check it
against numpy's FFT (a library routine), closed forms for pure tones and constants, the projection property,
block independence, hand cases of the top-m rule, and Corollary 1 (a streaming top-m maintained as blocks close
equals the one-shot top-m). One planted mistake in the oracle must be caught.
"""
import heapq

import numpy as np
import pytest

import oracle

TOL = 1e-9


def sigma_numpy(r, T, kappa):
    """The same residual through numpy's real FFT: keep bins [0, kappa) of each closed block, invert, subtract."""
    N = r.shape[0]
    out = np.full(N, -1.0)
    for j in range(N // T):
        blk = r[j * T:(j + 1) * T]
        spec = np.fft.rfft(blk, axis=0)
        spec[min(kappa, spec.shape[0]):] = 0
        low = np.fft.irfft(spec, n=T, axis=0)
        out[j * T:(j + 1) * T] = np.linalg.norm(blk - low, axis=1)
    return out


@pytest.mark.parametrize("T,kappa,N", [(64, 1, 200), (64, 4, 128), (256, 16, 3 * 256 + 17), (128, 64, 300),
                                       (128, 65, 256), (60, 7, 130)])
def test_sigma_matches_numpy_fft(T, kappa, N):
    rng = np.random.default_rng(T * 1000 + kappa)
    r = rng.standard_normal((N, 64))
    got = oracle.sigma(r, T=T, kappa=kappa)
    want = sigma_numpy(r, T, kappa)
    np.testing.assert_allclose(got, want, rtol=TOL, atol=TOL)
    assert np.all(got[(N // T) * T:] == -1.0)          # the open tail has no sigma


def test_all_bins_kept_gives_zero():
    # kappa past the Nyquist bin keeps the whole spectrum: the reconstruction is the block itself
    rng = np.random.default_rng(1)
    for T in (64, 63):
        r = rng.standard_normal((2 * T, 64))
        s = oracle.sigma(r, T=T, kappa=T // 2 + 1)
        assert np.abs(s).max() < 1e-9 * np.abs(r).max() * 8


@pytest.mark.parametrize("k0,kappa", [(3, 4), (3, 3), (10, 16), (20, 16), (31, 8)])
def test_pure_tone_closed_form(k0, kappa):
    # one dim holds a cos(2 pi k0 u / T + phi): inside the band it is reconstructed exactly (sigma = 0); outside
    # the band (0 < k0 < T/2) it is removed whole, so sigma_u = |a cos(2 pi k0 u / T + phi)|
    T, a, phi = 64, 2.5, 0.7
    u = np.arange(2 * T)
    r = np.zeros((2 * T, 64))
    r[:, 5] = a * np.cos(2 * np.pi * k0 * (u % T) / T + phi)
    s = oracle.sigma(r, T=T, kappa=kappa)
    want = np.zeros(2 * T) if k0 < kappa else np.abs(r[:, 5])
    np.testing.assert_allclose(s, want, atol=1e-10)


def test_constant_rows_have_zero_sigma():
    r = np.tile(np.linspace(-3, 3, 64), (128, 1))
    for kappa in (1, 16):
        assert np.abs(oracle.sigma(r, T=64, kappa=kappa)).max() < 1e-10


def test_in_band_signal_leaves_sigma_unchanged():
    # the residual is a projection: adding any signal made of kept bins does not move it
    rng = np.random.default_rng(2)
    T, kappa = 128, 8
    r = rng.standard_normal((2 * T, 64))
    u = np.arange(2 * T) % T
    band = sum(rng.standard_normal(64)[None, :] * np.cos(2 * np.pi * k * u / T + rng.uniform(0, 6))[:, None]
               for k in range(kappa))
    np.testing.assert_allclose(oracle.sigma(r + band, T=T, kappa=kappa), oracle.sigma(r, T=T, kappa=kappa),
                               rtol=1e-9, atol=1e-9)


def test_blocks_are_independent():
    # each block is transformed once, on its own rows: changing another block leaves it exactly as it was
    rng = np.random.default_rng(3)
    T = 64
    r = rng.standard_normal((3 * T + 10, 64))
    s0 = oracle.sigma(r, T=T, kappa=4)
    r2 = r.copy()
    r2[T:2 * T] *= 3.0
    r2[3 * T:] = 7.0
    s1 = oracle.sigma(r2, T=T, kappa=4)
    assert np.array_equal(s0[:T], s1[:T]) and np.array_equal(s0[2 * T:3 * T], s1[2 * T:3 * T])
    assert not np.allclose(s0[T:2 * T], s1[T:2 * T])


def test_select_hand_cases():
    T, N = 16, 3 * 16 + 5
    tail = list(range(48, N))
    # sigma rising with position: the top-m closed rows are the last m of the closed range
    sig = np.concatenate([np.arange(48, dtype=float), -np.ones(5)])
    ids = oracle.sigma_select(sig, T, n_sink=4, m=6).tolist()
    assert ids == [0, 1, 2, 3] + list(range(42, 48)) + tail
    # all equal: ties go to the smaller positions after the sinks
    ids = oracle.sigma_select(np.concatenate([np.ones(48), -np.ones(5)]), T, n_sink=4, m=6).tolist()
    assert ids == [0, 1, 2, 3] + list(range(4, 10)) + tail
    # m beyond the closed rows outside the sinks: everything is attended
    assert oracle.sigma_select(sig, T, n_sink=4, m=1000).tolist() == list(range(N))
    # no sinks, m = 0: only the open tail
    assert oracle.sigma_select(sig, T, n_sink=0, m=0).tolist() == tail


def test_streaming_top_m_equals_one_shot():
    # Corollary 1: sigma is row-intrinsic, so a global top-m kept incrementally as blocks close (later rows
    # displacing earlier ones) ends equal to the top-m computed once at the end
    rng = np.random.default_rng(4)
    T, nb, n_sink, m = 32, 9, 4, 40
    N = nb * T + 11
    sig = np.round(rng.standard_normal(N) * 2) / 2          # coarse values: many ties
    sig[nb * T:] = -1.0
    heap = []                                               # min-heap of the kept rows, worst first
    for j in range(nb):
        for u in range(j * T, (j + 1) * T):
            if u < n_sink:
                continue
            key = (sig[u], -u)                              # larger sigma, then smaller position, is better
            if len(heap) < m:
                heapq.heappush(heap, key)
            elif key > heap[0]:
                heapq.heapreplace(heap, key)
    streamed = sorted(set(range(n_sink)) | {-k[1] for k in heap} | set(range(nb * T, N)))
    assert oracle.sigma_select(sig, T, n_sink=n_sink, m=m).tolist() == streamed


def test_planted_one_sided_inverse_is_caught():
    rng = np.random.default_rng(5)
    r = rng.standard_normal((128, 64))
    oracle.set_mutation(oracle.MUT_SIGMA_ONE_SIDED)
    try:
        bad = oracle.sigma(r, T=64, kappa=8)
    finally:
        oracle.set_mutation(oracle.MUT_NONE)
    assert not np.allclose(bad, sigma_numpy(r, 64, 8), rtol=TOL, atol=TOL)
    np.testing.assert_allclose(oracle.sigma(r, T=64, kappa=8), sigma_numpy(r, 64, 8), rtol=TOL, atol=TOL)
