"""Pins of the oracle's rank-r_sk content sketch (Sec. 4.2, Eq. 4, Lemma 1) against facts other than itself.

* The basis from queries against numpy's symmetric eigensolver on their second moment (a library routine on a
  special case), and an exactly known spectrum built from orthonormal frames.
* The index entry against Pythagoras (|s_u|^2 + eta_u^2 = |L_u|^2 for any orthonormal basis) and against rows built
  inside and orthogonal to the basis's span.
* The query side against the same identity and against rank 0 (rho = |qc|).
* The trigger against a hand case whose trigger score is worked out by hand, just above and just below s*, and
  against Lemma 1 itself: with the sound multiplier z_eff = 1, every row whose exact logit beats s* (by more than the
  bf16 rounding of its stored sketch can hide) fires.
* The decode step with a sketch against the row-level trigger composed by hand from the pinned pieces.

A planted mistake (the certificate keeping |qc| instead of the residual norm) fails the hand case.
"""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2609_03949_gb300 import datagen

LAM = 1.0 / math.sqrt(192.0)


def _f32_workload(latent: np.ndarray, qc: np.ndarray, qr: np.ndarray | None = None, krope: np.ndarray | None = None):
    """A fp32 workload from explicit rows (latent [B,N,512]) and queries (qc [B,H,512])."""
    B, N, _ = latent.shape
    H = qc.shape[1]
    cache = np.zeros((B, N, 576))
    cache[..., :512] = latent
    if krope is not None:
        cache[..., 512:] = krope
    qr = np.zeros((B, H, 64)) if qr is None else qr
    wl = datagen.Workload(B=B, H=H, N=N, dtype="f32", cache=torch.as_tensor(cache, dtype=torch.float32),
                          q_latent=torch.as_tensor(qc, dtype=torch.float32),
                          q_rope=torch.as_tensor(qr, dtype=torch.float32), rot=torch.eye(64),
                          planted_pos=torch.zeros(B, 0, dtype=torch.int64),
                          planted_head=torch.zeros(0, dtype=torch.int64), seed=0)
    return oracle.HostInputs(wl), wl


def pin_basis_matches_eigh():
    wl = datagen.make_workload(1, 4, 64, seed=11, query_rank=12)
    q = datagen.prefix_queries(wl, 200).double().numpy()
    r_sk = 16
    vb, eig = oracle.sketch_basis(q, r_sk)
    w, V = np.linalg.eigh(q.T @ q)                    # ascending
    w, V = w[::-1][:r_sk], V[:, ::-1][:, :r_sk].T
    assert np.allclose(eig, w, rtol=1e-9, atol=1e-9 * w[0])
    gaps = np.abs(np.diff(w))
    for i in range(r_sk):
        sep = min(gaps[i - 1] if i > 0 else np.inf, gaps[i] if i < r_sk - 1 else np.inf)
        if sep > 1e-6 * w[0]:
            assert abs(abs(vb[i] @ V[i]) - 1.0) < 1e-8, i
    assert np.allclose(vb @ vb.T, np.eye(r_sk), atol=1e-10)
    big = np.argmax(np.abs(vb), axis=1)
    assert np.all(vb[np.arange(r_sk), big] > 0)       # the sign rule


def pin_basis_known_spectrum():
    # queries sqrt(lambda_i) f_i for an orthonormal frame f: the second moment is sum_i lambda_i f_i f_i^T exactly
    F = datagen.haar_orthogonal(5, 512)[:6]
    lam = np.array([9.0, 7.5, 4.0, 2.0, 1.0, 0.25])
    q = np.sqrt(lam)[:, None] * F
    vb, eig = oracle.sketch_basis(q, 4)
    assert np.allclose(eig, lam[:4], rtol=1e-12)
    for i in range(4):
        assert abs(abs(vb[i] @ F[i]) - 1.0) < 1e-12
    with pytest.raises(ValueError):
        oracle.sketch_basis(q, 7)                      # six queries span six directions


def pin_basis_direct_route():
    # at least 512 queries: the eigensolver runs on the 512 x 512 moment itself (about 15 s of CPU)
    F = datagen.haar_orthogonal(6, 512)
    lam = np.linspace(10.0, 0.5, 512)
    q = (np.random.default_rng(0).standard_normal((520, 512)) * np.sqrt(lam)) @ F
    vb, eig = oracle.sketch_basis(q, 4)
    w, V = np.linalg.eigh(q.T @ q)
    assert np.allclose(eig, w[::-1][:4], rtol=1e-11)
    for i in range(4):
        assert abs(abs(vb[i] @ V[:, -1 - i]) - 1.0) < 1e-9


def pin_index_entry():
    rng = np.random.default_rng(3)
    V = datagen.haar_orthogonal(9, 512)[:24]
    N = 40
    L = rng.standard_normal((1, N, 512)) * 0.05
    coef = rng.standard_normal((8, 24))
    L[0, :8] = coef @ V                                # inside span(V)
    W = rng.standard_normal((8, 512))
    L[0, 8:16] = W - (W @ V.T) @ V                     # orthogonal to span(V)
    L = L.astype(np.float32).astype(np.float64)        # the stored fp32 values
    hi, _ = _f32_workload(L, rng.standard_normal((1, 1, 512)))
    s, s16, eta = oracle.build_sketch(hi, V)
    ln = np.linalg.norm(L[0], axis=1)
    assert np.allclose(np.linalg.norm(s[0], axis=1) ** 2 + eta[0] ** 2, ln ** 2, rtol=1e-10)
    assert np.all(eta[0, :8] <= 1e-6 * ln[:8])         # fp32 storage of rows built inside the span
    assert np.allclose(s[0, :8], coef, atol=1e-6)
    assert np.all(np.abs(s[0, 8:16]) <= 1e-6 * ln[8:16, None])
    assert np.allclose(eta[0, 8:16], ln[8:16], rtol=1e-10)
    for x, h in ((s[0, 20, 3], s16[0, 20, 3]), (s[0, 33, 0], s16[0, 33, 0])):
        assert h == oracle.bf16_rne(x)


def pin_query_side():
    rng = np.random.default_rng(4)
    V = datagen.haar_orthogonal(10, 512)[:32]
    qc = rng.standard_normal((2, 3, 512))
    hi, _ = _f32_workload(rng.standard_normal((2, 8, 512)), qc)
    p, rho = oracle.sketch_query(hi, V)
    qcs = qc.astype(np.float32).astype(np.float64)
    assert np.allclose((p ** 2).sum(-1) + rho ** 2, (qcs ** 2).sum(-1), rtol=1e-10)
    p0, rho0 = oracle.sketch_query(hi, np.zeros((0, 512)))
    assert p0.shape[-1] == 0 and np.allclose(rho0, np.linalg.norm(qcs, axis=-1), rtol=1e-12)


def _hand_case():
    # one head, eight rows, V = e_0. qc = (3, 4, 0, ...): p = 3, rho = 4. Row 5: L = (0.5, 0.25, 0, ...), so s = 0.5 and
    # eta = 0.25; its RoPE score is 0. T(row 5) = lam (3 * 0.5 + z * 4 * 0.25) = lam (1.5 + z).
    N = 8
    L = np.zeros((1, N, 512))
    L[0, 5, :2] = (0.5, 0.25)
    qc = np.zeros((1, 1, 512))
    qc[0, 0, :2] = (3.0, 4.0)
    hi, wl = _f32_workload(L, qc)
    V = np.zeros((1, 512))
    V[0, 0] = 1.0
    return hi, V


def pin_trigger_hand_case():
    hi, V = _hand_case()
    s, s16, eta = oracle.build_sketch(hi, V)
    p, rho = oracle.sketch_query(hi, V)
    assert p[0, 0, 0] == 3.0 and rho[0, 0] == 4.0 and s[0, 5, 0] == 0.5 and eta[0, 5] == 0.25
    a = np.zeros((1, 1, 8))
    pres = np.zeros((1, 1))
    idx = np.array([[[0, 1, 2, 3, 4, 6, 7, 0]]], np.int32)   # every row but 5 is attended
    cnt = np.array([[7]], np.int32)
    z = 0.4
    T5 = LAM * (1.5 + z)
    for smax, fires in ((T5 * (1 - 1e-9), True), (T5 * (1 + 1e-9), False)):
        fidx, fcnt = oracle.trigger(hi, 64, LAM, z, 0, a, eta, pres, idx, cnt, np.array([[smax]]), 0,
                                    sketch=(s16, p, rho))
        assert (fcnt[0, 0] == 1 and fidx[0, 0, 0] == 5) == fires


def pin_lemma1_soundness():
    # z_eff = 1: the trigger score bounds the exact logit up to the bf16 rounding of the stored sketch
    wl = datagen.make_workload(2, 8, 512, seed=21, query_rank=8, n_planted=0)
    rng = np.random.default_rng(5)
    for b in range(2):
        for h in range(0, 8, 2):
            u = int(rng.integers(0, 400))
            qc = wl.q_latent[b, h].float()
            wl.cache[b, u, :512] = (3.0 * qc / qc.norm()).to(wl.cache.dtype)
    hi = oracle.HostInputs(wl)
    q = datagen.prefix_queries(wl, 300).double().numpy()
    V, _ = oracle.sketch_basis(q, 16)
    a = oracle.scores(hi)
    W, k = 32, 16
    idx, cnt, _ = oracle.select(a, k, W)
    _, _, smax = oracle.attention(hi, LAM, idx, cnt)
    s, s16, eta = oracle.build_sketch(hi, V)
    p, rho = oracle.sketch_query(hi, V)
    _, _, _, pres = oracle.build_index(hi, 64)
    fidx, fcnt = oracle.trigger(hi, 64, LAM, 1.0, 0, a, eta, pres, idx, cnt, smax, W, sketch=(s16, p, rho))
    L = wl.latent.double().numpy()
    K = wl.rope.double().numpy()
    qc = wl.q_latent.double().numpy()
    qr = wl.q_rope.double().numpy()
    sh = s16.astype(np.uint32) << 16
    shat = sh.view(np.float32).astype(np.float64)
    n_must = 0
    for b in range(2):
        for h in range(8):
            logits = LAM * (L[b] @ qc[b, h] + K[b] @ qr[b, h])      # Eq. 1, exact
            slack = LAM * np.linalg.norm(p[b, h]) * np.linalg.norm(s[b] - shat[b], axis=1)
            S = set(idx[b, h, :cnt[b, h]].tolist())
            F = set(fidx[b, h, :fcnt[b, h]].tolist())
            for u in range(0, 512 - W):
                if u not in S and logits[u] > smax[b, h] + slack[u]:
                    assert u in F, (b, h, u)
                    n_must += 1
    assert n_must > 0                                  # the planted rows beat s*


def pin_decode_step_composes():
    wl = datagen.make_workload(1, 4, 384, seed=23, query_rank=8, n_planted=4)
    hi = oracle.HostInputs(wl)
    V, _ = oracle.sketch_basis(datagen.prefix_queries(wl, 100).double().numpy(), 12)
    W, rho_keep, z = 32, 1 / 16, 0.3
    res = oracle.decode_step(hi, rho=rho_keep, window=W, trigger=1, z_eff=z, sketch_basis=V)
    a = oracle.scores(hi)
    k = oracle.keep_count(384, rho_keep, W)
    idx, cnt, _ = oracle.select(a, k, W)
    _, _, smax = oracle.attention(hi, LAM, idx, cnt)
    _, s16, eta = oracle.build_sketch(hi, V)
    p, rho = oracle.sketch_query(hi, V)
    _, _, _, pres = oracle.build_index(hi, 64)
    fidx, fcnt = oracle.trigger(hi, 64, LAM, z, 0, a, eta, pres, idx, cnt, smax, W, sketch=(s16, p, rho))
    for h in range(4):
        c0 = cnt[0, h]
        assert res["count"][0, h] == c0 + fcnt[0, h]
        assert res["idx"][0, h, c0:c0 + fcnt[0, h]].tolist() == fidx[0, h, :fcnt[0, h]].tolist()
    assert res["rc"] == 0
    assert oracle.decode_step(hi, rho=rho_keep, window=W, trigger=2, sketch_basis=V)["rc"] == -1


def pin_calibration_matches_sketch_trigger():
    # hard queries (the argmax row's RoPE score is ordinary, so tier 1 leaves it out): the required inflation computed
    # with the sketch puts the row exactly on s* in the sketch trigger at z_eff = zq / sqrt(512 - r_sk) -- just above
    # it fires, just below it does not
    # the planted row points along the query's residual outside span(V): its logit dominates but the sketch term
    # cannot see it, so only the certificate can bring it back (a positive required inflation)
    wl = datagen.make_workload(1, 4, 512, seed=33, query_rank=8, n_planted=0)
    r_sk, W = 16, 32
    V, _ = oracle.sketch_basis(datagen.prefix_queries(wl, 100).double().numpy(), r_sk)
    for h in range(4):
        qc = wl.q_latent[0, h].double().numpy()
        res = qc - V.T @ (V @ qc)
        wl.cache[0, 100 + 37 * h, :512] = torch.as_tensor(12.0 * res / np.linalg.norm(res)).to(wl.cache.dtype)
    hi = oracle.HostInputs(wl)
    a = oracle.scores(hi)
    idx, cnt, _ = oracle.select(a, 8, W)
    _, s16, eta = oracle.build_sketch(hi, V)
    p, rho = oracle.sketch_query(hi, V)
    pres = oracle.build_index(hi, 64)[3]
    zq, ustar, n = oracle.calib_zq(hi, 64, LAM, a, eta, pres, idx, cnt, sketch=(s16, p, rho))
    _, _, smax = oracle.attention(hi, LAM, idx, cnt)
    checked = 0
    for h in range(4):
        if np.isnan(zq[0, h]) or zq[0, h] <= 0:
            continue
        for f, fires in ((1 + 1e-9, True), (1 - 1e-9, False)):
            z_eff = f * zq[0, h] / math.sqrt(512 - r_sk)
            fidx, fcnt = oracle.trigger(hi, 64, LAM, z_eff, 0, a, eta, pres, idx, cnt, smax, W, sketch=(s16, p, rho))
            assert (int(ustar[0, h]) in fidx[0, h, :fcnt[0, h]].tolist()) == fires, (h, f)
        checked += 1
    assert checked >= 1 and n >= checked
    # without the sketch the same queries need a different (rank-0) inflation
    _, _, eta0, _ = oracle.build_index(hi, 64)
    zq0, _, _ = oracle.calib_zq(hi, 64, LAM, a, eta0, pres, idx, cnt)
    assert np.nanmax(np.abs(zq0 - zq)) > 1e-3


PINS = [pin_basis_matches_eigh, pin_basis_known_spectrum, pin_basis_direct_route, pin_index_entry, pin_query_side, pin_trigger_hand_case,
        pin_lemma1_soundness, pin_decode_step_composes, pin_calibration_matches_sketch_trigger]


@pytest.mark.parametrize("pin", PINS, ids=lambda f: f.__name__)
def test_pin(pin):
    oracle.set_mutation(oracle.MUT_NONE)
    pin()


def test_planted_mistake_is_caught():
    oracle.set_mutation(oracle.MUT_SKETCH_QNORM)
    try:
        with pytest.raises(AssertionError):
            pin_trigger_hand_case()
    finally:
        oracle.set_mutation(oracle.MUT_NONE)


def test_sketch_tightens_the_trigger():
    """The point of the sketch (Sec. 4.2): with low-rank queries the certificate shrinks, so at the same sound z the
    trigger admits far fewer rows than with sketch rank 0."""
    wl = datagen.make_workload(1, 8, 1024, seed=29, query_rank=8, n_planted=8)
    hi = oracle.HostInputs(wl)
    V, _ = oracle.sketch_basis(datagen.prefix_queries(wl, 200).double().numpy(), 16)
    r0 = oracle.decode_step(hi, rho=1 / 32, window=64, trigger=1, z_eff=1.0)
    r1 = oracle.decode_step(hi, rho=1 / 32, window=64, trigger=1, z_eff=1.0, sketch_basis=V)
    k = oracle.keep_count(1024, 1 / 32, 64) + 64
    f0 = int((r0["count"] - k).sum())
    f1 = int((r1["count"] - k).sum())
    assert f1 < 0.5 * f0, (f0, f1)
    print(f"fired rows, rank 0: {f0}; rank 16: {f1}")
