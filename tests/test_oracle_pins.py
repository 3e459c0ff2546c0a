"""Pins for the CPU oracle: what the paper and plain mathematics fix, independent of the oracle itself.

Each pin is a function that raises AssertionError when the oracle disagrees with a closed form, a hand case
with a known answer, a library routine on a special case (numpy sort / matmul, scipy softmax), brute force on
a tiny input, or one of the paper's lemmas. ``test_planted_mistakes_are_caught`` plants plausible mistakes
in the oracle (a flipped tie-break, a dropped window, a wrong scale, a transposed rotation, a dropped RoPE
summand, a dropped certificate term) and checks that some pin fails on each.
"""
import json
import math
import os

import numpy as np
import pytest
import scipy.special
import torch

import oracle
from paper_2609_03949_gb300 import datagen
from paper_2609_03949_gb300.bytes_model import paper_read_budget

LAM = 1.0 / math.sqrt(192.0)
GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def host(cache, qc, qr, rot=None, dtype="f32"):
    cache = torch.as_tensor(np.asarray(cache), dtype=torch.float64)
    qc = torch.as_tensor(np.asarray(qc), dtype=torch.float64)
    qr = torch.as_tensor(np.asarray(qr), dtype=torch.float64)
    t = torch.float32 if dtype == "f32" else torch.bfloat16
    B, N, _ = cache.shape
    rot = torch.eye(64) if rot is None else torch.as_tensor(np.asarray(rot), dtype=torch.float32)
    wl = datagen.Workload(B=B, H=qc.shape[1], N=N, dtype=dtype, cache=cache.to(t), q_latent=qc.to(t),
                          q_rope=qr.to(t), rot=rot, planted_pos=torch.zeros(B, 0, dtype=torch.int64),
                          planted_head=torch.zeros(0, dtype=torch.int64), seed=0)
    return oracle.HostInputs(wl), wl


def f64(t):
    return t.detach().cpu().double().numpy()


def exact_logits(wl, lam=LAM):
    """lambda * (qc . L + qr . K) for every (b, h, u), fp64 via numpy matmul."""
    L, K = f64(wl.latent), f64(wl.rope)
    qc, qr = f64(wl.q_latent), f64(wl.q_rope)
    return lam * (np.einsum("bhj,bnj->bhn", qc, L) + np.einsum("bhj,bnj->bhn", qr, K))


def small_random(B=2, H=4, N=300, dtype="bf16", seed=5, **kw):
    wl = datagen.make_workload(B, H, N, dtype=dtype, seed=seed, **kw)
    return oracle.HostInputs(wl), wl


# ------------------------------------------------------------------------------------------------ pins
def pin_keep_count():
    # k = min(ceil(rho N), |A|), A = [n_sink, N - W)
    assert oracle.keep_count(1024, 1 / 8, 64) == 128
    assert oracle.keep_count(1001, 1 / 8, 0) == 126          # ceil, not floor
    assert oracle.keep_count(100, 0.5, 90) == 10              # clamped to the archive
    assert oracle.keep_count(64, 1 / 32, 64) == 0             # window covers the whole context
    assert oracle.keep_count(8192, 1 / 128, 128) == 64
    assert oracle.keep_count(65536, 1 / 32, 256) == 2048
    assert oracle.keep_count(100, 0.5, 10, 4) == 50
    assert oracle.keep_count(100, 1.0, 10, 4) == 86


def pin_scores_r64_matmul():
    hi, wl = small_random()
    a = oracle.scores(hi, 64)
    ref = np.einsum("bhj,bnj->bhn", f64(wl.q_rope), f64(wl.rope))
    np.testing.assert_allclose(a, ref, rtol=1e-13, atol=1e-13)


def pin_digest_orientation_permutation():
    # O = permutation with row j = e_{pi(j)}, so (O x)[j] = x[pi(j)]; pi has 3-cycles, so O != O^T.
    pi = np.roll(np.arange(64), -5)
    pi[:3] = [7, 2, 40]
    pi = np.array(list(dict.fromkeys(list(pi[:3]) + [i for i in range(64) if i not in pi[:3]])))
    O = np.zeros((64, 64))
    O[np.arange(64), pi] = 1.0
    rng = np.random.default_rng(3)
    N, H, r = 70, 2, 8
    cache = np.zeros((1, N, 576))
    cache[0, :, 512:] = rng.integers(-8, 9, size=(N, 64))
    qr = rng.integers(-4, 5, size=(1, H, 64)).astype(float)
    hi, _ = host(cache, np.zeros((1, H, 512)), qr, rot=O)
    dig, dig16, _, pres = oracle.build_index(hi, r)
    K = cache[0, :, 512:]
    np.testing.assert_array_equal(dig[0], K[:, pi[:r]])
    a = oracle.scores(hi, r, dig16)
    np.testing.assert_array_equal(a[0], qr[0][:, pi[:r]] @ K[:, pi[:r]].T)
    res = np.linalg.norm(K[:, pi[r:]], axis=1)
    np.testing.assert_allclose(pres[0], [res[p * 64:(p + 1) * 64].max() for p in range(2)], rtol=1e-15)


def pin_digest_haar_matches_numpy():
    hi, wl = small_random(B=1, N=130)
    O = f64(wl.rot)
    np.testing.assert_allclose(O @ O.T, np.eye(64), atol=1e-6)
    for r in (4, 16, 32):
        dig, dig16, eta, pres = oracle.build_index(hi, r)
        Y = f64(wl.rope) @ O.T
        np.testing.assert_allclose(dig, Y[..., :r], rtol=1e-12, atol=1e-12)
        # orthogonal invariance: digest score + the uncovered coordinates' dot = the full RoPE score
        a = oracle.scores(hi, r, dig16)
        qt = f64(wl.q_rope) @ O.T
        full = np.einsum("bhj,bnj->bhn", f64(wl.q_rope), f64(wl.rope))
        rest = np.einsum("bhj,bnj->bhn", qt[..., r:], Y[..., r:])
        slack = np.einsum("bhj,bnj->bhn", np.abs(qt[..., :r]), np.abs(Y[..., :r])) * 2.0 ** -8 + 1e-5
        assert np.all(np.abs(a + rest - full) <= slack)


def pin_select_ramp():
    # K_u = u e_0, qr = e_0 => a[u] = u: the top-k are the largest archive positions
    N, W, s, rho = 200, 16, 3, 1 / 8
    cache = np.zeros((1, N, 576))
    cache[0, :, 512] = np.arange(N)
    qr = np.zeros((1, 1, 64))
    qr[0, 0, 0] = 1.0
    hi, _ = host(cache, np.zeros((1, 1, 512)), qr)
    k = oracle.keep_count(N, rho, W, s)
    idx, cnt, kth = oracle.select(oracle.scores(hi), k, W, s)
    want = sorted(set(range(s)) | set(range(N - W - k, N - W)) | set(range(N - W, N)))
    assert cnt[0, 0] == len(want) == k + W + s
    assert list(idx[0, 0, :cnt[0, 0]]) == want
    assert kth[0, 0] == N - W - k


def pin_select_all_equal_ties():
    # all scores equal => ties go to the smaller positions
    a = np.full((1, 2, 120), 0.25)
    idx, cnt, kth = oracle.select(a, 10, 8, 2)
    want = list(range(0, 12)) + list(range(112, 120))
    assert list(idx[0, 1, :cnt[0, 1]]) == want
    assert kth[0, 1] == 0.25


def pin_select_window_only():
    a = np.random.default_rng(1).standard_normal((1, 3, 40))
    k = oracle.keep_count(40, 1 / 4, 40)
    idx, cnt, kth = oracle.select(a, k, 40, 0)
    assert k == 0 and np.all(cnt == 40) and np.all(np.isinf(kth))
    assert np.all(idx[0, :, :40] == np.arange(40))


def pin_select_bruteforce_lexsort():
    rng = np.random.default_rng(11)
    for N, W, s, k in ((50, 5, 2, 7), (37, 0, 0, 37), (64, 10, 0, 1), (65, 3, 1, 30)):
        a = rng.integers(0, 5, size=(2, 3, N)).astype(float)       # many ties
        idx, cnt, kth = oracle.select(a, k, W, s)
        for b in range(2):
            for h in range(3):
                arch = np.arange(s, N - W)
                order = np.lexsort((arch, -a[b, h, arch]))        # score desc, then position asc
                top = arch[order[:k]]
                want = sorted(set(range(s)) | set(top.tolist()) | set(range(N - W, N)))
                assert cnt[b, h] == len(want) == k + W + s
                assert list(idx[b, h, :cnt[b, h]]) == want
                assert kth[b, h] == a[b, h, top[-1]]


def pin_select_count_invariant():
    hi, wl = small_random(N=500)
    for rho, W, s in ((1 / 8, 64, 0), (1 / 32, 100, 4), (1.0, 0, 0)):
        k = oracle.keep_count(500, rho, W, s)
        _, cnt, _ = oracle.select(oracle.scores(hi), k, W, s)
        assert np.all(cnt == k + W + s)


def pin_attention_dense_rho1():
    # rho = 1, W = 0: every row attended => dense absorbed-MLA attention (softmax from scipy)
    hi, wl = small_random(B=2, H=3, N=257, dtype="bf16")
    k = oracle.keep_count(257, 1.0, 0)
    idx, cnt, _ = oracle.select(oracle.scores(hi), k, 0)
    out, lse, smax = oracle.attention(hi, LAM, idx, cnt)
    s = exact_logits(wl)
    p = scipy.special.softmax(s, axis=-1)
    ref = np.einsum("bhn,bnj->bhj", p, f64(wl.latent))
    np.testing.assert_allclose(out, ref, rtol=1e-11, atol=1e-13)
    np.testing.assert_allclose(lse, scipy.special.logsumexp(s, axis=-1), rtol=1e-13)
    np.testing.assert_allclose(smax, s.max(-1), rtol=1e-13)


def pin_attention_constant_rows():
    # L_u = c for every row => sum p = 1 gives out = c
    rng = np.random.default_rng(2)
    N = 90
    cache = np.zeros((1, N, 576))
    c = rng.integers(-3, 4, size=512) / 8.0
    cache[0, :, :512] = c
    cache[0, :, 512:] = rng.standard_normal((N, 64)).round(2)
    hi, _ = host(cache, rng.standard_normal((1, 2, 512)).round(2), rng.standard_normal((1, 2, 64)).round(2))
    idx = np.tile(np.arange(0, N, 3, dtype=np.int32), (1, 2, 1))
    out, _, _ = oracle.attention(hi, LAM, idx, np.full((1, 2), idx.shape[-1], np.int32))
    np.testing.assert_allclose(out[0], np.tile(c, (2, 1)), rtol=0, atol=1e-13)


def pin_attention_hull_and_permutation():
    hi, wl = small_random(B=1, H=4, N=200, dtype="f32")
    rng = np.random.default_rng(4)
    sel = np.sort(rng.choice(200, size=(4, 37), replace=True), axis=1)
    sel = np.stack([np.unique(r)[:20] for r in sel])[None].astype(np.int32)
    cnt = np.full((1, 4), 20, np.int32)
    out, lse, smax = oracle.attention(hi, LAM, sel, cnt)
    Lm = f64(wl.latent)[0]
    for h in range(4):
        assert np.linalg.norm(out[0, h]) <= np.linalg.norm(Lm[sel[0, h]], axis=1).max() + 1e-12
    # shuffle the cache rows, remap the ids: identical output (Lemma 1)
    perm = rng.permutation(200)
    inv = np.argsort(perm)
    wl2 = datagen.Workload(**{**wl.__dict__, "cache": wl.cache[:, perm].clone()})
    hi2 = oracle.HostInputs(wl2)
    sel2 = inv[sel].astype(np.int32)
    out2, lse2, smax2 = oracle.attention(hi2, LAM, sel2, cnt)
    np.testing.assert_allclose(out2, out, rtol=1e-12, atol=1e-14)
    np.testing.assert_allclose(lse2, lse, rtol=1e-13)
    np.testing.assert_allclose(smax2, smax, rtol=1e-13)


def pin_attention_single_row_and_uniform():
    hi, wl = small_random(B=1, H=2, N=100, dtype="f32")
    s = exact_logits(wl)
    idx = np.array([[[17], [63]]], np.int32)
    out, lse, smax = oracle.attention(hi, LAM, idx, np.ones((1, 2), np.int32))
    np.testing.assert_allclose(out[0, 0], f64(wl.latent)[0, 17], rtol=1e-15)
    np.testing.assert_allclose(out[0, 1], f64(wl.latent)[0, 63], rtol=1e-15)
    np.testing.assert_allclose(lse[0], [s[0, 0, 17], s[0, 1, 63]], rtol=1e-13)
    np.testing.assert_allclose(smax[0], lse[0], rtol=1e-15)
    # zero query => all logits equal => mean of the attended rows, lse = log n
    cache = f64(wl.cache)
    hz, _ = host(cache, np.zeros((1, 1, 512)), np.zeros((1, 1, 64)))
    sel = np.array([[[1, 5, 9, 40, 99]]], np.int32)
    out, lse, smax = oracle.attention(hz, LAM, sel, np.array([[5]], np.int32))
    np.testing.assert_allclose(out[0, 0], cache[0, sel[0, 0], :512].mean(0), rtol=1e-13, atol=1e-16)
    np.testing.assert_allclose(lse[0, 0], math.log(5), rtol=1e-15)
    out, lse, smax = oracle.attention(hz, LAM, sel, np.array([[0]], np.int32))
    assert np.all(out == 0) and np.isneginf(lse[0, 0]) and np.isneginf(smax[0, 0])


def pin_attention_leakage_bound():
    # Lemma 3: with F attended, s* its max logit, gamma = s* - max excluded logit:
    # excluded weight <= (T - |F|) e^{-gamma} * (max included weight), and |o_F - o_dense| <= 2 * mass * max|v|.
    hi, wl = small_random(B=1, H=4, N=400, dtype="bf16", n_planted=8)
    k = oracle.keep_count(400, 1 / 8, 32)
    idx, cnt, _ = oracle.select(oracle.scores(hi), k, 32)
    out, lse, smax = oracle.attention(hi, LAM, idx, cnt)
    s = exact_logits(wl)[0]
    Lm = f64(wl.latent)[0]
    dense = scipy.special.softmax(s, axis=-1) @ Lm
    for h in range(4):
        inc = np.zeros(400, bool)
        inc[idx[0, h, :cnt[0, h]]] = True
        sstar = s[h, inc].max()
        assert abs(sstar - smax[0, h]) < 1e-12
        gamma = sstar - s[h, ~inc].max()
        excl_rel = np.exp(s[h, ~inc] - sstar).sum()
        assert excl_rel <= (~inc).sum() * math.exp(-gamma) * (1 + 1e-12)
        mass = np.exp(s[h, ~inc]).sum() / np.exp(s[h]).sum()
        err = np.linalg.norm(out[0, h] - dense[h])
        assert err <= 2.0 * mass * np.linalg.norm(Lm, axis=1).max() + 1e-13


def _trigger_case(r, z, top_j=0, N=600, H=6, W=40, rho=1 / 16, seed=9):
    hi, wl = small_random(B=1, H=H, N=N, dtype="bf16", seed=seed, n_planted=6, planted_hi=N - W)
    dig, dig16, eta, pres = oracle.build_index(hi, r)
    a = oracle.scores(hi, r, dig16)
    k = oracle.keep_count(N, rho, W)
    idx, cnt, _ = oracle.select(a, k, W)
    _, _, smax = oracle.attention(hi, LAM, idx, cnt)
    fidx, fcnt = oracle.trigger(hi, r, LAM, z, top_j, a, eta, pres, idx, cnt, smax, W)
    return hi, wl, a, eta, pres, idx, cnt, smax, fidx, fcnt, k


def pin_trigger_sound():
    # Lemma 2 with sketch rank 0: with z_eff = 1, no archived row left out of S u F has a logit above s*.
    for r in (64, 16):
        hi, wl, a, eta, pres, idx, cnt, smax, fidx, fcnt, k = _trigger_case(r, 1.0)
        s = exact_logits(wl)[0]
        dig_slack = 0.0
        if r < 64:
            qt = f64(wl.q_rope)[0] @ f64(wl.rot).T
            Y = f64(wl.rope)[0] @ f64(wl.rot).T
            dig_slack = LAM * (np.abs(qt[:, :r]) @ np.abs(Y[:, :r]).T) * 2.0 ** -8
        for h in range(wl.H):
            att = set(idx[0, h, :cnt[0, h]].tolist()) | set(fidx[0, h, :fcnt[0, h]].tolist())
            assert set(fidx[0, h, :fcnt[0, h]].tolist()).isdisjoint(idx[0, h, :cnt[0, h]].tolist())
            out_rows = np.array(sorted(set(range(wl.N)) - att), dtype=int)
            if len(out_rows):
                slack = dig_slack[h, out_rows] if r < 64 else 0.0
                assert np.all(s[h, out_rows] <= smax[0, h] + slack + 1e-9)
    # a row whose content summand alone beats s* must fire
    N, W = 128, 8
    cache = np.zeros((1, N, 576))
    rng = np.random.default_rng(0)
    qc = rng.standard_normal((1, 1, 512)).round(1)
    cache[0, :, :512] = rng.standard_normal((N, 512)).round(1) * 0.01
    cache[0, 5, :512] = qc[0, 0] / np.linalg.norm(qc[0, 0])
    qr = np.zeros((1, 1, 64))
    qr[0, 0, 0] = 1.0
    cache[0, :, 512] = np.linspace(0, 1, N).round(3)
    hi, wl = host(cache, qc, qr)
    a = oracle.scores(hi)
    idx, cnt, _ = oracle.select(a, 4, W)
    _, _, smax = oracle.attention(hi, LAM, idx, cnt)
    _, _, eta, pres = oracle.build_index(hi, 64)
    fidx, fcnt = oracle.trigger(hi, 64, LAM, 1.0, 0, a, eta, pres, idx, cnt, smax, W)
    assert 5 in fidx[0, 0, :fcnt[0, 0]].tolist()


def pin_trigger_z0_and_monotone():
    hi, wl, a, eta, pres, idx, cnt, smax, f0, c0, k = _trigger_case(64, 0.0)
    for h in range(wl.H):
        S = set(idx[0, h, :cnt[0, h]].tolist())
        want = [u for u in range(0, wl.N - 40) if u not in S and LAM * a[0, h, u] > smax[0, h]]
        assert f0[0, h, :c0[0, h]].tolist() == want
    prev = None
    for z in (0.0, 0.05, 0.2, 1.0):
        _, _, _, _, _, _, _, _, f, c, _ = _trigger_case(64, z)
        sets = [set(f[0, h, :c[0, h]].tolist()) for h in range(wl.H)]
        if prev is not None:
            assert all(p <= q for p, q in zip(prev, sets))
        prev = sets


def pin_trigger_top_j():
    hi, wl, a, eta, pres, idx, cnt, smax, fall, call, k = _trigger_case(16, 0.3)
    _, _, _, _, _, _, _, _, fj, cj, _ = _trigger_case(16, 0.3, top_j=5)
    qt = f64(wl.q_rope)[0] @ f64(wl.rot).T
    qres = np.linalg.norm(qt[:, 16:], axis=1)
    qcn = np.linalg.norm(f64(wl.q_latent)[0], axis=1)
    for h in range(wl.H):
        fired = fall[0, h, :call[0, h]]
        T = LAM * (a[0, h, fired] + qres[h] * pres[0, fired // 64] + 0.3 * qcn[h] * eta[0, fired])
        order = np.lexsort((fired, -T))
        assert cj[0, h] == min(5, len(fired))
        assert fj[0, h, :cj[0, h]].tolist() == sorted(fired[order[:5]].tolist())


def pin_page_norms():
    # per 64-row page: the largest |K_u| over all 64 RoPE dims and the largest |L_u| (numpy norms, ragged tail)
    hi, wl = small_random(B=2, N=150, dtype="bf16")
    pk, pe = oracle.page_norms(hi)
    kn = np.linalg.norm(f64(wl.rope), axis=-1)
    ln = np.linalg.norm(f64(wl.latent), axis=-1)
    for b in range(2):
        for p in range(3):
            assert pk[b, p] == pytest.approx(kn[b, p * 64:(p + 1) * 64].max(), rel=1e-14)
            assert pe[b, p] == pytest.approx(ln[b, p * 64:(p + 1) * 64].max(), rel=1e-14)


def _page_hand_case():
    # four pages; page 3 is the recent window. Page p holds RoPE keys of norm <= p + 1 (largest on its last row)
    # and latent rows of norm <= 0.5 (p + 1); qr = e_0 (|qr| = 1), |qc| = 2.
    N, W = 256, 64
    cache = np.zeros((1, N, 576))
    for u in range(N):
        p = u // 64
        f = (u % 64 + 1) / 64.0
        cache[0, u, 512 + 1] = (p + 1) * f            # K_u = (p + 1) f e_1: qr . K_u = 0, |K_u| = (p + 1) f
        cache[0, u, 3] = 0.5 * (p + 1) * f            # |L_u| = 0.5 (p + 1) f
    qc = np.zeros((1, 1, 512))
    qc[0, 0, 7] = 2.0
    qr = np.zeros((1, 1, 64))
    qr[0, 0, 0] = 1.0
    hi, wl = host(cache, qc, qr)
    idx = np.arange(N - W, N, dtype=np.int32)[None, None, :]      # S = the window only
    cnt = np.array([[W]], np.int32)
    return hi, wl, idx, cnt, N, W


def pin_page_trigger_hand():
    # reading B: page p fires (all its archived rows outside S) iff lam (|qr| max|K| + z |qc| max eta) > s*
    hi, wl, idx, cnt, N, W = _page_hand_case()
    pk, pe = oracle.page_norms(hi)
    for z in (1.0, 0.5):
        bound = [LAM * ((p + 1) + z * 2.0 * 0.5 * (p + 1)) for p in range(3)]
        for s_star, want_pages in ((bound[1] * (1 - 1e-9), (1, 2)), (bound[1] * (1 + 1e-9), (2,)),
                                   (bound[0] * (1 - 1e-9), (0, 1, 2)), (bound[2] * (1 + 1e-9), ())):
            fidx, fcnt = oracle.trigger_page(hi, LAM, z, 0, pk, pe, idx, cnt, np.array([[s_star]]), W)
            want = [u for p in want_pages for u in range(64 * p, 64 * p + 64)]
            assert fidx[0, 0, :fcnt[0, 0]].tolist() == want, (z, s_star)
    # top_j: the highest page bound first, then the smaller position
    fidx, fcnt = oracle.trigger_page(hi, LAM, 1.0, 70, pk, pe, idx, cnt, np.array([[0.0]]), W)
    assert fidx[0, 0, :fcnt[0, 0]].tolist() == list(range(64, 70)) + list(range(128, 192))


def pin_page_trigger_sound_and_contains_row_level():
    # with z_eff = 1 no row left out of S u F beats s* (Lemma 2 on the page's extreme norms); at r = 64 every row
    # the row-level rule fires also fires under the page rule (its trigger score is at most the page bound); z = 0
    # reduces the bound to lam |qr| max|K|
    hi, wl, a, eta, pres, idx, cnt, smax, fidx, fcnt, k = _trigger_case(64, 1.0)
    pk, pe = oracle.page_norms(hi)
    s = exact_logits(wl)[0]
    qrn = np.linalg.norm(f64(wl.q_rope)[0], axis=1)
    for z in (1.0, 0.3, 0.0):
        fb, cb = oracle.trigger_page(hi, LAM, z, 0, pk, pe, idx, cnt, smax, 40)
        fa, ca = oracle.trigger(hi, 64, LAM, z, 0, a, eta, pres, idx, cnt, smax, 40)
        for h in range(wl.H):
            S = set(idx[0, h, :cnt[0, h]].tolist())
            FB = set(fb[0, h, :cb[0, h]].tolist())
            assert FB.isdisjoint(S)
            assert set(fa[0, h, :ca[0, h]].tolist()) <= FB
            if z == 1.0:
                out_rows = np.array(sorted(set(range(wl.N)) - S - FB), dtype=int)
                assert np.all(s[h, out_rows] <= smax[0, h] + 1e-9)
            if z == 0.0:
                want = [u for u in range(0, wl.N - 40) if u not in S and LAM * qrn[h] * pk[0, u // 64] > smax[0, h]]
                assert fb[0, h, :cb[0, h]].tolist() == want


def pin_index_norms():
    hi, wl = small_random(B=2, N=150, dtype="bf16")
    for r in (8, 64):
        _, _, eta, pres = oracle.build_index(hi, r)
        np.testing.assert_allclose(eta, np.linalg.norm(f64(wl.latent), axis=-1), rtol=1e-14)
        Y = f64(wl.rope) @ f64(wl.rot).T
        res = np.linalg.norm(Y[..., r:], axis=-1) if r < 64 else np.zeros(Y.shape[:2])
        want = np.stack([[res[b, p * 64:(p + 1) * 64].max() for p in range(3)] for b in range(2)])
        np.testing.assert_allclose(pres, want, rtol=1e-13, atol=0)


def pin_bf16_rne():
    rng = np.random.default_rng(0)
    xs = rng.standard_normal(4000).astype(np.float32) * 10.0 ** rng.integers(-6, 6, 4000)
    want = torch.from_numpy(xs).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    got = np.array([oracle.bf16_rne(float(x)) for x in xs], np.uint16)
    np.testing.assert_array_equal(got, want)
    one = 0x3F80
    assert oracle.bf16_rne(1.0 + 2.0 ** -8) == one                  # tie -> even (down)
    assert oracle.bf16_rne(1.0 + 3 * 2.0 ** -8) == one + 2          # tie -> even (up)
    assert oracle.bf16_rne(1.0 + 2.0 ** -8 + 2.0 ** -30) == one + 1  # just above the tie


def pin_two_tier_is_lse_merge():
    # Lemma 1: attention over S u F equals the LSE merge of the attentions over S and over F.
    hi, wl = small_random(B=1, H=4, N=700, dtype="bf16", seed=21, n_planted=8, planted_hi=700 - 50)
    res = oracle.decode_step(hi, rho=1 / 16, window=50, trigger=1, z_eff=0.3)
    k = oracle.keep_count(700, 1 / 16, 50)
    s = exact_logits(wl)[0]
    Lm = f64(wl.latent)[0]
    nS = k + 50
    for h in range(4):
        c = res["count"][0, h]
        S, F = res["idx"][0, h, :nS], res["idx"][0, h, nS:c]
        assert np.all(np.diff(S) > 0) and np.all(np.diff(F) > 0)
        parts = []
        for rows in (S, F):
            if len(rows):
                parts.append((scipy.special.logsumexp(s[h, rows]),
                              scipy.special.softmax(s[h, rows]) @ Lm[rows]))
        lse = scipy.special.logsumexp([p[0] for p in parts])
        o = sum(math.exp(p[0] - lse) * p[1] for p in parts)
        np.testing.assert_allclose(res["out"][0, h], o, rtol=1e-10, atol=1e-13)
        np.testing.assert_allclose(res["lse"][0, h], lse, rtol=1e-12)
        np.testing.assert_allclose(res["smax"][0, h], s[h, S].max(), rtol=1e-12)


def pin_planted_rows_selected():
    for idx_cfg, over in (("fp32_h16_n1k", {}), ("h128_n8k", dict(N=2048, H=32))):
        wl = datagen.config_workload(idx_cfg, **over)
        hi = oracle.HostInputs(wl)
        p = datagen.CONFIG_PARAMS[idx_cfg]
        res = oracle.decode_step(hi, rho=p["rho"], window=p["window"])
        for b in range(wl.B):
            for pos, h in zip(wl.planted_pos[b].tolist(), wl.planted_head.tolist()):
                assert pos in res["idx"][b, h, :res["count"][b, h]].tolist()


PINS = [pin_keep_count, pin_scores_r64_matmul, pin_digest_orientation_permutation, pin_digest_haar_matches_numpy,
        pin_select_ramp, pin_select_all_equal_ties, pin_select_window_only, pin_select_bruteforce_lexsort,
        pin_select_count_invariant, pin_attention_dense_rho1, pin_attention_constant_rows,
        pin_attention_hull_and_permutation, pin_attention_single_row_and_uniform, pin_attention_leakage_bound,
        pin_trigger_sound, pin_trigger_z0_and_monotone, pin_trigger_top_j, pin_page_norms, pin_page_trigger_hand,
        pin_page_trigger_sound_and_contains_row_level, pin_index_norms, pin_bf16_rne,
        pin_two_tier_is_lse_merge, pin_planted_rows_selected]


@pytest.mark.parametrize("pin", PINS, ids=lambda f: f.__name__)
def test_pin(pin):
    oracle.set_mutation(oracle.MUT_NONE)
    pin()


@pytest.mark.parametrize("mutation,pin", [
    (oracle.MUT_TIE_LARGER, pin_select_all_equal_ties),
    (oracle.MUT_TIE_LARGER, pin_select_bruteforce_lexsort),
    (oracle.MUT_DROP_WINDOW, pin_select_ramp),
    (oracle.MUT_DROP_WINDOW, pin_select_count_invariant),
    (oracle.MUT_SCALE_SQUARED, pin_attention_dense_rho1),
    (oracle.MUT_ROT_TRANSPOSE, pin_digest_orientation_permutation),
    (oracle.MUT_ROT_TRANSPOSE, pin_digest_haar_matches_numpy),
    (oracle.MUT_DROP_ROPE, pin_attention_dense_rho1),
    (oracle.MUT_TRIGGER_NO_Z, pin_trigger_sound),
    (oracle.MUT_TRIGGER_NO_Z, pin_page_trigger_hand),
])
def test_planted_mistakes_are_caught(mutation, pin):
    oracle.set_mutation(mutation)
    try:
        with pytest.raises(AssertionError):
            pin()
    finally:
        oracle.set_mutation(oracle.MUT_NONE)


def test_read_budget_golden():
    g = json.load(open(os.path.join(GOLDEN, "read_budget.json")))
    lo = paper_read_budget(g["rho"], g["r_sk"], g["f_range"][0])
    hi = paper_read_budget(g["rho"], g["r_sk"], g["f_range"][1])
    assert lo <= g["total_bytes_per_token_approx"] + 3 and hi >= g["total_bytes_per_token_approx"] - 3
    assert abs((64 + g["r_sk"] + 1) * 2 - g["index_scan_bytes_per_row_approx"]) <= 3
    mid = paper_read_budget(g["rho"], g["r_sk"], sum(g["f_range"]) / 2)
    assert round(g["dense_bytes_per_token"] / mid, 1) == g["ratio_16bit_index_approx"]
    full = paper_read_budget(g["rho"], g["r_sk"], sum(g["f_range"]) / 2, index_bytes=4)
    assert round(g["dense_bytes_per_token"] / full, 1) == g["ratio_full_precision_index_approx"]
