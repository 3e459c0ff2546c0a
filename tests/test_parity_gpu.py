"""GPU parity: the CUDA path through the C ABI against the CPU oracle on seeded synthetic workloads.

Tolerances (from the specification of the path): selections exact except rows within 1e-3 relative of the
k-th threshold; outputs within max relative error 2e-2 (bf16 inputs, fp32 accumulation); lse within 2e-2.
Small and medium cases are checked on every sequence; the large throughput-sweep cases on sequences 0 and B-1.
"""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2609_03949_gb300 import datagen
from paper_2609_03949_gb300 import vk

from parity_util import GpuStep, check_fired, check_fired_page, check_outputs, check_selection

pytestmark = pytest.mark.gpu
LAM = vk.DEFAULT_SM_SCALE


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2609_03949_gb300 import _build
    _build.build()
    vk.lib()


def run_case(wl, *, rho, r=64, window=0, n_sink=0, trigger=0, z_eff=1.0, top_j=0, flags=0, check_seqs=None,
             cap=None):
    """Run one step on the GPU and check it against the oracle on the sequences `check_seqs`."""
    seqs = list(range(wl.B)) if check_seqs is None else check_seqs
    sub = wl.slice_batch(seqs) if check_seqs is not None else wl
    hi = oracle.HostInputs(sub)
    dig16 = None
    if r < 64:
        hi_all = oracle.HostInputs(wl)
        _, dig16, _, _ = oracle.build_index(hi_all, r)
    g = GpuStep(wl, rho=rho, r=r, window=window, n_sink=n_sink, trigger=trigger, z_eff=z_eff, top_j=top_j,
                flags=flags, digest_bf16=dig16, cap=cap).run()
    for key in ("out", "lse", "smax", "idx", "count"):
        g[key] = g[key][seqs]
    a = oracle.scores(hi, r, None if dig16 is None else dig16[seqs])
    k = oracle.keep_count(wl.N, rho, window, n_sink)
    nS = k + window + n_sink
    st = check_selection(a, g["idx"], g["count"], k, window, n_sink)
    res = dict(gpu=g, a=a, k=k, sel=st, hi=hi, sub=sub)
    if not trigger:
        assert np.all(g["count"] == nS)
        res["out"] = check_outputs(hi, LAM, g)
        return res
    # two-tier: s* of the GPU's tier-1 set, the fired rows, then the output over S u F
    _, _, smax_ref = oracle.attention(hi, LAM, g["idx"][..., :nS], np.full_like(g["count"], nS))
    np.testing.assert_allclose(g["smax"], smax_ref, rtol=1e-4, atol=1e-4)
    _, _, eta, pres = oracle.build_index(hi, r)
    gF = [[g["idx"][b, h, nS:g["count"][b, h]].tolist() for h in range(wl.H)] for b in range(len(seqs))]
    if trigger == vk.VK_TRIG_CS_PAGE:
        res["swaps"] = check_fired_page(hi, sub, LAM, z_eff, smax_ref, g["idx"], np.full_like(g["count"], nS), gF,
                                        window, n_sink, top_j)
    else:
        res["swaps"] = check_fired(a, eta, pres, sub, LAM, z_eff, r, smax_ref, g["idx"], np.full_like(g["count"], nS),
                                   gF, window, n_sink, top_j)
    res["out"] = check_outputs(hi, LAM, g)
    res["fired"] = int((g["count"] - nS).sum())
    return res


# ------------------------------------------------------------------------------------------------ configs
def test_fp32_h16_n1k():
    wl = datagen.config_workload("fp32_h16_n1k")
    res = run_case(wl, rho=1 / 8, window=64)
    for pos, h in zip(wl.planted_pos[0].tolist(), wl.planted_head.tolist()):
        assert pos in res["gpu"]["idx"][0, h].tolist()
    assert res["out"]["out_rel"] < 1e-4


@pytest.mark.parametrize("r", [4, 8, 16, 32, 64])
@pytest.mark.parametrize("rho", [1 / 8, 1 / 32, 1 / 128])
def test_h128_n8k_rho_r(rho, r):
    wl = datagen.config_workload("h128_n8k", device="cuda")
    res = run_case(wl, rho=rho, r=r, window=128)
    # tighter than the 2e-2 gate: the only rounding beyond fp32 accumulation is the bf16 softmax weight
    assert res["out"]["out_rel"] < 1e-2


@pytest.mark.parametrize("rho", [1 / 32, 1 / 128])
def test_h64_n32k_lognormal(rho):
    wl = datagen.config_workload("h64_n32k_lognormal", device="cuda")
    run_case(wl, rho=rho, window=256)


def test_h128_n64k_two_tier():
    wl = datagen.config_workload("h128_n64k_two_tier", device="cuda")
    res = run_case(wl, rho=1 / 32, window=256, trigger=1, z_eff=1.0, check_seqs=[0, wl.B - 1])
    assert res["fired"] > 0


@pytest.mark.parametrize("r,z,top_j", [(16, 1.0, 0), (64, 1.0, 16), (8, 0.5, 0)])
def test_two_tier_variants(r, z, top_j):
    wl = datagen.config_workload("h128_n64k_two_tier", device="cuda", B=2, N=8192)
    res = run_case(wl, rho=1 / 32, r=r, window=256, trigger=1, z_eff=z, top_j=top_j)
    assert res["fired"] > 0


@pytest.mark.parametrize("top_j,z", [(0, 1.0), (0, 0.05), (40, 0.05)])
def test_h128_n64k_page_trigger(top_j, z):
    # reading B at config 4's shape (two sequences checked): whole pages admitted by their page-level bound. With the
    # sound z_eff = 1 nearly every page fires on this data; z_eff = 0.05 leaves a mix of fired and quiet pages.
    wl = datagen.config_workload("h128_n64k_two_tier", device="cuda")
    res = run_case(wl, rho=1 / 32, window=256, trigger=vk.VK_TRIG_CS_PAGE, z_eff=z, top_j=top_j,
                   check_seqs=[0, wl.B - 1])
    assert res["fired"] > 0


@pytest.mark.parametrize("r,top_j", [(64, 0), (16, 0), (64, 7)])
def test_page_trigger_variants(r, top_j):
    wl = datagen.config_workload("h128_n64k_two_tier", device="cuda", B=2, N=8192)
    res = run_case(wl, rho=1 / 32, r=r, window=256, n_sink=3, trigger=vk.VK_TRIG_CS_PAGE, z_eff=0.05, top_j=top_j)
    assert res["fired"] > 0


def _skippable_workload():
    # every head finds a strong row in its recent window (K = 4.5 Qr_h / |Qr_h|, so s*_h >~ 4.5 |Qr_h| lambda), while the
    # RoPE keys of rows 1024 .. 5119 are scaled by 1/40: on those pages no head's bound can reach s*, so the r = 64
    # trigger scan skips their tiles
    wl = datagen.make_workload(2, 64, 8192, seed=51, n_planted=0, device="cuda")
    wl.cache[:, 1024:5120, 512:] = (wl.cache[:, 1024:5120, 512:].float() / 40).to(wl.cache.dtype)
    for b in range(wl.B):
        for h in range(64):
            qr = wl.q_rope[b, h].float()
            wl.cache[b, 8192 - 1 - h, 512:] = (4.5 * qr / qr.norm()).to(wl.cache.dtype)
    return wl


@pytest.mark.parametrize("top_j", [0, 5])
def test_page_skip_keeps_fired_sets(top_j):
    # the sound page skip of the row-level scan changes cost, not results: with and without it the fired sets and
    # outputs are identical, and both meet the oracle
    wl = _skippable_workload()
    hi = oracle.HostInputs(wl)
    pk, pe = oracle.page_norms(hi)
    qrn = np.linalg.norm(wl.q_rope.double().cpu().numpy(), axis=-1)
    qcn = np.linalg.norm(wl.q_latent.double().cpu().numpy(), axis=-1)
    res = run_case(wl, rho=1 / 32, window=256, trigger=vk.VK_TRIG_CS, z_eff=0.25, top_j=top_j)
    # the workload really has tiles that every head skips: both pages of the tile stay below every head's s*
    smax = res["gpu"]["smax"]
    bound = LAM * (qrn[:, :, None] * pk[:, None, :] + 0.25 * qcn[:, :, None] * pe[:, None, :])   # [B,H,P]
    quiet = np.all(bound * (1 + 2.0 ** -10) <= smax[:, :, None], axis=1)                        # [B,P]
    tile_quiet = quiet[:, 0::2] & quiet[:, 1::2]
    assert tile_quiet.sum() >= 20, tile_quiet.sum()
    on = GpuStep(wl, rho=1 / 32, window=256, trigger=vk.VK_TRIG_CS, z_eff=0.25, top_j=top_j).run()
    off = GpuStep(wl, rho=1 / 32, window=256, trigger=vk.VK_TRIG_CS, z_eff=0.25, top_j=top_j,
                  flags=vk.VK_FLAG_NO_PAGE_SKIP).run()
    for key in ("idx", "count", "out", "lse"):
        np.testing.assert_array_equal(on[key], off[key])
    assert on["status"] == vk.VK_OK and off["status"] == vk.VK_OK


@pytest.mark.parametrize("N", [16384, 65536, 131072])
@pytest.mark.parametrize("B", [1, 8, 32, 64])
def test_h64_sweep(N, B):
    wl = datagen.make_workload(B, 64, N, dtype="bf16", seed=1000 + 10 * B + N // 16384, n_planted=64,
                               planted_hi=N - 256, device="cuda")
    res = run_case(wl, rho=1 / 32, window=256, check_seqs=sorted({0, B - 1}))
    sub = res["sub"]
    for i in range(sub.B):
        for pos, h in zip(sub.planted_pos[i].tolist(), sub.planted_head.tolist()):
            assert pos in res["gpu"]["idx"][i, h].tolist()


# ------------------------------------------------------------------------------------------------ edges
EDGES = [
    dict(B=1, H=4, N=1, rho=1.0, window=1),
    dict(B=1, H=4, N=1, rho=1.0, window=0),
    dict(B=2, H=8, N=7, rho=0.5, window=2),
    dict(B=1, H=8, N=63, rho=1 / 8, window=16),
    dict(B=1, H=8, N=64, rho=1 / 8, window=64),            # k = 0: window only
    dict(B=1, H=8, N=65, rho=1 / 8, window=16),
    dict(B=3, H=16, N=1000, rho=1 / 8, window=100, n_sink=4),
    dict(B=1, H=100, N=4097, rho=1 / 32, window=128),      # two head groups, ragged tail
    dict(B=1, H=1, N=5000, rho=1 / 16, window=0),
    dict(B=2, H=64, N=2048, rho=1.0, window=0),            # dense
    dict(B=2, H=64, N=3000, rho=1 / 8, window=64, dtype="f32"),
    dict(B=1, H=256, N=2048, rho=1 / 8, window=64),
    dict(B=3, H=192, N=5000, rho=1 / 16, window=64),        # three head groups: ranges of (sequence, row tile) x 3
    dict(B=5, H=128, N=700, rho=1 / 4, window=32),          # two groups, ranges that cross sequence boundaries
    dict(B=300, H=16, N=100, rho=1 / 4, window=8),         # attention CTAs that span several whole segments
    dict(B=1, H=16, N=300000, rho=1 / 64, window=256),      # bitmaps past the selection's shared-memory limit
]


@pytest.mark.parametrize("case", EDGES, ids=lambda c: "-".join(f"{k}{v}" for k, v in c.items()))
def test_edge_cases(case):
    c = dict(case)
    B, H, N = c.pop("B"), c.pop("H"), c.pop("N")
    dtype = c.pop("dtype", "bf16")
    wl = datagen.make_workload(B, H, N, dtype=dtype, seed=77 + N + H, n_planted=min(4, N),
                               planted_hi=max(1, N - c["window"]), device="cuda")
    res = run_case(wl, **c)
    if c["rho"] == 1.0 and c.get("window", 0) == 0:
        assert np.all(res["gpu"]["count"] == N)


def test_two_tier_many_partials():
    # one sequence spread over 64 attention CTAs per tier: the combine merges 64 tier-1 and 64 fired partials per
    # head (the block-per-head merge); most fired tiles are empty, so many CTAs close segments with no tile
    wl = datagen.make_workload(1, 64, 16384, seed=41, n_planted=16, planted_hi=16384 - 256, device="cuda")
    res = run_case(wl, rho=1 / 32, window=256, trigger=1, z_eff=0.6)
    assert res["fired"] > 0


def test_two_tier_sinks_and_capacity():
    wl = datagen.make_workload(2, 32, 6000, seed=5, n_planted=16, planted_hi=6000 - 128, device="cuda")
    run_case(wl, rho=1 / 32, window=128, n_sink=4, trigger=1, z_eff=0.5)
    # a list cap below |S| + |F|: the fired list is cut and the device status says so, outputs stay exact
    k = oracle.keep_count(6000, 1 / 32, 128, 4)
    step = GpuStep(wl, rho=1 / 32, window=128, n_sink=4, trigger=1, z_eff=1.0, cap=k + 128 + 4 + 3)
    g = step.run()
    assert g["status"] == vk.VK_ERR_CAPACITY
    full = GpuStep(wl, rho=1 / 32, window=128, n_sink=4, trigger=1, z_eff=1.0).run()
    np.testing.assert_array_equal(g["out"], full["out"])
    np.testing.assert_array_equal(g["lse"], full["lse"])


# ------------------------------------------------------------------------------------------------ entry points
def test_vk_score_matches_oracle():
    wl = datagen.config_workload("h128_n8k", device="cuda", N=3000, H=32)
    hi = oracle.HostInputs(wl)
    for r in (64, 16):
        _, dig16, _, _ = oracle.build_index(hi, r)
        step = GpuStep(wl, rho=1 / 8, r=r, window=0, digest_bf16=dig16)
        scores = torch.empty(wl.B, wl.H, wl.N, dtype=torch.float32, device="cuda")
        vk.vk_score(step.view, step.params, step.index, scores, step.buf.ws)
        got = scores.cpu().double().numpy()
        ref = oracle.scores(hi, r, dig16)
        np.testing.assert_allclose(got, ref, rtol=1e-5, atol=1e-4)


def test_vk_select_exact_on_integer_ties():
    # integer-valued scores are exact in fp32, so the selection must match the oracle bit for bit
    rng = np.random.default_rng(3)
    B, H, N = 2, 5, 3333
    a = rng.integers(0, 7, size=(B, H, N)).astype(np.float64)
    wl = datagen.make_workload(B, H, N, seed=1, device="cuda")
    view = vk.make_view(wl.cache, wl.q_latent, wl.q_rope)
    for rho, W, s in ((1 / 8, 100, 3), (1 / 3, 0, 0), (1.0, 50, 0)):
        p = vk.make_params(rho, window=W, n_sink=s)
        k = oracle.keep_count(N, rho, W, s)
        cap = k + W + s
        idx = torch.full((B, H, cap), -1, dtype=torch.int32, device="cuda")
        cnt = torch.zeros(B, H, dtype=torch.int32, device="cuda")
        kth = torch.zeros(B, H, dtype=torch.float32, device="cuda")
        vk.vk_select(view, p, torch.from_numpy(a).float().cuda(), idx, cnt, kth)
        ridx, rcnt, rkth = oracle.select(a, k, W, s, cap)
        np.testing.assert_array_equal(cnt.cpu().numpy(), rcnt)
        np.testing.assert_array_equal(idx.cpu().numpy(), ridx)
        np.testing.assert_array_equal(kth.cpu().double().numpy(), rkth)


def test_vk_sparse_attn_given_sets():
    wl = datagen.make_workload(2, 64, 5000, seed=8, device="cuda")
    hi = oracle.HostInputs(wl)
    rng = np.random.default_rng(0)
    cap = 700
    idx = np.full((2, 64, cap), -1, np.int32)
    cnt = rng.integers(0, cap + 1, size=(2, 64)).astype(np.int32)
    cnt[0, 0] = 0
    for b in range(2):
        for h in range(64):
            idx[b, h, :cnt[b, h]] = rng.choice(5000, size=cnt[b, h], replace=False)   # unsorted on purpose
    view = vk.make_view(wl.cache, wl.q_latent, wl.q_rope)
    p = vk.make_params(1 / 8)
    ws = vk.alloc_workspace(view, p, cap)
    out = torch.empty(2, 64, 512, device="cuda")
    lse = torch.empty(2, 64, device="cuda")
    smax = torch.empty(2, 64, device="cuda")
    vk.vk_sparse_attn(view, p, torch.from_numpy(idx).cuda(), torch.from_numpy(cnt).cuda(), out, lse, smax, ws)
    assert vk.vk_poll_status(ws) == vk.VK_OK
    g = dict(out=out.cpu().double().numpy(), lse=lse.cpu().double().numpy())
    r = check_outputs(hi, LAM, g, idx, cnt)
    np.testing.assert_allclose(smax.cpu().double().numpy()[cnt > 0], r["smax"][cnt > 0], rtol=1e-4, atol=1e-4)
    # an id out of range is skipped and reported in the device status
    idx[1, 3, 0] = 5000
    vk.vk_sparse_attn(view, p, torch.from_numpy(idx).cuda(), torch.from_numpy(cnt).cuda(), out, lse, smax, ws)
    assert vk.vk_poll_status(ws) == vk.VK_ERR_INVALID_ARG
    assert vk.vk_poll_status(ws) == vk.VK_OK


def test_build_digest_matches_oracle():
    wl = datagen.make_workload(2, 4, 1000, seed=12, device="cuda")
    hi = oracle.HostInputs(wl)
    view = vk.make_view(wl.cache, wl.q_latent, wl.q_rope)
    for r in (4, 16, 32, 64):
        p = vk.make_params(1 / 8, r=r)
        dig = torch.empty(2, 1000, r, dtype=torch.bfloat16, device="cuda") if r < 64 else None
        eta = torch.empty(2, 1000, device="cuda")
        pres = torch.empty(2, 16, device="cuda")
        vk.vk_build_digest(view, p, wl.rot.cuda(), dig, eta, pres)
        d64, d16, reta, rpres = oracle.build_index(hi, r)
        np.testing.assert_allclose(eta.cpu().double().numpy(), reta, rtol=1e-5)
        np.testing.assert_allclose(pres.cpu().double().numpy(), rpres, rtol=1e-4, atol=1e-5)
        if r < 64:
            got = dig.float().cpu().double().numpy()
            ulp = np.exp2(np.floor(np.log2(np.maximum(np.abs(d64), 1e-30))) - 7)
            assert np.all(np.abs(got - d64) <= ulp * 1.0001)


def test_deterministic_and_graph_capturable():
    wl = datagen.config_workload("h64_n64k", device="cuda", B=4, N=16384)
    step = GpuStep(wl, rho=1 / 32, window=256)
    a = step.run()
    b = step.run()
    for key in ("out", "lse", "idx", "count"):
        np.testing.assert_array_equal(a[key], b[key])
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    step.buf.out.zero_()
    with torch.cuda.graph(g, stream=s):
        vk.vk_decode_step(step.view, step.params, step.index, step.buf.out, step.buf.lse, step.buf.smax, step.buf.idx,
                          step.buf.count, step.buf.ws, stream=s)
    step.buf.out.zero_()
    g.replay()
    torch.cuda.synchronize()
    np.testing.assert_array_equal(step.buf.out.cpu().double().numpy(), a["out"])
    np.testing.assert_array_equal(step.buf.idx.cpu().numpy(), a["idx"])


def test_permutation_invariance_gpu():
    # Lemma 1 on the GPU: permuting the cache rows and remapping the ids leaves the attention output unchanged
    wl = datagen.make_workload(1, 64, 3000, seed=4, device="cuda")
    rng = np.random.default_rng(1)
    cap = 300
    idx = np.stack([np.sort(rng.choice(3000, cap, replace=False)) for _ in range(64)])[None].astype(np.int32)
    cnt = np.full((1, 64), cap, np.int32)
    perm = rng.permutation(3000)
    inv = np.argsort(perm)
    outs = []
    for cache, ids in ((wl.cache, idx), (wl.cache[:, perm].contiguous(), inv[idx].astype(np.int32))):
        view = vk.make_view(cache, wl.q_latent, wl.q_rope)
        p = vk.make_params(1 / 8)
        ws = vk.alloc_workspace(view, p, cap)
        out = torch.empty(1, 64, 512, device="cuda")
        vk.vk_sparse_attn(view, p, torch.from_numpy(ids).cuda(), torch.from_numpy(cnt).cuda(), out, None, None, ws)
        outs.append(out.cpu().numpy())
    # equal up to rounding: a different row order changes the running max, hence the bf16 weights' rounding
    rel = np.abs(outs[0] - outs[1]).max(-1) / np.abs(outs[0]).max(-1)
    assert rel.max() < 5e-3, rel.max()


@pytest.mark.parametrize("flags", [0, vk.VK_FLAG_FORCE_FALLBACK, vk.VK_FLAG_FORCE_DENSE],
                         ids=["fused", "fallback", "dense"])
@pytest.mark.parametrize("trigger,top_j", [(0, 0), (1, 0), (1, 8)])
def test_selection_paths(flags, trigger, top_j):
    # the threshold-candidate path, its exact fallback and the materialised-score path all meet the oracle
    wl = datagen.make_workload(2, 64, 20000, seed=17, n_planted=16, planted_hi=20000 - 256, device="cuda")
    run_case(wl, rho=1 / 32, window=256, n_sink=2, trigger=trigger, z_eff=0.7, top_j=top_j, flags=flags)


@pytest.mark.parametrize("r", [8, 16, 32])
@pytest.mark.parametrize("flags,trigger,top_j", [(0, 0, 0), (vk.VK_FLAG_FORCE_FALLBACK, 0, 0), (0, 1, 0), (0, 1, 6)],
                         ids=["fused", "fallback", "trigger", "trigger-top_j"])
def test_digest_selection_paths(r, flags, trigger, top_j):
    # width-r digests on the tensor cores (query as bf16 high + low parts): the threshold-candidate selection, its
    # exact fallback over recomputed digest scores, and the trigger scan all meet the oracle
    wl = datagen.make_workload(2, 64, 20000, seed=19 + r, n_planted=16, planted_hi=20000 - 256, device="cuda")
    run_case(wl, rho=1 / 32, r=r, window=256, n_sink=2, trigger=trigger, z_eff=0.6, top_j=top_j, flags=flags)


def test_bounded_wait_reports_timeout():
    # Failure detection without a GPU fault: the test hook withholds one CTA's first tile; that CTA's bounded waits
    # give up after about a second, the status word reads VK_ERR_TIMEOUT and the context stays usable.
    wl = datagen.make_workload(2, 64, 8192, seed=23, device="cuda")
    step = GpuStep(wl, rho=1 / 32, window=256, n_sink=4, flags=vk.VK_FLAG_TEST_TIMEOUT)
    g = step.run()
    assert g["status"] == vk.VK_ERR_TIMEOUT
    assert vk.vk_poll_status(step.buf.ws) == vk.VK_OK         # reading the status clears it
    clean = GpuStep(wl, rho=1 / 32, window=256, n_sink=4)
    h = clean.run()
    assert h["status"] == vk.VK_OK
    # the tier-1 selection ran before the withheld attention tile and is unaffected
    np.testing.assert_array_equal(g["idx"], h["idx"])
    hi = oracle.HostInputs(wl)
    check_outputs(hi, LAM, h)


@pytest.mark.parametrize("c", [60.0, 200.0])
def test_attention_rescale_on_logit_jump(c):
    # A row whose logit jumps tens of log2 units above the rows attended before it (in the same attention CTA)
    # moves the running max by more than the kernel's slack: the O^T accumulator is rescaled mid-segment (by
    # 2^-40..-50 for c = 60; underflowing to 0 for c = 200). The output must still match the oracle.
    wl = datagen.make_workload(1, 64, 4096, seed=29, device="cuda")
    qr0 = wl.q_rope[0, 0].float()
    wl.cache[0, 200, 512:] = (c * qr0 / qr0.norm()).to(wl.cache.dtype)
    hi = oracle.HostInputs(wl)
    ids = sorted(set(range(0, 4096, 3)) | {200})
    cap = len(ids)
    idx = np.tile(np.array(ids, np.int32), (1, 64, 1))
    cnt = np.full((1, 64), cap, np.int32)
    view = vk.make_view(wl.cache, wl.q_latent, wl.q_rope)
    p = vk.make_params(1 / 8)
    ws = vk.alloc_workspace(view, p, cap)
    out = torch.empty(1, 64, 512, device="cuda")
    lse = torch.empty(1, 64, device="cuda")
    smax = torch.empty(1, 64, device="cuda")
    vk.vk_sparse_attn(view, p, torch.from_numpy(idx).cuda(), torch.from_numpy(cnt).cuda(), out, lse, smax, ws)
    assert vk.vk_poll_status(ws) == vk.VK_OK
    g = dict(out=out.cpu().double().numpy(), lse=lse.cpu().double().numpy())
    r = check_outputs(hi, LAM, g, idx, cnt)
    np.testing.assert_allclose(smax.cpu().double().numpy(), r["smax"], rtol=1e-4, atol=1e-4)


@pytest.mark.parametrize("z,top_j", [(0.05, 0), (1.0, 0), (0.3, 12)])
def test_fired_passes_agree(z, top_j):
    """The fired rows' two passes (per head over its fired bitmap when no head fired more than 512 rows, else by
    tiles) give the same outputs up to fp32 rounding, and both meet the oracle."""
    wl = datagen.config_workload("h128_n64k_two_tier", device="cuda", B=2, N=8192)
    a = run_case(wl, rho=1 / 32, window=256, trigger=1, z_eff=z, top_j=top_j)
    b = run_case(wl, rho=1 / 32, window=256, trigger=1, z_eff=z, top_j=top_j, flags=vk.VK_FLAG_FIRED_TILES)
    ga, gb = a["gpu"], b["gpu"]
    np.testing.assert_array_equal(ga["idx"], gb["idx"])
    np.testing.assert_array_equal(ga["count"], gb["count"])
    np.testing.assert_allclose(ga["out"], gb["out"], rtol=1e-4, atol=1e-5)
    np.testing.assert_allclose(ga["lse"], gb["lse"], rtol=1e-5, atol=1e-5)


@pytest.mark.parametrize("N,r,sketch", [(5003, 64, 0), (4097, 16, 0), (6001, 64, 32)])
def test_two_tier_ragged_context(N, r, sketch):
    """A context that is not a multiple of 4 rows: the trigger scan reads eta from global memory instead of staging
    it by TMA (its row stride is no multiple of 16 bytes), and the last tile is ragged."""
    H, W = 64, 128
    if sketch:
        wl = datagen.make_workload(1, H, N, seed=N + r, n_planted=8, planted_hi=N - W, query_rank=8)
        hi = oracle.HostInputs(wl)
        V, _ = oracle.sketch_basis(datagen.prefix_queries(wl, 150).double().numpy(), sketch)
        _, s16, eta = oracle.build_sketch(hi, V)
        p, rho = oracle.sketch_query(hi, V)
        g = GpuStep(wl, rho=1 / 32, window=W, trigger=1, z_eff=0.2, sketch=(s16, V, eta)).run()
        a = oracle.scores(hi)
        k = oracle.keep_count(N, 1 / 32, W)
        nS = k + W
        check_selection(a, g["idx"], g["count"], k, W, 0)
        _, _, smax = oracle.attention(hi, LAM, g["idx"][..., :nS], np.full_like(g["count"], nS))
        pres = oracle.build_index(hi, 64)[3]
        fidx, fcnt = oracle.trigger(hi, 64, LAM, 0.2, 0, a, eta, pres, g["idx"], np.full_like(g["count"], nS), smax, W,
                                    sketch=(s16, p, rho))
        for h in range(H):
            got = set(g["idx"][0, h, nS:g["count"][0, h]].tolist())
            ref = set(fidx[0, h, :fcnt[0, h]].tolist())
            assert len(got ^ ref) <= 2, (h, sorted(got ^ ref)[:5])
        check_outputs(hi, LAM, g)
        return
    wl = datagen.make_workload(1, H, N, seed=N + r, n_planted=8, planted_hi=N - W, device="cuda")
    res = run_case(wl, rho=1 / 32, r=r, window=W, trigger=1, z_eff=0.3)
    assert res["fired"] >= 0
