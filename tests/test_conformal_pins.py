"""Pins for the oracle's conformal calibration of the trigger's z (Sec. 4.2; Sec. 5): the paper's printed constants,
the closed-form order statistic on a synthetic stream of required inflations, the exchangeability guarantee by
simulation, and the required inflation of a hand-built hard query checked against the trigger rule itself (at z just
above zq the argmax row fires, just below it does not). A planted mistake (floor instead of ceiling in the order
statistic) must fail a pin."""
import json
import math
import os

import numpy as np
import pytest
import torch

import oracle
from paper_2609_03949_gb300 import datagen

LAM = 1.0 / math.sqrt(192.0)
GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "conformal.json")


def pin_paper_constants():
    g = json.load(open(GOLDEN))
    assert oracle.min_hard(g["tau"]) == g["min_hard"]
    assert oracle.tau_s(g["tau"]) == pytest.approx(g["tau"] / (1 - g["alpha"]), rel=1e-15)
    # below min_hard no order statistic certifies tau_s: the clamp
    assert oracle.conformal_quantile(np.zeros(g["min_hard"] - 1), g["tau"], g["z_max"]) == g["z_max"]


def pin_quantile_closed_form():
    rng = np.random.default_rng(0)
    ts = oracle.tau_s(0.9)
    for n in (18, 19, 50, 100, 333):
        vals = rng.permutation(np.arange(1, n + 1)) * 0.01          # the k-th smallest is k / 100
        k = math.ceil((n + 1) * ts - 1e-9)
        want = k * 0.01 if k <= n else 8.0
        assert oracle.conformal_quantile(vals, 0.9, 8.0) == pytest.approx(want, abs=1e-12), n
    assert oracle.conformal_quantile(np.full(40, 9.5), 0.9, 8.0) == 8.0        # clamped above
    assert oracle.conformal_quantile(np.full(40, -0.5), 0.9, 8.0) == 0.0       # and below
    # n = 18: k = ceil(19 tau_s) = 18 exactly (tau_s = 18/19), the largest value
    assert oracle.conformal_quantile(np.arange(1, 19) * 0.1, 0.9, 8.0) == pytest.approx(1.8)


def pin_exchangeable_coverage():
    # with n + 1 exchangeable draws, the (n+1)-th is at most the calibrated z with probability >= tau_s
    rng = np.random.default_rng(1)
    n, trials, hit = 60, 4000, 0
    for _ in range(trials):
        x = rng.exponential(size=n + 1)
        hit += x[n] <= oracle.conformal_quantile(x[:n], 0.9, 1e9)
    cov = hit / trials
    assert cov >= oracle.tau_s(0.9) - 3 * math.sqrt(0.05 / trials), cov


def _hard_case():
    # rows 0..7 are the tier-1 archive picks (all RoPE scores tie at 0, so the smallest positions win), the last 16
    # rows the window; row 40 carries the query's content direction and is left out: the hard query's argmax
    N, W = 64, 16
    rng = np.random.default_rng(2)
    cache = np.zeros((1, N, 576))
    cache[0, :, :512] = rng.standard_normal((N, 512)).round(2) * 0.01
    qc = rng.standard_normal((1, 1, 512)).round(1)
    cache[0, 40, :512] = (2.0 * qc[0, 0] / np.linalg.norm(qc[0, 0])).round(2)
    qr = np.zeros((1, 1, 64))
    qr[0, 0, 3] = 1.0
    t = torch.as_tensor(cache).to(torch.bfloat16)
    wl = datagen.Workload(B=1, H=1, N=N, dtype="bf16", cache=t, q_latent=torch.as_tensor(qc).to(torch.bfloat16),
                          q_rope=torch.as_tensor(qr).to(torch.bfloat16), rot=torch.eye(64),
                          planted_pos=torch.zeros(1, 0, dtype=torch.int64), planted_head=torch.zeros(0, dtype=torch.int64),
                          seed=0)
    return oracle.HostInputs(wl), wl, W


def pin_hard_query_zq():
    hi, wl, W = _hard_case()
    a = oracle.scores(hi)
    k = 8
    idx, cnt, _ = oracle.select(a, k, W)
    _, _, eta, pres = oracle.build_index(hi, 64)
    zq, ustar, n = oracle.calib_zq(hi, 64, LAM, a, eta, pres, idx, cnt)
    L = wl.latent.double().numpy()[0]
    qc = wl.q_latent.double().numpy()[0, 0]
    s = LAM * (L @ qc)                                          # RoPE scores are 0 here
    assert n == 1 and ustar[0, 0] == int(np.argmax(s)) == 40
    S = idx[0, 0, :cnt[0, 0]]
    assert 40 not in S.tolist()
    # the trigger rule at z_eff = zq / sqrt(512) puts row 40 exactly on s*: just above it fires, just below it does not
    _, _, smax = oracle.attention(hi, LAM, idx, cnt)
    for f, fires in ((1 + 1e-9, True), (1 - 1e-9, False)):
        z_eff = f * zq[0, 0] / math.sqrt(512.0)
        fidx, fcnt = oracle.trigger(hi, 64, LAM, z_eff, 0, a, eta, pres, idx, cnt, smax, W)
        assert (40 in fidx[0, 0, :fcnt[0, 0]].tolist()) == fires
    # the argmax inside the attended set: not hard
    idx2, cnt2, _ = oracle.select(a, 48, W)
    zq2, ustar2, n2 = oracle.calib_zq(hi, 64, LAM, a, eta, pres, idx2, cnt2)
    assert n2 == 0 and np.isnan(zq2[0, 0]) and ustar2[0, 0] == 40


PINS = [pin_paper_constants, pin_quantile_closed_form, pin_exchangeable_coverage, pin_hard_query_zq]


@pytest.mark.parametrize("pin", PINS, ids=lambda f: f.__name__)
def test_pin(pin):
    oracle.set_mutation(oracle.MUT_NONE)
    pin()


def test_planted_mistake_is_caught():
    oracle.set_mutation(oracle.MUT_CONFORMAL_FLOOR)
    try:
        with pytest.raises(AssertionError):
            pin_quantile_closed_form()
    finally:
        oracle.set_mutation(oracle.MUT_NONE)
