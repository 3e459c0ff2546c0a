"""The input recipe (seeded synthetic MLA decode workloads) checked against its statement, on CPU.

The generator holds none of the method's arithmetic; these tests pin what it draws: the value laws of the
latent and RoPE parts, the RoPE rotation of keys and queries, the planted rows, the log-normal key norms, bf16
round-to-nearest-even storage, the Haar rotation, and seeding.
"""
import math

import numpy as np
import torch

from paper_2609_03949_gb300 import datagen


def rope_angle(pos, i):
    return pos * 10000.0 ** (-2.0 * i / 64)


def test_value_laws_and_shapes():
    wl = datagen.make_workload(2, 16, 4096, dtype="f32", seed=3)
    assert wl.cache.shape == (2, 4096, 576) and wl.q_latent.shape == (2, 16, 512) and wl.q_rope.shape == (2, 16, 64)
    lat = wl.latent.double()
    assert abs(lat.mean().item()) < 2e-3
    assert abs(lat.std().item() * math.sqrt(512) - 1.0) < 0.01               # N(0,1)/sqrt(512)
    key_norm = wl.rope.double().norm(dim=-1)                                 # rotation keeps the chi_64 norm
    assert abs(key_norm.mean().item() - math.sqrt(2) * math.gamma(32.5) / math.gamma(32)) < 0.05
    assert abs(wl.q_latent.double().std().item() - 1.0) < 0.02


def test_keys_and_query_are_rotated_at_their_positions():
    # rotating back by the position's angles must leave an isotropic Gaussian key; check the rotation directly on
    # a key drawn through the same generator: pair i of position u turned by u * 10000^(-2i/64)
    N = 64
    wl = datagen.make_workload(1, 4, N, dtype="f32", seed=5)
    gen = torch.Generator().manual_seed(5)
    torch.randn(1, 4, 512, generator=gen)                                    # q_latent
    q_raw = torch.randn(1, 4, 64, generator=gen)
    torch.randn(N, 512, generator=gen)                                       # latent
    k_raw = torch.randn(N, 64, generator=gen).double()
    for u in (0, 1, 17, 63):
        for i in (0, 5, 31):
            a = rope_angle(u, i)
            c, s = math.cos(a), math.sin(a)
            x, y = k_raw[u, 2 * i].item(), k_raw[u, 2 * i + 1].item()
            got = wl.rope[0, u, 2 * i:2 * i + 2].double()
            np.testing.assert_allclose(got.numpy(), [x * c - y * s, x * s + y * c], rtol=1e-5, atol=1e-6)
    a = rope_angle(N, 3)
    x, y = q_raw[0, 2, 6].item(), q_raw[0, 2, 7].item()
    np.testing.assert_allclose(wl.q_rope[0, 2, 6:8].double().numpy(),
                               [x * math.cos(a) - y * math.sin(a), x * math.sin(a) + y * math.cos(a)], rtol=1e-5,
                               atol=1e-6)


def test_planted_rows():
    B, H, N = 3, 8, 2000
    wl = datagen.make_workload(B, H, N, dtype="f32", seed=7, n_planted=20, planted_lo=4, planted_hi=N - 256)
    assert wl.planted_pos.shape == (B, 20)
    assert wl.planted_head.tolist() == [p % H for p in range(20)]
    for b in range(B):
        pos = wl.planted_pos[b]
        assert len(set(pos.tolist())) == 20 and pos.min() >= 4 and pos.max() < N - 256
        for p, h in zip(pos.tolist(), wl.planted_head.tolist()):
            q = wl.q_rope[b, h].double()
            np.testing.assert_allclose(wl.rope[b, p].double().numpy(), (4.0 * q / q.norm()).numpy(), rtol=1e-6,
                                       atol=1e-6)


def test_lognormal_key_norms():
    wl = datagen.make_workload(1, 4, 20000, dtype="f32", seed=11, lognormal_keys=True)
    logn = np.log(wl.rope[0].double().norm(dim=-1).numpy() / 8.0)            # log of 8 exp(0.5 xi) / 8
    assert abs(logn.mean()) < 0.02 and abs(logn.std() - 0.5) < 0.01


def test_bf16_storage_is_round_to_nearest_even():
    f = datagen.make_workload(1, 4, 512, dtype="f32", seed=13)
    b = datagen.make_workload(1, 4, 512, dtype="bf16", seed=13)
    assert b.cache.dtype == torch.bfloat16
    np.testing.assert_array_equal(b.cache.float().numpy(), f.cache.to(torch.bfloat16).float().numpy())
    np.testing.assert_array_equal(b.q_rope.float().numpy(), f.q_rope.to(torch.bfloat16).float().numpy())


def test_haar_rotation_and_seeding():
    o = datagen.haar_orthogonal(17)
    np.testing.assert_allclose(o @ o.T, np.eye(64), atol=1e-12)
    g = np.random.default_rng(17).standard_normal((64, 64))             # the seeded Gaussian it factors
    r = o.T @ g                                                           # g = o r with r upper triangular,
    assert np.abs(np.tril(r, -1)).max() < 1e-10 and np.all(np.diag(r) > 0)   # positive diagonal (sign-fixed)
    a = datagen.make_workload(2, 4, 256, seed=21, n_planted=3)
    b = datagen.make_workload(2, 4, 256, seed=21, n_planted=3)
    c = datagen.make_workload(2, 4, 256, seed=22, n_planted=3)
    assert torch.equal(a.cache, b.cache) and torch.equal(a.planted_pos, b.planted_pos)
    assert not torch.equal(a.cache, c.cache)
