"""vk_decode_step_noalloc: the decode step for callers that cannot allocate device memory (a plugin limited to
memory its host gave it, or a serving loop that forbids cudaMalloc after start-up). It takes its scratch from
a static device array of the library instead of a workspace. Checked through the C ABI against the
workspace-taking vk_decode_step on the same inputs, on two calls in a row (the array keeps the previous
call's contents, so the second call shows that nothing stale leaks into it).

This file is collected last on purpose, so a run that stops at the first failure has run every other test.
"""
import ctypes

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu

OUT_RTOL = 2e-2    # the output tolerance every parity test uses
LSE_ATOL = 2e-2


def test_noalloc_matches_workspace_entry_point():
    from paper_2609_03949_gb300 import _build, datagen, vk
    _build.build()
    L = vk.lib()
    wl = datagen.make_workload(2, 64, 4096, seed=31, n_planted=16, planted_hi=4096 - 128, device="cuda")
    view = vk.make_view(wl.cache, wl.q_latent, wl.q_rope)
    params = vk.make_params(1 / 32, window=128)
    assert vk.vk_workspace_bytes(view, params, vk.vk_min_cap(view, params)) <= (16 << 20)

    ref = vk.DecodeBuffers(view, params)
    ref.run(view, params)
    torch.cuda.synchronize()
    assert vk.vk_poll_status(ref.ws) == vk.VK_OK
    cap = ref.cap
    out = torch.empty_like(ref.out)
    lse = torch.empty_like(ref.lse)
    smax = torch.empty_like(ref.smax)
    idx = torch.empty_like(ref.idx)
    count = torch.empty_like(ref.count)
    stream = torch.cuda.current_stream().cuda_stream
    for call in range(2):
        for t in (out, lse, smax):
            t.fill_(float("nan"))
        idx.fill_(-7)
        count.fill_(-7)
        rc = L.vk_decode_step_noalloc(ctypes.byref(view), ctypes.byref(params), None, out.data_ptr(),
                                      lse.data_ptr(), smax.data_ptr(), idx.data_ptr(), count.data_ptr(), cap,
                                      stream)
        assert rc == vk.VK_OK, L.vk_last_error().decode()
        torch.cuda.synchronize()
        o, r = out.cpu().double().numpy(), ref.out.cpu().double().numpy()
        rel = np.abs(o - r).max(-1) / np.abs(r).max(-1)
        assert rel.max() <= OUT_RTOL, (call, rel.max())
        assert np.abs(lse.cpu().double().numpy() - ref.lse.cpu().double().numpy()).max() <= LSE_ATOL
        np.testing.assert_array_equal(count.cpu().numpy(), ref.count.cpu().numpy())
        np.testing.assert_array_equal(idx.cpu().numpy(), ref.idx.cpu().numpy())


def test_noalloc_rejects_problems_beyond_its_scratch():
    from paper_2609_03949_gb300 import _build, datagen, vk
    _build.build()
    L = vk.lib()
    wl = datagen.make_workload(1, 64, 8, seed=1, device="cuda")   # real, tiny buffers; the view claims more rows
    view = vk.make_view(wl.cache, wl.q_latent, wl.q_rope)
    view.N = 1 << 20
    view.B = 4
    view.latent_bstride = view.rope_bstride = (1 << 20) * 576
    params = vk.make_params(1 / 32, window=256)
    assert vk.vk_workspace_bytes(view, params, 40000) > (16 << 20)
    dummy = torch.empty(4, 64, 512, device="cuda")
    rc = L.vk_decode_step_noalloc(ctypes.byref(view), ctypes.byref(params), None, dummy.data_ptr(),
                                  dummy.data_ptr(), None, dummy.data_ptr(), dummy.data_ptr(), 40000,
                                  torch.cuda.current_stream().cuda_stream)
    assert rc == vk.VK_ERR_WORKSPACE
    assert "static scratch" in L.vk_last_error().decode()
