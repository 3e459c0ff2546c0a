"""The C ABI without a GPU: libvk.so builds and loads, exports every entry point include/vk.h declares, and
refuses bad arguments on the host before any launch (so these run on a CPU-only machine)."""
import ctypes
import os
import re

import pytest

from paper_2609_03949_gb300 import _build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def vk():
    _build.build()
    from paper_2609_03949_gb300 import vk as mod
    mod.lib()
    return mod


def declared_functions():
    text = open(os.path.join(ROOT, "include", "vk.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(vk_[a-z_]+)\s*\(", text)))


def test_header_and_binding_agree(vk):
    assert declared_functions() == sorted(vk.exported_symbols())


def test_every_declared_symbol_is_exported(vk):
    lib = ctypes.CDLL(vk.LIB_PATH)
    for name in declared_functions():
        assert hasattr(lib, name), name


FAKE = 1 << 32   # a 16-byte aligned pointer value; never dereferenced because validation refuses first


def fake_view(vk, B=2, H=8, N=1000, dtype=0, **kw):
    esz = 2 if dtype == 0 else 4
    v = dict(B=B, H=H, N=N, dtype=dtype, latent=FAKE, latent_ld=576, latent_bstride=N * 576,
             rope=FAKE + 512 * esz, rope_ld=576, rope_bstride=N * 576, q_latent=FAKE, q_rope=FAKE)
    v.update(kw)
    return vk.vk_view(**v)


def test_keep_count_and_min_cap(vk):
    assert vk.vk_keep_count(1024, 1 / 8, 64) == 128
    assert vk.vk_keep_count(1001, 1 / 8, 0) == 126
    assert vk.vk_keep_count(100, 0.5, 90) == 10
    assert vk.vk_keep_count(100, 0.0, 0) == -1
    assert vk.vk_keep_count(100, 0.5, 101) == -1
    v = fake_view(vk, N=65536, H=64)
    assert vk.vk_min_cap(v, vk.make_params(1 / 32, window=256)) == 2048 + 256
    assert vk.vk_min_cap(v, vk.make_params(1 / 32, window=256, n_sink=4)) == 2048 + 256 + 4


def test_workspace_bytes_grows_with_shapes(vk):
    p = vk.make_params(1 / 32, window=256)
    small = vk.vk_workspace_bytes(fake_view(vk, N=4096), p, 400)
    big = vk.vk_workspace_bytes(fake_view(vk, N=65536), p, 2400)
    two = vk.vk_workspace_bytes(fake_view(vk, N=65536), vk.make_params(1 / 32, window=256, trigger=1), 65536)
    assert 0 < small < big < two
    assert small % 256 == 0


def call_decode(vk, view, params, index=None, cap=None, ws_bytes=1 << 40, out=FAKE, idx=FAKE):
    L = vk.lib()
    cap = cap if cap is not None else 1 << 20
    return L.vk_decode_step(ctypes.byref(view), ctypes.byref(params), ctypes.byref(index) if index else None,
                            out, FAKE, None, idx, FAKE, cap, FAKE, ws_bytes, None)


BAD_VIEWS = [
    dict(B=0), dict(H=0), dict(N=0), dict(N=1 << 24), dict(H=300), dict(dtype=7), dict(latent=0), dict(q_rope=0),
    dict(latent=FAKE + 8), dict(rope=FAKE + 2), dict(latent_ld=500), dict(rope_ld=63), dict(latent_ld=580),
    dict(latent_bstride=576 * 100),
]


@pytest.mark.parametrize("bad", BAD_VIEWS, ids=lambda d: ",".join(f"{k}={v}" for k, v in d.items()))
def test_bad_view_is_refused(vk, bad):
    rc = call_decode(vk, fake_view(vk, **bad), vk.make_params(1 / 8, window=16))
    assert rc in (vk.VK_ERR_INVALID_ARG, vk.VK_ERR_UNSUPPORTED)
    assert vk.lib().vk_last_error().decode()


BAD_PARAMS = [
    dict(rho=0.0), dict(rho=1.5), dict(rho=float("nan")), dict(r=12), dict(r=128), dict(window=-1),
    dict(window=1001), dict(n_sink=-1), dict(window=990, n_sink=20), dict(sm_scale=0.0),
    dict(sm_scale=float("inf")), dict(trigger=5), dict(z_eff=-1.0), dict(top_j=-3), dict(flags=0x80),
]


@pytest.mark.parametrize("bad", BAD_PARAMS, ids=lambda d: ",".join(f"{k}={v}" for k, v in d.items()))
def test_bad_params_are_refused(vk, bad):
    p = dict(rho=1 / 8, window=16)
    p.update(bad)
    rc = call_decode(vk, fake_view(vk), vk.make_params(**p))
    assert rc == vk.VK_ERR_INVALID_ARG, vk.lib().vk_last_error().decode()


def test_cap_workspace_and_index_are_checked(vk):
    v, p = fake_view(vk), vk.make_params(1 / 8, window=16)
    k = vk.vk_keep_count(1000, 1 / 8, 16)
    assert call_decode(vk, v, p, cap=k + 15) == vk.VK_ERR_INVALID_ARG
    assert call_decode(vk, v, p, ws_bytes=1024) == vk.VK_ERR_WORKSPACE
    # a digest width needs the digest and the rotation
    assert call_decode(vk, v, vk.make_params(1 / 8, r=16, window=16)) == vk.VK_ERR_INVALID_ARG
    # the trigger needs eta and page_res
    assert call_decode(vk, v, vk.make_params(1 / 8, window=16, trigger=1)) == vk.VK_ERR_INVALID_ARG
    idx = vk.make_index(eta=FAKE, page_res=None)
    assert call_decode(vk, v, vk.make_params(1 / 8, window=16, trigger=1), index=idx) == vk.VK_ERR_INVALID_ARG
    # the page skip's two page arrays go together; the page trigger needs both
    idx = vk.make_index(eta=FAKE, page_res=FAKE, page_knorm=FAKE)
    assert call_decode(vk, v, vk.make_params(1 / 8, window=16, trigger=1), index=idx) == vk.VK_ERR_INVALID_ARG
    idx = vk.make_index(eta=FAKE, page_res=FAKE, page_eta=FAKE)
    assert call_decode(vk, v, vk.make_params(1 / 8, window=16, trigger=2), index=idx) == vk.VK_ERR_INVALID_ARG
    assert call_decode(vk, v, vk.make_params(1 / 8, window=16, trigger=3)) == vk.VK_ERR_INVALID_ARG
    assert call_decode(vk, v, p, out=FAKE + 4) == vk.VK_ERR_INVALID_ARG


def test_other_entry_points_refuse(vk):
    L = vk.lib()
    v, p = fake_view(vk), vk.make_params(1 / 8, window=16)
    assert L.vk_score(ctypes.byref(v), ctypes.byref(p), None, None, FAKE, 1 << 40, None) == vk.VK_ERR_INVALID_ARG
    assert L.vk_select(ctypes.byref(v), ctypes.byref(p), FAKE, FAKE, FAKE, None, 3, None, 0, None) == vk.VK_ERR_INVALID_ARG
    assert L.vk_sparse_attn(ctypes.byref(v), ctypes.byref(p), FAKE, FAKE, 10, FAKE, None, None, None, 0,
                            None) == vk.VK_ERR_WORKSPACE
    assert L.vk_build_digest(ctypes.byref(v), ctypes.byref(vk.make_params(1 / 8, r=8)), None, FAKE, None, None,
                             None, None, None) == vk.VK_ERR_INVALID_ARG
    assert L.vk_build_digest(ctypes.byref(v), ctypes.byref(p), None, None, None, None, FAKE + 4, None,
                             None) == vk.VK_ERR_INVALID_ARG
    assert L.vk_poll_status(None, None) == vk.VK_ERR_WORKSPACE
    assert L.vk_workspace_init(None, 0, None) == vk.VK_ERR_WORKSPACE


def test_sigma_entry_points_refuse(vk):
    L = vk.lib()
    v = fake_view(vk, N=20000)
    assert L.vk_sigma_workspace_bytes(4096, 16) > 0
    assert L.vk_sigma_workspace_bytes(4000, 16) == 0          # T must be a multiple of 128
    assert L.vk_sigma_workspace_bytes(4096, 65) == 0          # kappa in [1, 64]
    nb = L.vk_sigma_workspace_bytes(4096, 16)
    assert L.vk_sigma(ctypes.byref(v), 4000, 16, FAKE, FAKE, nb, None) == vk.VK_ERR_INVALID_ARG
    assert L.vk_sigma(ctypes.byref(v), 4096, 0, FAKE, FAKE, nb, None) == vk.VK_ERR_INVALID_ARG
    assert L.vk_sigma(ctypes.byref(v), 4096, 16, FAKE, FAKE, nb - 1, None) == vk.VK_ERR_WORKSPACE
    assert L.vk_sigma(ctypes.byref(v), 4096, 16, None, FAKE, nb, None) == vk.VK_ERR_INVALID_ARG
    assert L.vk_sigma(ctypes.byref(fake_view(vk, N=20000, dtype=1)), 4096, 16, FAKE, FAKE, nb, None) == \
        vk.VK_ERR_UNSUPPORTED
    # the attended set must fit: sinks + m + open tail (20000 rows: 4 closed blocks, a tail of 3616)
    assert L.vk_sigma_select(2, 20000, 4096, FAKE, 4, 100, FAKE, FAKE, 3616 + 104 - 1, FAKE, 256, None) == \
        vk.VK_ERR_INVALID_ARG
    assert L.vk_sigma_select(2, 20000, 4096, FAKE, 4, 100, FAKE, FAKE, 3720, FAKE, 255, None) == vk.VK_ERR_WORKSPACE


def test_sketch_entry_points_refuse(vk):
    L = vk.lib()
    v = fake_view(vk)
    # the sketch rank: 0, 16, 32 or 64, and only with the row-level trigger
    assert call_decode(vk, v, vk.make_params(1 / 8, window=16, trigger=1, r_sk=24)) == vk.VK_ERR_INVALID_ARG
    assert call_decode(vk, v, vk.make_params(1 / 8, window=16, trigger=0, r_sk=16)) == vk.VK_ERR_INVALID_ARG
    assert call_decode(vk, v, vk.make_params(1 / 8, window=16, trigger=2, r_sk=16)) == vk.VK_ERR_INVALID_ARG
    # with r_sk > 0 the index needs the stored sketch and its basis
    idx = vk.make_index(eta=FAKE, page_res=FAKE)
    assert call_decode(vk, v, vk.make_params(1 / 8, window=16, trigger=1, r_sk=16), index=idx) == vk.VK_ERR_INVALID_ARG
    idx = vk.make_index(eta=FAKE, page_res=FAKE, sketch=FAKE, sketch_basis=FAKE + 4)
    assert call_decode(vk, v, vk.make_params(1 / 8, window=16, trigger=1, r_sk=16), index=idx) == vk.VK_ERR_INVALID_ARG
    assert L.vk_build_sketch(ctypes.byref(v), 8, FAKE, FAKE, FAKE, None) == vk.VK_ERR_INVALID_ARG
    assert L.vk_build_sketch(ctypes.byref(v), 16, None, FAKE, FAKE, None) == vk.VK_ERR_INVALID_ARG
    assert L.vk_build_sketch(ctypes.byref(v), 16, FAKE, FAKE + 2, None, None) == vk.VK_ERR_INVALID_ARG
    nb = L.vk_sketch_basis_workspace_bytes(100, 32)
    assert nb > 0
    assert L.vk_sketch_basis_workspace_bytes(20, 32) == 0     # 20 queries cannot span 32 directions
    assert L.vk_sketch_basis_workspace_bytes(100, 48) == 0
    assert L.vk_sketch_basis(FAKE, 0, 20, 32, FAKE, None, FAKE, nb, None) == vk.VK_ERR_INVALID_ARG
    assert L.vk_sketch_basis(FAKE, 3, 100, 32, FAKE, None, FAKE, nb, None) == vk.VK_ERR_INVALID_ARG
    assert L.vk_sketch_basis(FAKE, 0, 100, 32, FAKE, None, FAKE, nb - 1, None) == vk.VK_ERR_WORKSPACE
