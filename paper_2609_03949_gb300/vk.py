"""ctypes binding of libvk.so (include/vk.h). Argument marshalling only: every step runs in the CUDA library.

Tensors are torch CUDA tensors; their ``data_ptr()`` is passed straight through. There is no CPU fallback:
loading fails loudly when libvk.so has not been built.
"""
from __future__ import annotations

import ctypes
import math
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libvk.so")

VK_OK, VK_ERR_INVALID_ARG, VK_ERR_UNSUPPORTED, VK_ERR_WORKSPACE = 0, -1, -2, -3
VK_ERR_CAPACITY, VK_ERR_CUDA, VK_ERR_TIMEOUT = -4, -5, -6
VK_BF16, VK_F32 = 0, 1
VK_TRIG_OFF, VK_TRIG_CS, VK_TRIG_CS_PAGE = 0, 1, 2
VK_FLAG_FORCE_FALLBACK, VK_FLAG_FORCE_DENSE, VK_FLAG_TEST_TIMEOUT, VK_FLAG_NO_PAGE_SKIP = 0x1, 0x2, 0x4, 0x8
VK_FLAG_FIRED_TILES = 0x10
D_LATENT, D_ROPE, PAGE = 512, 64, 64
DEFAULT_SM_SCALE = 1.0 / math.sqrt(192.0)


class VkError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"vk error {code}: {msg}")
        self.code = code


class vk_view(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int32), ("H", ctypes.c_int32), ("N", ctypes.c_int32), ("dtype", ctypes.c_int32),
                ("latent", ctypes.c_void_p), ("latent_ld", ctypes.c_int64), ("latent_bstride", ctypes.c_int64),
                ("rope", ctypes.c_void_p), ("rope_ld", ctypes.c_int64), ("rope_bstride", ctypes.c_int64),
                ("q_latent", ctypes.c_void_p), ("q_rope", ctypes.c_void_p)]


class vk_params(ctypes.Structure):
    _fields_ = [("rho", ctypes.c_double), ("r", ctypes.c_int32), ("window", ctypes.c_int32),
                ("n_sink", ctypes.c_int32), ("sm_scale", ctypes.c_float), ("trigger", ctypes.c_int32),
                ("z_eff", ctypes.c_float), ("top_j", ctypes.c_int32), ("flags", ctypes.c_uint32),
                ("r_sk", ctypes.c_int32)]


class vk_index(ctypes.Structure):
    _fields_ = [("digest", ctypes.c_void_p), ("eta", ctypes.c_void_p), ("page_res", ctypes.c_void_p),
                ("rot", ctypes.c_void_p), ("page_knorm", ctypes.c_void_p), ("page_eta", ctypes.c_void_p),
                ("sketch", ctypes.c_void_p), ("sketch_basis", ctypes.c_void_p)]


_lib = None


def lib():
    """Load libvk.so (built by ``paper_2609_03949_gb300._build.build()``); raises if it is missing."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is not built; run paper_2609_03949_gb300._build.build() first")
        L = ctypes.CDLL(LIB_PATH)
        P, I32, I64, SZ, D = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t, ctypes.c_double
        VP, PP, IP = ctypes.POINTER(vk_view), ctypes.POINTER(vk_params), ctypes.POINTER(vk_index)
        sig = {
            "vk_keep_count": ([I32, D, I32, I32], I64),
            "vk_min_cap": ([VP, PP], I32),
            "vk_workspace_bytes": ([VP, PP, I32], SZ),
            "vk_build_digest": ([VP, PP, P, P, P, P, P, P, P], ctypes.c_int),
            "vk_score": ([VP, PP, IP, P, P, SZ, P], ctypes.c_int),
            "vk_select": ([VP, PP, P, P, P, P, I32, P, SZ, P], ctypes.c_int),
            "vk_sparse_attn": ([VP, PP, P, P, I32, P, P, P, P, SZ, P], ctypes.c_int),
            "vk_decode_step": ([VP, PP, IP, P, P, P, P, P, I32, P, SZ, P], ctypes.c_int),
            "vk_decode_step_noalloc": ([VP, PP, IP, P, P, P, P, P, I32, P], ctypes.c_int),
            "vk_workspace_init": ([P, SZ, P], ctypes.c_int),
            "vk_poll_status": ([P, P], ctypes.c_int),
            "vk_profile_set_events": ([ctypes.POINTER(ctypes.c_void_p), I32], ctypes.c_int),
            "vk_profile_launches": ([], I64),
            "vk_last_error": ([], ctypes.c_char_p),
            "vk_sigma_workspace_bytes": ([I32, I32], SZ),
            "vk_pca_workspace_bytes": ([], SZ),
            "vk_conformal_workspace_bytes": ([VP, PP], SZ),
            "vk_conformal_z": ([VP, PP, IP, P, P, I32, ctypes.c_float, ctypes.c_float, P, P, P, SZ, P], ctypes.c_int),
            "vk_pca_basis": ([VP, P, P, P, SZ, P], ctypes.c_int),
            "vk_sigma": ([VP, I32, I32, P, P, SZ, P], ctypes.c_int),
            "vk_sigma_select": ([I32, I32, I32, P, I32, I64, P, P, I32, P, SZ, P], ctypes.c_int),
            "vk_build_sketch": ([VP, I32, P, P, P, P], ctypes.c_int),
            "vk_sketch_basis_workspace_bytes": ([I64, I32], SZ),
            "vk_sketch_basis": ([P, I32, I64, I32, P, P, P, SZ, P], ctypes.c_int),
        }
        for name, (args, res) in sig.items():
            fn = getattr(L, name)
            fn.argtypes = args
            fn.restype = res
        _lib = L
    return _lib


def exported_symbols():
    """Names of the C entry points declared in include/vk.h."""
    return ["vk_keep_count", "vk_min_cap", "vk_workspace_bytes", "vk_build_digest", "vk_score", "vk_select",
            "vk_sparse_attn", "vk_decode_step", "vk_decode_step_noalloc", "vk_workspace_init", "vk_poll_status",
            "vk_profile_set_events", "vk_profile_launches", "vk_last_error", "vk_sigma_workspace_bytes", "vk_sigma",
            "vk_sigma_select", "vk_pca_workspace_bytes", "vk_pca_basis", "vk_conformal_workspace_bytes",
            "vk_conformal_z", "vk_build_sketch", "vk_sketch_basis_workspace_bytes", "vk_sketch_basis"]


def _check(rc: int):
    if rc != VK_OK:
        raise VkError(rc, lib().vk_last_error().decode())


def _ptr(t) -> int | None:
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(stream) -> int | None:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


# ------------------------------------------------------------------------------------------------ structs
def make_view(cache: torch.Tensor, q_latent: torch.Tensor, q_rope: torch.Tensor) -> vk_view:
    """View of a [B, N, 576] cache (latent = [..., :512], rope = [..., 512:]) and the absorbed query."""
    if cache.dim() != 3 or cache.shape[-1] != D_LATENT + D_ROPE or cache.stride(-1) != 1:
        raise ValueError("cache must be [B, N, 576] with unit stride in the last dimension")
    if cache.dtype not in (torch.bfloat16, torch.float32) or q_latent.dtype != cache.dtype or q_rope.dtype != cache.dtype:
        raise ValueError("cache and queries must share dtype bf16 or f32")
    if not (q_latent.is_contiguous() and q_rope.is_contiguous()):
        raise ValueError("queries must be contiguous")
    B, N, _ = cache.shape
    esz = cache.element_size()
    return vk_view(B=B, H=q_latent.shape[1], N=N, dtype=VK_BF16 if cache.dtype == torch.bfloat16 else VK_F32,
                   latent=cache.data_ptr(), latent_ld=cache.stride(1), latent_bstride=cache.stride(0),
                   rope=cache.data_ptr() + D_LATENT * esz, rope_ld=cache.stride(1), rope_bstride=cache.stride(0),
                   q_latent=q_latent.data_ptr(), q_rope=q_rope.data_ptr())


def make_params(rho: float, r: int = 64, window: int = 0, n_sink: int = 0, sm_scale: float = DEFAULT_SM_SCALE,
                trigger: int = VK_TRIG_OFF, z_eff: float = 1.0, top_j: int = 0, flags: int = 0,
                r_sk: int = 0) -> vk_params:
    return vk_params(rho=rho, r=r, window=window, n_sink=n_sink, sm_scale=sm_scale, trigger=trigger, z_eff=z_eff,
                     top_j=top_j, flags=flags, r_sk=r_sk)


def make_index(digest=None, eta=None, page_res=None, rot=None, page_knorm=None, page_eta=None, sketch=None,
               sketch_basis=None) -> vk_index:
    return vk_index(digest=_ptr(digest), eta=_ptr(eta), page_res=_ptr(page_res), rot=_ptr(rot),
                    page_knorm=_ptr(page_knorm), page_eta=_ptr(page_eta), sketch=_ptr(sketch),
                    sketch_basis=_ptr(sketch_basis))


# ------------------------------------------------------------------------------------------------ entry points
def vk_keep_count(N: int, rho: float, window: int, n_sink: int = 0) -> int:
    return int(lib().vk_keep_count(N, rho, window, n_sink))


def vk_min_cap(view: vk_view, params: vk_params) -> int:
    return int(lib().vk_min_cap(ctypes.byref(view), ctypes.byref(params)))


def vk_workspace_bytes(view: vk_view, params: vk_params, cap: int) -> int:
    n = int(lib().vk_workspace_bytes(ctypes.byref(view), ctypes.byref(params), cap))
    if n == 0:
        raise VkError(VK_ERR_INVALID_ARG, lib().vk_last_error().decode())
    return n


def vk_workspace_init(ws: torch.Tensor, stream=None) -> None:
    _check(lib().vk_workspace_init(_ptr(ws), ws.numel() * ws.element_size(), _stream(stream)))


def vk_build_digest(view, params, rot, digest=None, eta=None, page_res=None, page_knorm=None, page_eta=None,
                    stream=None) -> None:
    _check(lib().vk_build_digest(ctypes.byref(view), ctypes.byref(params), _ptr(rot), _ptr(digest), _ptr(eta),
                                 _ptr(page_res), _ptr(page_knorm), _ptr(page_eta), _stream(stream)))


def vk_score(view, params, index: vk_index | None, scores: torch.Tensor, ws: torch.Tensor, stream=None) -> None:
    _check(lib().vk_score(ctypes.byref(view), ctypes.byref(params), ctypes.byref(index) if index else None,
                          _ptr(scores), _ptr(ws), ws.numel() * ws.element_size(), _stream(stream)))


def vk_select(view, params, scores, idx, count, kth=None, ws=None, stream=None) -> None:
    nb = 0 if ws is None else ws.numel() * ws.element_size()
    _check(lib().vk_select(ctypes.byref(view), ctypes.byref(params), _ptr(scores), _ptr(idx), _ptr(count), _ptr(kth),
                           idx.shape[-1], _ptr(ws), nb, _stream(stream)))


def vk_sparse_attn(view, params, idx, count, out, lse=None, smax=None, ws=None, stream=None) -> None:
    nb = 0 if ws is None else ws.numel() * ws.element_size()
    _check(lib().vk_sparse_attn(ctypes.byref(view), ctypes.byref(params), _ptr(idx), _ptr(count), idx.shape[-1],
                                _ptr(out), _ptr(lse), _ptr(smax), _ptr(ws), nb, _stream(stream)))


def vk_decode_step(view, params, index: vk_index | None, out, lse, smax, idx, count, ws, stream=None) -> None:
    _check(lib().vk_decode_step(ctypes.byref(view), ctypes.byref(params), ctypes.byref(index) if index else None,
                                _ptr(out), _ptr(lse), _ptr(smax), _ptr(idx), _ptr(count), idx.shape[-1], _ptr(ws),
                                ws.numel() * ws.element_size(), _stream(stream)))


def vk_profile_set_events(events) -> None:
    """Record these 7 torch.cuda.Event objects at the stage boundaries of later vk_decode_step calls
    (None or [] turns recording off)."""
    events = list(events or [])
    for e in events:
        if e.cuda_event == 0:
            e.record()  # materialise the underlying cudaEvent_t
    arr = (ctypes.c_void_p * max(1, len(events)))(*[e.cuda_event for e in events])
    _check(lib().vk_profile_set_events(arr, len(events)))


def vk_profile_launches() -> int:
    return int(lib().vk_profile_launches())


def vk_decode_step_noalloc(view, params, index: vk_index | None, out, lse, smax, idx, count, stream=None) -> None:
    """vk_decode_step with the library's static scratch instead of a workspace (see include/vk.h)."""
    _check(lib().vk_decode_step_noalloc(ctypes.byref(view), ctypes.byref(params),
                                        ctypes.byref(index) if index else None, _ptr(out), _ptr(lse), _ptr(smax),
                                        _ptr(idx), _ptr(count), idx.shape[-1], _stream(stream)))


def vk_poll_status(ws: torch.Tensor, stream=None) -> int:
    """Device status since the last poll (VK_OK or a negative vk_status); the word is cleared."""
    return int(lib().vk_poll_status(_ptr(ws), _stream(stream)))


# ------------------------------------------------------------------------------------------------ plumbing
def alloc_workspace(view: vk_view, params: vk_params, cap: int, device="cuda") -> torch.Tensor:
    """A zero-initialised workspace of vk_workspace_bytes() (allocated by torch, 256-byte aligned)."""
    n = vk_workspace_bytes(view, params, cap)
    ws = torch.empty(n + 256, dtype=torch.uint8, device=device)
    off = (-ws.data_ptr()) % 256
    ws = ws[off:off + n]
    vk_workspace_init(ws)
    return ws


class DecodeBuffers:
    """Outputs and workspace of vk_decode_step for one set of shapes (allocated once, reused every step)."""

    def __init__(self, view: vk_view, params: vk_params, cap: int | None = None, device="cuda"):
        B, H = view.B, view.H
        self.cap = cap if cap is not None else (view.N if params.trigger else vk_min_cap(view, params))
        self.out = torch.empty(B, H, D_LATENT, dtype=torch.float32, device=device)
        self.lse = torch.empty(B, H, dtype=torch.float32, device=device)
        self.smax = torch.empty(B, H, dtype=torch.float32, device=device)
        self.idx = torch.empty(B, H, self.cap, dtype=torch.int32, device=device)
        self.count = torch.empty(B, H, dtype=torch.int32, device=device)
        self.ws = alloc_workspace(view, params, self.cap, device)

    def run(self, view, params, index=None, stream=None):
        vk_decode_step(view, params, index, self.out, self.lse, self.smax, self.idx, self.count, self.ws, stream)


# ------------------------------------------------------------------------------------------------ sigma selector
def vk_sigma_workspace_bytes(T: int, kappa: int) -> int:
    n = int(lib().vk_sigma_workspace_bytes(T, kappa))
    if n == 0:
        raise VkError(VK_ERR_INVALID_ARG, f"bad sigma parameters T={T} kappa={kappa}")
    return n


def vk_sigma(view, T: int, kappa: int, sigma, ws, stream=None) -> None:
    _check(lib().vk_sigma(ctypes.byref(view), T, kappa, _ptr(sigma), _ptr(ws), ws.numel() * ws.element_size(),
                          _stream(stream)))


def vk_sigma_select(B: int, N: int, T: int, sigma, n_sink: int, m: int, idx, count, ws, stream=None) -> None:
    _check(lib().vk_sigma_select(B, N, T, _ptr(sigma), n_sink, m, _ptr(idx), _ptr(count), idx.shape[-1], _ptr(ws),
                                 ws.numel() * ws.element_size(), _stream(stream)))


def alloc_bytes(n: int, device="cuda") -> torch.Tensor:
    """A zeroed, 256-byte aligned device buffer of n bytes (allocated by torch)."""
    buf = torch.zeros(n + 256, dtype=torch.uint8, device=device)
    off = (-buf.data_ptr()) % 256
    return buf[off:off + n]


# ------------------------------------------------------------------------------------------------ PCA digest basis
def vk_pca_basis(view, rot, eig=None, ws=None, stream=None) -> None:
    """Principal directions of the view's RoPE branch as the rows of rot [64, 64] fp32 (eigenvalues into eig)."""
    if ws is None:
        ws = alloc_bytes(int(lib().vk_pca_workspace_bytes()))
    _check(lib().vk_pca_basis(ctypes.byref(view), _ptr(rot), _ptr(eig), _ptr(ws), ws.numel() * ws.element_size(),
                              _stream(stream)))


# ------------------------------------------------------------------------------------------------ content sketch
def vk_build_sketch(view, r_sk: int, basis, sketch=None, eta=None, stream=None) -> None:
    """Sketch index entry of every cached row: sketch [B, N, r_sk] bf16 = V_r^T L_u, eta [B, N] fp32 its residual."""
    _check(lib().vk_build_sketch(ctypes.byref(view), int(r_sk), _ptr(basis), _ptr(sketch), _ptr(eta), _stream(stream)))


def vk_sketch_basis(queries: torch.Tensor, r_sk: int, basis, eig=None, ws=None, stream=None):
    """Sketch basis [r_sk, 512] fp32 (rows) from the context's queries [n, 512] (bf16 or fp32, contiguous)."""
    q = queries
    if q.dim() != 2 or q.shape[1] != D_LATENT or not q.is_contiguous():
        raise ValueError("queries must be a contiguous [n, 512] tensor")
    dt = VK_BF16 if q.dtype == torch.bfloat16 else VK_F32
    if ws is None:
        n = int(lib().vk_sketch_basis_workspace_bytes(q.shape[0], int(r_sk)))
        if n == 0:
            raise VkError(VK_ERR_INVALID_ARG, lib().vk_last_error().decode())
        ws = alloc_bytes(n)
    _check(lib().vk_sketch_basis(_ptr(q), dt, q.shape[0], int(r_sk), _ptr(basis), _ptr(eig), _ptr(ws),
                                 ws.numel() * ws.element_size(), _stream(stream)))
    return ws


# ------------------------------------------------------------------------------------------------ conformal z
def vk_conformal_z(view, params, index, idx, count, zq, z_out, tau: float = 0.9, z_max: float = 8.0, ws=None,
                   stream=None) -> None:
    """Calibrate the trigger's z from every (b, h) as a calibration query (S_h given by idx/count)."""
    if ws is None:
        n = int(lib().vk_conformal_workspace_bytes(ctypes.byref(view), ctypes.byref(params)))
        if n == 0:
            raise VkError(VK_ERR_INVALID_ARG, lib().vk_last_error().decode())
        ws = alloc_bytes(n)
    _check(lib().vk_conformal_z(ctypes.byref(view), ctypes.byref(params), ctypes.byref(index), _ptr(idx), _ptr(count),
                                idx.shape[-1], float(tau), float(z_max), _ptr(zq), _ptr(z_out), _ptr(ws),
                                ws.numel() * ws.element_size(), _stream(stream)))
    return ws
