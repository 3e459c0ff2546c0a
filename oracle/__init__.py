"""CPU oracle for the VestigeKV decode hot path (plain C, fp64).

TEST INFRASTRUCTURE ONLY: the test suite, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` are the only callers. The product (the CUDA library and its binding) never imports this
package. The C source is ``vk_oracle.c``; ``build()`` compiles it with gcc.

Every function takes a :class:`paper_2609_03949_gb300.datagen.Workload`-like set of host arrays, passes
their raw storage (bf16 bits or fp32) to C, and returns numpy arrays in fp64.
"""
from __future__ import annotations

import ctypes
import math
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "vk_oracle.c")
_LIB_PATH = os.path.join(_HERE, "libvk_oracle.so")
_lib = None

D_LATENT, D_ROPE, PAGE = 512, 64, 64

# Deliberate mistakes the "known-bad first" tests plant in the oracle (see vk_oracle.c).
MUT_NONE, MUT_TIE_LARGER, MUT_DROP_WINDOW, MUT_SCALE_SQUARED = 0, 1, 2, 3
MUT_ROT_TRANSPOSE, MUT_DROP_ROPE, MUT_TRIGGER_NO_Z, MUT_SIGMA_ONE_SIDED = 4, 5, 6, 7
MUT_PCA_ASCENDING, MUT_CONFORMAL_FLOOR, MUT_SKETCH_QNORM = 8, 9, 10


def build(force: bool = False) -> str:
    """Compile vk_oracle.c into libvk_oracle.so (gcc, -O2, OpenMP over (batch, head))."""
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.run(["gcc", "-O2", "-fopenmp", "-fPIC", "-shared", "-std=c11", "-o", tmp, _SRC, "-lm"],
                       check=True)
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


class _View(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int32), ("H", ctypes.c_int32), ("N", ctypes.c_int32), ("dtype", ctypes.c_int32),
                ("latent", ctypes.c_void_p), ("latent_ld", ctypes.c_int64), ("latent_bstride", ctypes.c_int64),
                ("rope", ctypes.c_void_p), ("rope_ld", ctypes.c_int64), ("rope_bstride", ctypes.c_int64),
                ("q_latent", ctypes.c_void_p), ("q_rope", ctypes.c_void_p)]


def lib():
    global _lib
    if _lib is None:
        build()
        L = ctypes.CDLL(_LIB_PATH)
        P, I32, I64, D, F = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_double, ctypes.c_float
        VP = ctypes.POINTER(_View)
        L.vko_keep_count.argtypes = [I32, D, I32, I32]
        L.vko_keep_count.restype = I64
        L.vko_bf16_rne.argtypes = [D]
        L.vko_bf16_rne.restype = ctypes.c_uint16
        L.vko_build_index.argtypes = [VP, I32, P, P, P, P, P]
        L.vko_scores.argtypes = [VP, I32, P, P, P]
        L.vko_select.argtypes = [I32, I32, I32, P, I64, I32, I32, I32, P, P, P]
        L.vko_attention.argtypes = [VP, D, P, P, I32, P, P, P]
        L.vko_trigger.argtypes = [VP, I32, P, D, D, I32, P, P, P, I32, P, P, P, P, P, I32, P, I32, I32, I32, P, P]
        L.vko_page_norms.argtypes = [VP, P, P]
        L.vko_trigger_page.argtypes = [VP, D, D, I32, P, P, P, P, I32, P, I32, I32, I32, P, P]
        L.vko_decode_step.argtypes = [VP, D, I32, I32, I32, D, I32, D, I32, P, P, I32, P, P, I32, P, P, P, P, P, P]
        L.vko_decode_step.restype = ctypes.c_int
        L.vko_sigma.argtypes = [P, I64, I32, I32, P]
        L.vko_sigma_select.argtypes = [P, I64, I32, I32, I64, P]
        L.vko_sigma_select.restype = I64
        L.vko_second_moment.argtypes = [VP, P]
        L.vko_sym_eig.argtypes = [P, P, P]
        L.vko_pca_basis.argtypes = [VP, P, P]
        L.vko_tau_s.argtypes = [D]
        L.vko_tau_s.restype = D
        L.vko_min_hard.argtypes = [D]
        L.vko_min_hard.restype = I64
        L.vko_conformal_quantile.argtypes = [P, I64, D, D]
        L.vko_conformal_quantile.restype = D
        L.vko_calib_zq.argtypes = [VP, I32, P, D, P, P, P, I32, P, P, P, P, P, I32, P, P]
        L.vko_calib_zq.restype = I64
        L.vko_sketch_basis.argtypes = [P, I64, I32, P, P]
        L.vko_sketch_basis.restype = ctypes.c_int
        L.vko_build_sketch.argtypes = [VP, I32, P, P, P, P]
        L.vko_sketch_query.argtypes = [VP, I32, P, P, P]
        L.vko_set_mutation.argtypes = [ctypes.c_int]
        L.vko_num_threads.restype = ctypes.c_int
        L.vko_set_threads.argtypes = [ctypes.c_int]
        del F
        _lib = L
    return _lib


def _ptr(a: np.ndarray) -> int:
    return a.ctypes.data if a is not None else 0


class HostInputs:
    """Host copies of one workload in its storage format, kept alive while C reads them."""

    def __init__(self, wl):
        import torch
        self.B, self.H, self.N, self.dtype = wl.B, wl.H, wl.N, wl.dtype
        if wl.dtype == "bf16":
            conv = lambda t: t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)
        else:
            conv = lambda t: t.detach().cpu().contiguous().float().numpy()
        self.cache = conv(wl.cache)
        self.q_latent = conv(wl.q_latent)
        self.q_rope = conv(wl.q_rope)
        self.rot = wl.rot.detach().cpu().contiguous().float().numpy()
        esz = self.cache.itemsize
        row = self.cache.shape[-1]
        self.view = _View(B=self.B, H=self.H, N=self.N, dtype=0 if self.dtype == "bf16" else 1,
                          latent=self.cache.ctypes.data, latent_ld=row, latent_bstride=self.N * row,
                          rope=self.cache.ctypes.data + D_LATENT * esz, rope_ld=row, rope_bstride=self.N * row,
                          q_latent=self.q_latent.ctypes.data, q_rope=self.q_rope.ctypes.data)


def set_mutation(m: int) -> None:
    lib().vko_set_mutation(int(m))


def num_threads() -> int:
    return int(lib().vko_num_threads())


def set_threads(n: int) -> None:
    """OpenMP threads of the oracle's (b, h) loops from now on."""
    lib().vko_set_threads(int(n))


def keep_count(N: int, rho: float, window: int, n_sink: int = 0) -> int:
    """k = min(ceil(rho*N), |A|), A = [n_sink, N-W)."""
    return int(lib().vko_keep_count(N, rho, window, n_sink))


def bf16_rne(x: float) -> int:
    return int(lib().vko_bf16_rne(float(x)))


def build_index(hi: HostInputs, r: int):
    """(digest fp64 [B,N,r] or None, digest bf16 bits [B,N,r] or None, eta [B,N], page_res [B,P])."""
    B, N = hi.B, hi.N
    P = (N + PAGE - 1) // PAGE
    dig = np.zeros((B, N, r), np.float64) if r < D_ROPE else None
    dig16 = np.zeros((B, N, r), np.uint16) if r < D_ROPE else None
    eta = np.zeros((B, N), np.float64)
    pres = np.zeros((B, P), np.float64)
    lib().vko_build_index(ctypes.byref(hi.view), r, _ptr(hi.rot), _ptr(dig), _ptr(dig16), _ptr(eta), _ptr(pres))
    return dig, dig16, eta, pres


def scores(hi: HostInputs, r: int = 64, digest_bf16: np.ndarray | None = None) -> np.ndarray:
    """a[b,h,u] (unscaled RoPE-branch or digest score), fp64 [B,H,N]."""
    a = np.zeros((hi.B, hi.H, hi.N), np.float64)
    dg = None if digest_bf16 is None else np.ascontiguousarray(digest_bf16, dtype=np.uint16)
    if r < D_ROPE and dg is None:
        raise ValueError("a width-r digest needs the stored bf16 digest")
    lib().vko_scores(ctypes.byref(hi.view), r, _ptr(hi.rot), _ptr(dg), _ptr(a))
    return a


def select(a: np.ndarray, k: int, window: int, n_sink: int = 0, cap: int | None = None):
    """(idx [B,H,cap] int32, count [B,H] int32, kth [B,H] fp64) — per-head top-k + window (+ sinks)."""
    a = np.ascontiguousarray(a, dtype=np.float64)
    B, H, N = a.shape
    cap = cap if cap is not None else max(1, k + window + n_sink)
    idx = np.full((B, H, cap), -1, np.int32)
    count = np.zeros((B, H), np.int32)
    kth = np.zeros((B, H), np.float64)
    lib().vko_select(B, H, N, _ptr(a), k, window, n_sink, cap, _ptr(idx), _ptr(count), _ptr(kth))
    return idx, count, kth


def attention(hi: HostInputs, lam: float, idx: np.ndarray, count: np.ndarray):
    """(out [B,H,512], lse [B,H], smax [B,H]) over the attended sets idx[b,h,:count]."""
    idx = np.ascontiguousarray(idx, dtype=np.int32)
    count = np.ascontiguousarray(count, dtype=np.int32)
    cap = idx.shape[-1]
    out = np.zeros((hi.B, hi.H, D_LATENT), np.float64)
    lse = np.zeros((hi.B, hi.H), np.float64)
    smax = np.zeros((hi.B, hi.H), np.float64)
    lib().vko_attention(ctypes.byref(hi.view), float(lam), _ptr(idx), _ptr(count), cap, _ptr(out), _ptr(lse),
                        _ptr(smax))
    return out, lse, smax


def trigger(hi: HostInputs, r: int, lam: float, z_eff: float, top_j: int, a: np.ndarray, eta: np.ndarray,
            page_res: np.ndarray, idx: np.ndarray, count: np.ndarray, smax: np.ndarray, window: int,
            n_sink: int = 0, sketch=None):
    """(fired idx [B,H,N] int32, fired count [B,H]) of the row-level Cauchy-Schwarz trigger.

    ``sketch`` = (s16 [B,N,r_sk] bf16 bits, p [B,H,r_sk], rho [B,H]) adds the rank-r_sk content sketch term; eta
    must then be the sketch residual norms (``build_sketch``)."""
    a = np.ascontiguousarray(a, dtype=np.float64)
    idx = np.ascontiguousarray(idx, dtype=np.int32)
    count = np.ascontiguousarray(count, dtype=np.int32)
    smax = np.ascontiguousarray(smax, dtype=np.float64)
    eta = np.ascontiguousarray(eta, dtype=np.float64)
    page_res = np.ascontiguousarray(page_res, dtype=np.float64)
    capf = hi.N
    fidx = np.full((hi.B, hi.H, capf), -1, np.int32)
    fcount = np.zeros((hi.B, hi.H), np.int32)
    r_sk, s16, p, rho = 0, None, None, None
    if sketch is not None:
        s16 = np.ascontiguousarray(sketch[0], dtype=np.uint16)
        p = np.ascontiguousarray(sketch[1], dtype=np.float64)
        rho = np.ascontiguousarray(sketch[2], dtype=np.float64)
        r_sk = s16.shape[-1]
    lib().vko_trigger(ctypes.byref(hi.view), r, _ptr(hi.rot), float(lam), float(z_eff), int(top_j), _ptr(a),
                      _ptr(eta), _ptr(page_res), r_sk, _ptr(s16), _ptr(p), _ptr(rho), _ptr(idx), _ptr(count),
                      idx.shape[-1], _ptr(smax), window, n_sink, capf, _ptr(fidx), _ptr(fcount))
    return fidx, fcount


def page_norms(hi: HostInputs):
    """(page_knorm [B,P], page_eta [B,P]): per 64-row page the largest |K_u| (64 RoPE dims) and |L_u|."""
    P = (hi.N + PAGE - 1) // PAGE
    pk = np.zeros((hi.B, P), np.float64)
    pe = np.zeros((hi.B, P), np.float64)
    lib().vko_page_norms(ctypes.byref(hi.view), _ptr(pk), _ptr(pe))
    return pk, pe


def trigger_page(hi: HostInputs, lam: float, z_eff: float, top_j: int, page_knorm: np.ndarray,
                 page_eta: np.ndarray, idx: np.ndarray, count: np.ndarray, smax: np.ndarray, window: int,
                 n_sink: int = 0):
    """(fired idx [B,H,N] int32, fired count [B,H]) of the page-level trigger (reading B): archived rows outside
    S_h of every page whose bound lam (|qr| page_knorm + z_eff |qc| page_eta) beats s*_h."""
    idx = np.ascontiguousarray(idx, dtype=np.int32)
    count = np.ascontiguousarray(count, dtype=np.int32)
    smax = np.ascontiguousarray(smax, dtype=np.float64)
    pk = np.ascontiguousarray(page_knorm, dtype=np.float64)
    pe = np.ascontiguousarray(page_eta, dtype=np.float64)
    capf = hi.N
    fidx = np.full((hi.B, hi.H, capf), -1, np.int32)
    fcount = np.zeros((hi.B, hi.H), np.int32)
    lib().vko_trigger_page(ctypes.byref(hi.view), float(lam), float(z_eff), int(top_j), _ptr(pk), _ptr(pe),
                           _ptr(idx), _ptr(count), idx.shape[-1], _ptr(smax), window, n_sink, capf, _ptr(fidx),
                           _ptr(fcount))
    return fidx, fcount


def decode_step(hi: HostInputs, *, rho: float, r: int = 64, window: int = 0, n_sink: int = 0,
                sm_scale: float | None = None, trigger: int = 0, z_eff: float = 1.0, top_j: int = 0,
                digest_bf16: np.ndarray | None = None, cap: int | None = None, sketch_basis=None,
                sketch_bf16: np.ndarray | None = None):
    """Whole step (trigger: 0 off, 1 row-level reading A, 2 page-level reading B). ``sketch_basis`` [r_sk, 512]
    turns on the rank-r_sk content sketch of the row-level trigger (``sketch_bf16`` [B,N,r_sk]: the stored entries,
    else the bf16 rounding of the exact projection). Returns dict(out, lse, smax, idx, count, kth, rc)."""
    lam = (1.0 / math.sqrt(192.0)) if sm_scale is None else float(sm_scale)
    if cap is None:
        cap = hi.N if trigger else max(1, keep_count(hi.N, rho, window, n_sink) + window + n_sink)
    out = np.zeros((hi.B, hi.H, D_LATENT), np.float64)
    lse = np.zeros((hi.B, hi.H), np.float64)
    smax = np.zeros((hi.B, hi.H), np.float64)
    kth = np.zeros((hi.B, hi.H), np.float64)
    idx = np.full((hi.B, hi.H, cap), -1, np.int32)
    count = np.zeros((hi.B, hi.H), np.int32)
    dg = None if digest_bf16 is None else np.ascontiguousarray(digest_bf16, dtype=np.uint16)
    if r < D_ROPE and dg is None:
        raise ValueError("a width-r digest needs the stored bf16 digest")
    vb = None if sketch_basis is None else np.ascontiguousarray(sketch_basis, dtype=np.float64)
    r_sk = 0 if vb is None else vb.shape[0]
    s16 = None if sketch_bf16 is None else np.ascontiguousarray(sketch_bf16, dtype=np.uint16)
    rc = lib().vko_decode_step(ctypes.byref(hi.view), float(rho), r, window, n_sink, lam, int(trigger),
                               float(z_eff), int(top_j), _ptr(hi.rot), _ptr(dg), r_sk, _ptr(vb), _ptr(s16), cap,
                               _ptr(out), _ptr(lse), _ptr(smax), _ptr(idx), _ptr(count), _ptr(kth))
    return dict(out=out, lse=lse, smax=smax, idx=idx, count=count, kth=kth, rc=int(rc))


# ------------------------------------------------------------------------------------------------ sigma selector
def sigma(branch: np.ndarray, T: int = 4096, kappa: int = 16) -> np.ndarray:
    """Low-pass residual norms of the RoPE branch (Sec. 4.1, Eq. 3) over fixed blocks of T rows.

    ``branch`` is [N, 64] (any float dtype; used in fp64). Returns sigma [N] in fp64; rows past the last whole
    block (the open tail) get -1.
    """
    r = np.ascontiguousarray(np.asarray(branch, dtype=np.float64))
    assert r.ndim == 2 and r.shape[1] == D_ROPE
    out = np.empty(r.shape[0], dtype=np.float64)
    lib().vko_sigma(_ptr(r), r.shape[0], int(T), int(kappa), _ptr(out))
    return out


def sigma_select(sig: np.ndarray, T: int, n_sink: int, m: int) -> np.ndarray:
    """The sigma selector's attended set (Sec. 4.1): sinks, the open tail, and the top-m closed rows by sigma
    (ties: the smaller position). Returns the ascending ids."""
    s = np.ascontiguousarray(np.asarray(sig, dtype=np.float64))
    out = np.empty(max(1, s.shape[0]), dtype=np.int32)
    c = lib().vko_sigma_select(_ptr(s), s.shape[0], int(T), int(n_sink), int(m), _ptr(out))
    return out[:c].copy()



# ------------------------------------------------------------------------------------------------ PCA digest basis
def second_moment(hi: HostInputs) -> np.ndarray:
    """sum over every row of every sequence of K_u K_u^T, [64, 64] fp64."""
    M = np.zeros((D_ROPE, D_ROPE), np.float64)
    lib().vko_second_moment(ctypes.byref(hi.view), _ptr(M))
    return M


def sym_eig(M: np.ndarray):
    """(eigenvalues desc [64], eigenvectors as rows [64, 64]) of a symmetric 64x64 matrix by cyclic Jacobi."""
    A = np.ascontiguousarray(M, dtype=np.float64)
    eig = np.zeros(D_ROPE, np.float64)
    vec = np.zeros((D_ROPE, D_ROPE), np.float64)
    lib().vko_sym_eig(_ptr(A), _ptr(eig), _ptr(vec))
    return eig, vec


def pca_basis(hi: HostInputs):
    """(eigenvalues desc, rotation [64, 64] whose rows are the RoPE branch's principal directions)."""
    eig = np.zeros(D_ROPE, np.float64)
    rot = np.zeros((D_ROPE, D_ROPE), np.float64)
    lib().vko_pca_basis(ctypes.byref(hi.view), _ptr(eig), _ptr(rot))
    return eig, rot


# ------------------------------------------------------------------------------------------------ content sketch
def sketch_basis(q, r_sk: int):
    """(basis [r_sk, 512] whose rows are the leading eigenvectors of sum_i q_i q_i^T, eigenvalues [r_sk]) from
    queries q [n, 512] (Sec. 4.2: V_r from the context's own queries)."""
    qq = np.ascontiguousarray(np.asarray(q, dtype=np.float64).reshape(-1, D_LATENT))
    vb = np.zeros((r_sk, D_LATENT), np.float64)
    eig = np.zeros(r_sk, np.float64)
    rc = lib().vko_sketch_basis(_ptr(qq), qq.shape[0], int(r_sk), _ptr(vb), _ptr(eig))
    if rc != 0:
        raise ValueError(f"no rank-{r_sk} basis from {qq.shape[0]} queries")
    return vb, eig


def build_sketch(hi: HostInputs, vb):
    """(s fp64 [B,N,r_sk], s bf16 bits [B,N,r_sk], eta [B,N]): the sketch index entry of every cached row and its
    residual norm |L_u - V_r s_u|."""
    vb = np.ascontiguousarray(vb, dtype=np.float64)
    r_sk = vb.shape[0]
    s = np.zeros((hi.B, hi.N, r_sk), np.float64)
    s16 = np.zeros((hi.B, hi.N, r_sk), np.uint16)
    eta = np.zeros((hi.B, hi.N), np.float64)
    lib().vko_build_sketch(ctypes.byref(hi.view), r_sk, _ptr(vb), _ptr(s), _ptr(s16), _ptr(eta))
    return s, s16, eta


def sketch_query(hi: HostInputs, vb):
    """(p [B,H,r_sk], rho [B,H]): the queries' sketch coordinates and residual norms."""
    vb = np.ascontiguousarray(vb, dtype=np.float64)
    r_sk = vb.shape[0]
    p = np.zeros((hi.B, hi.H, max(r_sk, 1)), np.float64)
    rho = np.zeros((hi.B, hi.H), np.float64)
    lib().vko_sketch_query(ctypes.byref(hi.view), r_sk, _ptr(vb), _ptr(p), _ptr(rho))
    return p[..., :r_sk], rho


# ------------------------------------------------------------------------------------------------ conformal z
def tau_s(tau: float) -> float:
    return float(lib().vko_tau_s(float(tau)))


def min_hard(tau: float) -> int:
    return int(lib().vko_min_hard(float(tau)))


def conformal_quantile(zq, tau: float = 0.9, z_max: float = 8.0) -> float:
    """z from the hard queries' required inflations (the ceil((n+1) tau_s)-th smallest, clamped to [0, z_max])."""
    v = np.ascontiguousarray(np.asarray(zq, dtype=np.float64).ravel())
    return float(lib().vko_conformal_quantile(_ptr(v) if v.size else 0, v.size, float(tau), float(z_max)))


def calib_zq(hi: HostInputs, r: int, lam: float, a: np.ndarray, eta: np.ndarray, page_res: np.ndarray,
             idx: np.ndarray, count: np.ndarray, sketch=None):
    """(zq [B,H] with NaN where the query is not hard, ustar [B,H], n_hard) for every (b, h) as a calibration query.
    ``sketch`` = (s16, p, rho) as for ``trigger``: the sketch term and certificate (eta then the sketch residual)."""
    a = np.ascontiguousarray(a, dtype=np.float64)
    eta = np.ascontiguousarray(eta, dtype=np.float64)
    page_res = np.ascontiguousarray(page_res, dtype=np.float64)
    idx = np.ascontiguousarray(idx, dtype=np.int32)
    count = np.ascontiguousarray(count, dtype=np.int32)
    zq = np.zeros((hi.B, hi.H), np.float64)
    ustar = np.zeros((hi.B, hi.H), np.int32)
    r_sk, s16, p, rho = 0, None, None, None
    if sketch is not None:
        s16 = np.ascontiguousarray(sketch[0], dtype=np.uint16)
        p = np.ascontiguousarray(sketch[1], dtype=np.float64)
        rho = np.ascontiguousarray(sketch[2], dtype=np.float64)
        r_sk = s16.shape[-1]
    n = lib().vko_calib_zq(ctypes.byref(hi.view), int(r), _ptr(hi.rot), float(lam), _ptr(a), _ptr(eta), _ptr(page_res),
                           r_sk, _ptr(s16), _ptr(p), _ptr(rho), _ptr(idx), _ptr(count), idx.shape[-1], _ptr(zq),
                           _ptr(ustar))
    return zq, ustar, int(n)
