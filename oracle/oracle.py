"""Python wrapper (ctypes + numpy) around the plain-C CPU oracle.

TEST INFRASTRUCTURE ONLY: the test suite, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` are the only callers.  The CUDA product path
never imports this module.

``build()`` compiles ``qwm_oracle.c`` with gcc (``-O2 -ffp-contract=off``,
OpenMP over independent heads/rows) into ``oracle/_build/libqwm_oracle.so``.
All arrays are numpy; bf16 and fp16 values travel as their uint16 bit
patterns.  Every function states which part of the paper it follows in the C
source.
"""
from __future__ import annotations

import ctypes as ct
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "qwm_oracle.c")
_OUT_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_OUT_DIR, "libqwm_oracle.so")
_lib = None
_lock = threading.Lock()


def build(force: bool = False) -> str:
    """Compile the oracle shared library (idempotent) and return its path."""
    os.makedirs(_OUT_DIR, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fopenmp",
           "-fPIC", "-shared", "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def lib():
    global _lib
    with _lock:
        if _lib is None:
            _lib = ct.CDLL(build())
            _declare(_lib)
    return _lib


_p = ct.c_void_p


def _declare(L):
    L.oracle_bf16_to_f32.argtypes = [ct.c_uint16]
    L.oracle_bf16_to_f32.restype = ct.c_float
    L.oracle_f32_to_bf16.argtypes = [ct.c_float]
    L.oracle_f32_to_bf16.restype = ct.c_uint16
    L.oracle_f16_to_f32.argtypes = [ct.c_uint16]
    L.oracle_f16_to_f32.restype = ct.c_float
    L.oracle_f32_to_f16_ru.argtypes = [ct.c_float]
    L.oracle_f32_to_f16_ru.restype = ct.c_uint16
    L.oracle_fit_centroids.argtypes = [ct.c_int, ct.c_int, ct.c_int, ct.c_int, _p, ct.c_int64,
                                       _p, _p, _p, _p, ct.c_int]
    L.oracle_fit_centroids.restype = ct.c_int
    L.oracle_quantize.argtypes = ([ct.c_int] * 7 + [_p, ct.c_int64, _p, _p, _p, _p]
                                  + [_p] * 7 + [_p] * 7 + [ct.c_int] + [ct.c_int, _p, _p, _p])
    L.oracle_quantize.restype = ct.c_int
    L.oracle_dequant.argtypes = [ct.c_int] * 5 + [ct.c_int64] + [_p] * 11
    L.oracle_dequant.restype = ct.c_int
    L.oracle_attend.argtypes = [ct.c_int, ct.c_int, ct.c_int64, ct.c_int64, _p, _p, _p,
                                ct.c_double, _p, ct.c_int64, _p, _p, ct.c_int]
    L.oracle_attend.restype = ct.c_int
    L.oracle_max_threads.argtypes = []
    L.oracle_max_threads.restype = ct.c_int


def _ptr(a):
    return None if a is None else a.ctypes.data_as(_p)


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


def max_threads() -> int:
    return lib().oracle_max_threads()


# ---------------------------------------------------------------- formats
def bf16_to_f32(bits):
    b = _c(bits, np.uint16)
    return (b.astype(np.uint32) << 16).view(np.float32)


def f32_to_bf16(x):
    L = lib()
    x = np.asarray(x, dtype=np.float32)
    return np.array([L.oracle_f32_to_bf16(float(v)) for v in x.ravel()], dtype=np.uint16).reshape(x.shape)


def f16_to_f32(bits):
    L = lib()
    b = np.asarray(bits, dtype=np.uint16)
    return np.array([L.oracle_f16_to_f32(int(v)) for v in b.ravel()], dtype=np.float32).reshape(b.shape)


def f32_to_f16_ru(x):
    L = lib()
    x = np.asarray(x, dtype=np.float32)
    return np.array([L.oracle_f32_to_f16_ru(float(v)) for v in x.ravel()], dtype=np.uint16).reshape(x.shape)


# ---------------------------------------------------------------- k-means
def fit_centroids(x_bits, C: int, iters: int, nthreads: int = 0):
    """Lloyd k-means per head (see oracle_fit_centroids).

    x_bits: uint16 [N][H][d] (bf16 bits).  Returns dict with ``centroids``
    (uint16 [H][C][d] bf16 bits), ``cent_f32`` ([H][C][d]), ``assign``
    ([N][H] final assignment) and ``objective`` ([iters][H]).
    """
    x = _c(x_bits, np.uint16)
    N, H, d = x.shape
    out = np.zeros((H, C, d), np.uint16)
    cf = np.zeros((H, C, d), np.float32)
    asg = np.zeros((N, H), np.int32)
    obj = np.zeros((max(iters, 1), H), np.float64)
    rc = lib().oracle_fit_centroids(H, d, C, iters, _ptr(x), N, _ptr(out), _ptr(cf), _ptr(asg),
                                    _ptr(obj), nthreads)
    if rc:
        raise ValueError(f"oracle_fit_centroids: invalid arguments (rc={rc})")
    return {"centroids": out, "cent_f32": cf, "assign": asg, "objective": obj[:iters]}


# ---------------------------------------------------------------- append
def quantize(x_bits, cent_bits, *, G: int, r: int, M: int, is_key: bool,
             w=None, U_bits=None, force_ids=None, keep_scores: bool = False, nthreads: int = 0,
             two_level_scales: bool = False, M_full=None):
    """QSAC + INT2 + PSAC for one chunk (see oracle_quantize).

    x_bits uint16 [N][H][d]; cent_bits uint16 [H][C][d]; w float32 [H][d] or
    None; U_bits uint16 [H][d][r] or None.  Returns a dict of token-major
    arrays: ids, codes, scales, zeros, coef, sigma, kept, khat0, cand,
    m_topm, m_sel, m_psac and, with keep_scores, dq [N][H][C] and S [N][H][M'].
    two_level_scales: the App. D.1 storage of group scales (uint8 codes with
    one binary16 secondary scale per token-head, see two_level_scales in the
    C source); adds scode [N][H][d/G] and s2 [N][H] (binary16 bits), and the
    binary16 scales are left zero.
    M_full: float32 [H][d][d] or None; for Keys, the top-M candidates come from
    the full quadratic form (k - mu)^T M (k - mu) instead of Eq. 9 (the
    ablation of App. C.4); the QSAC score and everything after still use w.
    """
    x = _c(x_bits, np.uint16)
    cent = _c(cent_bits, np.uint16)
    N, H, d = x.shape
    C = cent.shape[1]
    assert cent.shape == (H, C, d)
    ng = d // G
    zb = (2 * ng + 7) // 8
    Mc = min(M, C)
    wv = None if w is None else _c(w, np.float32)
    Uv = None if U_bits is None else _c(U_bits, np.uint16)
    fid = None if force_ids is None else _c(force_ids, np.uint8)
    o = {
        "ids": np.zeros((N, H), np.uint8),
        "codes": np.zeros((N, H, d // 4), np.uint8),
        "scales": np.zeros((N, H, ng), np.uint16),
        "zeros": np.zeros((N, H, zb), np.uint8),
        "coef": np.zeros((N, H, max(r, 0)), np.int8),
        "sigma": np.zeros((N, H), np.uint16),
        "kept": np.zeros((N, H), np.uint8),
        "khat0": np.zeros((N, H, d), np.float32),
        "cand": np.zeros((N, H, Mc), np.int32),
        "m_topm": np.ones((N, H), np.float32),
        "m_sel": np.ones((N, H), np.float32),
        "m_psac": np.ones((N, H), np.float32),
        "dq": np.zeros((N, H, C), np.float32) if keep_scores else None,
        "S": np.zeros((N, H, Mc), np.float32) if keep_scores else None,
        "scode": np.zeros((N, H, ng), np.uint8) if two_level_scales else None,
        "s2": np.zeros((N, H), np.uint16) if two_level_scales else None,
    }
    if N == 0:
        return o
    rc = lib().oracle_quantize(
        H, d, C, G, r, M, int(bool(is_key)), _ptr(x), N, _ptr(cent), _ptr(wv), _ptr(Uv), _ptr(fid),
        _ptr(o["ids"]), _ptr(o["codes"]), _ptr(o["scales"]), _ptr(o["zeros"]), _ptr(o["coef"]),
        _ptr(o["sigma"]), _ptr(o["kept"]), _ptr(o["khat0"]), _ptr(o["cand"]), _ptr(o["m_topm"]),
        _ptr(o["m_sel"]), _ptr(o["m_psac"]), _ptr(o["dq"]), _ptr(o["S"]), nthreads,
        1 if two_level_scales else 0, _ptr(o["scode"]), _ptr(o["s2"]),
        _ptr(None if M_full is None else _c(M_full, np.float32)))
    if rc:
        raise ValueError(f"oracle_quantize: invalid arguments (rc={rc})")
    return o


def dequant(q, cent_bits, *, G: int, r: int, U_bits=None):
    """fp64 reconstruction [N][H][d] from packed arrays (see oracle_dequant)."""
    cent = _c(cent_bits, np.uint16)
    H, C, d = cent.shape
    ids = _c(q["ids"], np.uint8)
    N = ids.shape[0]
    out = np.zeros((N, H, d), np.float64)
    use_psac = U_bits is not None and r > 0
    coef = _c(q["coef"], np.int8) if use_psac else None
    sig = _c(q["sigma"], np.uint16) if use_psac else None
    Uv = _c(U_bits, np.uint16) if use_psac else None
    rc = lib().oracle_dequant(H, d, C, G, r if use_psac else 0, N, _ptr(cent), _ptr(ids),
                              _ptr(_c(q["codes"], np.uint8)), _ptr(_c(q["scales"], np.uint16)),
                              _ptr(_c(q["zeros"], np.uint8)), _ptr(coef), _ptr(sig), _ptr(Uv),
                              _ptr(out), _ptr(None if q.get("scode") is None else _c(q["scode"], np.uint8)),
                              _ptr(None if q.get("s2") is None else _c(q["s2"], np.uint16)))
    if rc:
        raise ValueError(f"oracle_dequant: invalid arguments (rc={rc})")
    return out


# ---------------------------------------------------------------- attend
def attend(q_bits, k, v, scale: float, rows=None, nthreads: int = 0):
    """Exact fp64 softmax attention (see oracle_attend).

    q_bits uint16 [Nq][H][d]; k, v float64 [Nk][H][d].  rows: optional int64
    list of query rows.  Returns (out [n][H][d] fp64, lse [H][n] fp64).
    """
    q = _c(q_bits, np.uint16)
    kk = _c(k, np.float64)
    vv = _c(v, np.float64)
    Nq, H, d = q.shape
    Nk = kk.shape[0]
    rr = None if rows is None else _c(rows, np.int64)
    n = Nq if rr is None else rr.shape[0]
    out = np.zeros((n, H, d), np.float64)
    lse = np.zeros((H, n), np.float64)
    rc = lib().oracle_attend(H, d, Nq, Nk, _ptr(q), _ptr(kk), _ptr(vv), float(scale), _ptr(rr),
                             n, _ptr(out), _ptr(lse), nthreads)
    if rc:
        raise ValueError(f"oracle_attend: invalid arguments (rc={rc})")
    return out, lse


# ---------------------------------------------------------------- query statistics
def query_stats(q_bits, r: int):
    """Historical Query statistics of one set of past queries (fp64, numpy).

    Sec. 4.1 Eq. 6: M_h = (1/N) sum_i q_i q_i^T per head;
    Sec. 4.1 Eq. 8: w_hc = M_cc / ((1/d) sum_c' M_c'c');
    Sec. 4.2 Eq. 15: M_h = U Lambda U^T with eigenvalues in decreasing order,
    U_r = the first r eigenvectors (numpy.linalg.eigh as the eigen solver).
    N = 0 (no Query yet) gives w = 1 and U = 0 (App. C.3 cold start).
    q_bits: uint16 [N][H][d].  Returns (M [H][d][d], w [H][d] fp32,
    U [H][d][r] fp64, eigenvalues [H][d] descending).
    """
    q = bf16_to_f32(q_bits).astype(np.float64)
    N, H, d = q.shape
    if N == 0:
        # No Query seen yet (App. C.3 cold start): uniform sensitivity and no
        # principal subspace, so w = 1 and U = 0.
        return (np.zeros((H, d, d)), np.ones((H, d), np.float32), np.zeros((H, d, r)), np.zeros((H, d)))
    M = np.einsum("nhc,nhe->hce", q, q) / N
    diag = np.einsum("hcc->hc", M)
    mean = diag.mean(axis=-1, keepdims=True)
    # Eq. 8 is 0/0 when every past Query of a head is zero; that head falls
    # back to the cold-start weights w = 1 (App. C.3).
    w = np.where(mean > 0, diag / np.where(mean > 0, mean, 1.0), 1.0).astype(np.float32)
    lam, vec = np.linalg.eigh(M)             # ascending
    lam = lam[:, ::-1]
    vec = vec[:, :, ::-1]
    return M, w, np.ascontiguousarray(vec[:, :, :r]), np.ascontiguousarray(lam)


# ---------------------------------------------------------------- token selection
def top1(q_bits, k):
    """Top-1 key of every query (Sec. 5, the top-1 token-selection shift
    table): the key with the largest logit q . k, the first on ties (fp64,
    numpy).  q_bits uint16 [Nq][H][d] (bf16 bits); k float64 [Nk][H][d].
    Returns (idx int64 [H][Nq], margin [H][Nq]: best minus second-best logit
    (inf with one key), scale [H][Nq]: |q| max_j |k_j|, which bounds every
    logit)."""
    q = bf16_to_f32(q_bits).astype(np.float64)
    k = np.asarray(k, np.float64)
    Nq, H, d = q.shape
    idx = np.zeros((H, Nq), np.int64)
    margin = np.full((H, Nq), np.inf)
    scale = np.zeros((H, Nq))
    for h in range(H):
        L = q[:, h] @ k[:, h].T                      # [Nq][Nk]
        idx[h] = np.argmax(L, axis=1)                # first maximum
        if L.shape[1] > 1:
            top2 = -np.partition(-L, 1, axis=1)[:, :2]
            margin[h] = top2[:, 0] - top2[:, 1]
        scale[h] = np.linalg.norm(q[:, h], axis=1) * np.linalg.norm(k[:, h], axis=1).max()
    return idx, margin, scale


def top1_shift(idx_ref, idx):
    """Share of (query, head) pairs whose top-1 key differs from the reference's."""
    return float(np.mean(np.asarray(idx_ref) != np.asarray(idx)))


# ---------------------------------------------------------------- storage accounting
def psac_tile_layout(kept, r: int, tile: int = 128):
    """The App. D.1 choice between dense and sparse PSAC coefficient layouts,
    made for each tile of `tile` tokens of a chunk-head (reading: the cache's
    storage unit; the paper leaves the granularity and the index format open).
    Dense stores every row's r INT8 codes and binary16 scale, n_t (r + 2)
    bytes; sparse stores a keep bit per token of the tile (a tile/8-byte mask,
    the index) and the kept rows only, tile/8 + K_t (r + 2) bytes, in token
    order; the strictly smaller one is chosen.  kept: bool/uint8 [N].
    Returns (sparse [ntiles] bool, bytes [ntiles] of the chosen layout)."""
    kept = np.asarray(kept).astype(bool)
    N = kept.size
    nt = (N + tile - 1) // tile
    sparse = np.zeros(nt, bool)
    nbytes = np.zeros(nt, np.int64)
    for t in range(nt):
        k = kept[t * tile:(t + 1) * tile]
        dense_b = k.size * (r + 2)
        sparse_b = tile // 8 + int(k.sum()) * (r + 2)
        sparse[t] = sparse_b < dense_b
        nbytes[t] = min(dense_b, sparse_b)
    return sparse, nbytes


def psac_layout_bytes(kept, r: int, N: int | None = None):
    """Bytes of one chunk-head's PSAC coefficients in the two layouts App. D.1
    chooses between (reading: dense = every row's r INT8 codes and binary16
    scale; sparse = the kept rows only, each with a uint16 token index, plus a
    4-byte row count).  kept: bool/uint8 [N].  Returns (dense, sparse, chosen)."""
    kept = np.asarray(kept).astype(bool)
    n = kept.size if N is None else N
    K = int(kept.sum())
    dense = n * (r + 2)
    sparse = K * (r + 2 + 2) + 4
    return dense, sparse, min(dense, sparse)
