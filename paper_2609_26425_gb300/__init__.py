"""GB300-native QuantWM per-chunk 2-bit KV-cache path.

Thin Python binding (ctypes) over the C ABI of ``libqwm.so`` (see
include/qwm.h).  Every step of the path runs in the library's CUDA kernels;
this module only marshals arguments: it checks tensor dtypes, shapes and
devices, passes raw device pointers and the current CUDA stream, and uses
PyTorch for device memory.  There is no fallback: if the library is not
built, every call raises.

Functions carry the C names:
  qwm_cache_bytes, qwm_fit_workspace_bytes, qwm_fit_centroids,
  qwm_fit_centroids_noalloc, qwm_quantize_append, qwm_attend,
``Cache`` wraps qwm_cache_init / qwm_cache_free / qwm_cache_status /
qwm_cache_layout / qwm_cache_chunk_info, ``QueryStats`` wraps a Query
statistics buffer (qwm_query_stats_bytes / _reset / _update / _read and
qwm_query_basis), and qwm_dequant_chunk / qwm_top1_keys serve the
token-selection shift measurement.
"""
from __future__ import annotations

import ctypes as ct
import math
import os
import threading

import numpy as np
import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_build", "libqwm.so")

QWM_OK = 0
QWM_ROLE_V_REBUILD = 1
STATUS_NAMES = {0: "QWM_OK", 1: "QWM_ERR_INVALID_ARG", 2: "QWM_ERR_UNSUPPORTED", 3: "QWM_ERR_CAPACITY",
                4: "QWM_ERR_CUDA", 5: "QWM_ERR_TIMEOUT", 6: "QWM_ERR_NONFINITE"}


class QwmError(RuntimeError):
    def __init__(self, fn, status):
        self.status = status
        super().__init__(f"{fn} failed: {STATUS_NAMES.get(status, status)}")


class QwmConfig(ct.Structure):
    _fields_ = [("num_heads", ct.c_int32), ("head_dim", ct.c_int32), ("num_centroids", ct.c_int32),
                ("group_size", ct.c_int32), ("psac_rank", ct.c_int32), ("num_candidates", ct.c_int32),
                ("kmeans_iters", ct.c_int32), ("scale_format", ct.c_int32)]

    def __repr__(self):
        return ("QwmConfig(H=%d, d=%d, C=%d, G=%d, r=%d, M=%d, iters=%d, scale_format=%d)" %
                (self.num_heads, self.head_dim, self.num_centroids, self.group_size, self.psac_rank,
                 self.num_candidates, self.kmeans_iters, self.scale_format))


def config(heads, centroids, group_size=32, psac_rank=16, candidates=4, kmeans_iters=10, head_dim=128,
           scale_format=0):
    return QwmConfig(heads, head_dim, centroids, group_size, psac_rank, candidates, kmeans_iters, scale_format)


class QwmLayout(ct.Structure):
    _fields_ = [(n, ct.c_int64) for n in (
        "header_bytes", "slot_meta_bytes", "slot_bytes", "head_bytes",
        "ktab_offset", "vtab_offset", "ut_offset", "tiles_offset",
        "tile_tokens", "tiles_per_chunk", "tile_bytes",
        "k_codes", "k_scales", "k_ids", "k_zeros", "k_coef", "k_sigma", "k_bytes",
        "v_codes", "v_scales", "v_ids", "v_zeros", "v_bytes", "zero_bytes", "k_s2", "v_s2", "pmask_offset")]


_lib = None
_lock = threading.Lock()
_P = ct.c_void_p
_CFG = ct.POINTER(QwmConfig)


def lib():
    """Load libqwm.so (raises if it has not been built)."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(LIB_PATH):
                raise RuntimeError(f"{LIB_PATH} is missing: build it with "
                                   "`python -c 'import __graft_entry__ as g; g.build()'`")
            L = ct.CDLL(LIB_PATH)
            L.qwm_status_string.argtypes = [ct.c_int]
            L.qwm_status_string.restype = ct.c_char_p
            L.qwm_cache_bytes.argtypes = [_CFG, ct.c_int64, ct.c_int32]
            L.qwm_cache_bytes.restype = ct.c_size_t
            L.qwm_cache_init.argtypes = [ct.POINTER(_P), _CFG, _P, ct.c_size_t, ct.c_int64, ct.c_int32,
                                         ct.c_int32, _P]
            L.qwm_cache_init.restype = ct.c_int
            L.qwm_cache_free.argtypes = [_P]
            L.qwm_cache_free.restype = None
            L.qwm_cache_num_chunks.argtypes = [_P]
            L.qwm_cache_num_chunks.restype = ct.c_int32
            L.qwm_cache_chunk_info.argtypes = [_P, ct.c_int32, ct.POINTER(ct.c_int32), ct.POINTER(ct.c_int64)]
            L.qwm_cache_chunk_info.restype = ct.c_int
            L.qwm_cache_layout.argtypes = [_P, ct.POINTER(QwmLayout)]
            L.qwm_cache_layout.restype = ct.c_int
            L.qwm_cache_status.argtypes = [_P, ct.POINTER(ct.c_int32), _P]
            L.qwm_cache_status.restype = ct.c_int
            L.qwm_fit_workspace_bytes.argtypes = [_CFG, ct.c_int64]
            L.qwm_fit_workspace_bytes.restype = ct.c_size_t
            L.qwm_fit_centroids.argtypes = [_CFG, _P, ct.c_int64, _P, _P, ct.c_size_t, _P]
            L.qwm_fit_centroids.restype = ct.c_int
            L.qwm_quantize_append.argtypes = [_CFG, _P, _P, _P, ct.c_int64, _P, _P, _P, _P, _P]
            L.qwm_quantize_append.restype = ct.c_int
            L.qwm_attend.argtypes = [_CFG, _P, _P, ct.c_int64, _P, _P, ct.c_int64, ct.c_float, _P, _P, _P]
            L.qwm_attend.restype = ct.c_int
            L.qwm_attend_workspace_bytes.argtypes = [_CFG, _P, ct.c_int64, ct.c_int64]
            L.qwm_attend_workspace_bytes.restype = ct.c_size_t
            L.qwm_attend_ws.argtypes = [_CFG, _P, _P, ct.c_int64, _P, _P, ct.c_int64, ct.c_float, _P, _P, _P,
                                        ct.c_size_t, _P]
            L.qwm_attend_ws.restype = ct.c_int
            L.qwm_query_stats_bytes.argtypes = [_CFG]
            L.qwm_query_stats_bytes.restype = ct.c_size_t
            L.qwm_query_stats_reset.argtypes = [_CFG, _P, _P]
            L.qwm_query_stats_reset.restype = ct.c_int
            L.qwm_query_stats_update.argtypes = [_CFG, _P, _P, ct.c_int64, _P]
            L.qwm_query_stats_update.restype = ct.c_int
            L.qwm_query_basis.argtypes = [_CFG, _P, _P, _P, _P, _P]
            L.qwm_query_basis.restype = ct.c_int
            L.qwm_query_stats_read.argtypes = [_P, ct.POINTER(ct.c_int32), ct.POINTER(ct.c_int64), _P]
            L.qwm_query_stats_read.restype = ct.c_int
            L.qwm_dequant_chunk.argtypes = [_CFG, _P, ct.c_int32, _P, _P, _P]
            L.qwm_dequant_chunk.restype = ct.c_int
            L.qwm_top1_keys.argtypes = [_CFG, _P, ct.c_int64, _P, ct.c_int64, _P, _P]
            L.qwm_top1_keys.restype = ct.c_int
            L.qwm_quantize_append_full.argtypes = [_CFG, _P, _P, _P, ct.c_int64, _P, _P, _P, _P, _P, _P]
            L.qwm_quantize_append_full.restype = ct.c_int
            L.qwm_cache_set_wait_limit.argtypes = [_P, ct.c_uint64]
            L.qwm_cache_set_wait_limit.restype = ct.c_int
            L.qwm_cache_set_idle_role.argtypes = [_P, ct.c_int32]
            L.qwm_cache_set_idle_role.restype = ct.c_int
            _lib = L
    return _lib


def _check(fn, st):
    if st != QWM_OK:
        raise QwmError(fn, st)


def _stream():
    return ct.c_void_p(torch.cuda.current_stream().cuda_stream)


def _ptr(t):
    return None if t is None else ct.c_void_p(t.data_ptr())


def _bf16(t, shape, name):
    if not (isinstance(t, torch.Tensor) and t.is_cuda and t.dtype == torch.bfloat16 and t.is_contiguous()):
        raise ValueError(f"{name} must be a contiguous bf16 CUDA tensor")
    if tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} has shape {tuple(t.shape)}, expected {tuple(shape)}")
    return t


# ------------------------------------------------------------------ sizes
def qwm_cache_bytes(cfg: QwmConfig, tokens_per_chunk: int, max_chunks: int) -> int:
    return int(lib().qwm_cache_bytes(ct.byref(cfg), tokens_per_chunk, max_chunks))


def qwm_fit_workspace_bytes(cfg: QwmConfig, N: int) -> int:
    return int(lib().qwm_fit_workspace_bytes(ct.byref(cfg), N))


# ------------------------------------------------------------------ cache
class Cache:
    """A packed KV cache in a torch-allocated device buffer (qwm_cache_init)."""

    def __init__(self, cfg: QwmConfig, tokens_per_chunk: int, max_chunks: int, sliding_window: bool = False,
                 device=None):
        self.cfg = cfg
        self.tokens_per_chunk = tokens_per_chunk
        self.max_chunks = max_chunks
        nbytes = qwm_cache_bytes(cfg, tokens_per_chunk, max_chunks)
        if nbytes == 0:
            raise QwmError("qwm_cache_bytes", 2)
        dev = torch.device(device) if device is not None else torch.device("cuda", torch.cuda.current_device())
        self._raw = torch.empty(nbytes + 1024, dtype=torch.uint8, device=dev)
        off = (-self._raw.data_ptr()) % 1024
        self.buffer = self._raw[off:off + nbytes]
        self.nbytes = nbytes
        h = ct.c_void_p()
        _check("qwm_cache_init", lib().qwm_cache_init(ct.byref(h), ct.byref(cfg), _ptr(self.buffer), nbytes,
                                                      tokens_per_chunk, max_chunks, int(bool(sliding_window)),
                                                      _stream()))
        self.handle = h

    def __del__(self):
        h = getattr(self, "handle", None)
        if h and _lib is not None:
            _lib.qwm_cache_free(h)
            self.handle = None

    @property
    def num_chunks(self) -> int:
        return int(lib().qwm_cache_num_chunks(self.handle))

    def chunk_info(self, i: int):
        s, t = ct.c_int32(), ct.c_int64()
        _check("qwm_cache_chunk_info", lib().qwm_cache_chunk_info(self.handle, i, ct.byref(s), ct.byref(t)))
        return s.value, t.value

    def layout(self) -> QwmLayout:
        lay = QwmLayout()
        _check("qwm_cache_layout", lib().qwm_cache_layout(self.handle, ct.byref(lay)))
        return lay

    def set_wait_limit(self, ns: int):
        """qwm_cache_set_wait_limit: limit of the kernels' bounded waits (ns)."""
        _check("qwm_cache_set_wait_limit", lib().qwm_cache_set_wait_limit(self.handle, int(ns)))

    def set_idle_role(self, role: int):
        """qwm_cache_set_idle_role: test hook of the timeout path (0 = normal work)."""
        _check("qwm_cache_set_idle_role", lib().qwm_cache_set_idle_role(self.handle, int(role)))

    def status(self) -> int:
        v = ct.c_int32()
        _check("qwm_cache_status", lib().qwm_cache_status(self.handle, ct.byref(v), _stream()))
        return v.value

    def decode_chunk(self, i: int) -> dict:
        """Copy chunk i (0 = oldest held) back to the host as token-major numpy
        arrays (layout only; no arithmetic): ids [N][H], codes [N][H][d/4],
        scales [N][H][d/G] (binary16 bits), zeros [N][H][zb], coef [N][H][r],
        sigma [N][H] (binary16 bits), k_tab / v_tab [H][C][d] (binary16 bits,
        the tables as stored in the slot) and U [H][d][r] (bf16 bits).  With
        scale_format 1, scode [N][H][d/G] u8 and s2 [N][H] (binary16 bits)
        replace scales (and v_scode, v_s2 for Values).  PSAC rows are read
        through each tile's keep mask (row i is entry popcount(mask below i);
        rows the mask leaves out hold zeros) and returned per token; pmask
        [H][tiles][4] u32 holds the masks as stored."""
        slot, N = self.chunk_info(i)
        lay = self.layout()
        cfg = self.cfg
        H, d, C, G, r = cfg.num_heads, cfg.head_dim, cfg.num_centroids, cfg.group_size, cfg.psac_rank
        ng, zb = d // G, lay.zero_bytes
        start = lay.header_bytes + slot * lay.slot_bytes
        raw = self.buffer[start:start + lay.slot_bytes].cpu().numpy()
        T = lay.tile_tokens
        ntile = (N + T - 1) // T
        sf = cfg.scale_format
        keys = ("ids", "codes", "zeros", "coef", "sigma", "v_ids", "v_codes", "v_zeros")
        keys += ("scode", "s2", "v_scode", "v_s2") if sf else ("scales", "v_scales")
        out = {k: [] for k in keys}
        k_tab = np.zeros((H, C, d), np.uint16)
        v_tab = np.zeros((H, C, d), np.uint16)
        U = np.zeros((H, d, r), np.uint16)
        pmask = np.zeros((H, ntile, 4), np.uint32)
        for h in range(H):
            hb = lay.slot_meta_bytes + h * lay.head_bytes
            k_tab[h] = raw[hb + lay.ktab_offset: hb + lay.ktab_offset + C * d * 2].view(np.uint16).reshape(C, d)
            v_tab[h] = raw[hb + lay.vtab_offset: hb + lay.vtab_offset + C * d * 2].view(np.uint16).reshape(C, d)
            if r:
                U[h] = raw[hb + lay.ut_offset: hb + lay.ut_offset + r * d * 2].view(np.uint16).reshape(r, d).T
            tiles = raw[hb + lay.tiles_offset: hb + lay.tiles_offset + ntile * lay.tile_bytes].reshape(
                ntile, lay.tile_bytes)

            def f(off, width, dtype=np.uint8):
                b = tiles[:, off: off + T * width].reshape(ntile * T, width)[:N]
                return np.ascontiguousarray(b).view(dtype)

            out["codes"].append(f(lay.k_codes, d // 4))
            if sf:
                out["scode"].append(f(lay.k_scales, ng))
                out["s2"].append(f(lay.k_s2, 2, np.uint16)[:, 0])
                out["v_scode"].append(f(lay.v_scales, ng))
                out["v_s2"].append(f(lay.v_s2, 2, np.uint16)[:, 0])
            else:
                out["scales"].append(f(lay.k_scales, ng * 2, np.uint16))
                out["v_scales"].append(f(lay.v_scales, ng * 2, np.uint16))
            out["ids"].append(f(lay.k_ids, 1)[:, 0])
            out["zeros"].append(f(lay.k_zeros, zb))
            if r:
                pm = raw[hb + lay.pmask_offset: hb + lay.pmask_offset + ntile * 16].view(np.uint32).reshape(ntile, 4)
                pmask[h] = pm
                bitsel = ((pm[:, np.arange(T) // 32] >> (np.arange(T) % 32).astype(np.uint32)) & 1).astype(bool)
                entry = np.cumsum(bitsel, axis=1) - 1
                ct = np.ascontiguousarray(tiles[:, lay.k_coef: lay.k_coef + T * r]).view(np.int8).reshape(ntile, T, r)
                st = np.ascontiguousarray(tiles[:, lay.k_sigma: lay.k_sigma + T * 2]).view(np.uint16).reshape(ntile, T)
                tix = np.arange(ntile)[:, None]
                e = np.where(bitsel, entry, 0)
                cf = np.where(bitsel[..., None], ct[tix, e], 0).astype(np.int8).reshape(ntile * T, r)[:N]
                sg = np.where(bitsel, st[tix, e], 0).astype(np.uint16).reshape(ntile * T)[:N]
                out["coef"].append(cf)
                out["sigma"].append(sg)
            else:
                out["coef"].append(np.zeros((N, 0), np.int8))
                out["sigma"].append(np.zeros(N, np.uint16))
            out["v_codes"].append(f(lay.v_codes, d // 4))
            out["v_ids"].append(f(lay.v_ids, 1)[:, 0])
            out["v_zeros"].append(f(lay.v_zeros, zb))
        res = {k: np.stack(v, axis=1) for k, v in out.items()}
        res.update(k_tab=k_tab, v_tab=v_tab, U=U, tokens=N, slot=slot, pmask=pmask)
        return res


# ------------------------------------------------------------------ compute
def qwm_fit_centroids(cfg: QwmConfig, x: torch.Tensor, centroids=None, workspace=None) -> torch.Tensor:
    N = x.shape[0]
    H, d, C = cfg.num_heads, cfg.head_dim, cfg.num_centroids
    _bf16(x, (N, H, d), "x")
    if centroids is None:
        centroids = torch.empty(H, C, d, dtype=torch.bfloat16, device=x.device)
    _bf16(centroids, (H, C, d), "centroids")
    need = qwm_fit_workspace_bytes(cfg, N)
    if workspace is None:
        workspace = torch.empty(need, dtype=torch.uint8, device=x.device)
    _check("qwm_fit_centroids", lib().qwm_fit_centroids(ct.byref(cfg), _ptr(x), N, _ptr(centroids),
                                                        _ptr(workspace), workspace.numel(), _stream()))
    return centroids


def qwm_fit_centroids_noalloc(cfg: QwmConfig, x: torch.Tensor, centroids=None) -> torch.Tensor:
    """qwm_fit_centroids without a caller-provided workspace: the library keeps
    the scratch in a static device array (see include/qwm.h for the limit and
    the rule that overlapping calls race)."""
    N = x.shape[0]
    H, d, C = cfg.num_heads, cfg.head_dim, cfg.num_centroids
    _bf16(x, (N, H, d), "x")
    if centroids is None:
        centroids = torch.empty(H, C, d, dtype=torch.bfloat16, device=x.device)
    _bf16(centroids, (H, C, d), "centroids")
    fn = lib().qwm_fit_centroids_noalloc
    fn.argtypes = [_CFG, _P, ct.c_int64, _P, _P]
    fn.restype = ct.c_int
    _check("qwm_fit_centroids_noalloc", fn(ct.byref(cfg), _ptr(x), N, _ptr(centroids), _stream()))
    return centroids


def qwm_quantize_append(cfg: QwmConfig, cache: Cache, k, v, k_centroids, v_centroids, w=None, U=None):
    N = k.shape[0]
    H, d, C, r = cfg.num_heads, cfg.head_dim, cfg.num_centroids, cfg.psac_rank
    _bf16(k, (N, H, d), "k")
    _bf16(v, (N, H, d), "v")
    _bf16(k_centroids, (H, C, d), "k_centroids")
    _bf16(v_centroids, (H, C, d), "v_centroids")
    if w is not None:
        if not (w.is_cuda and w.dtype == torch.float32 and w.is_contiguous() and tuple(w.shape) == (H, d)):
            raise ValueError("w must be a contiguous fp32 CUDA tensor [H][d]")
    if U is not None:
        _bf16(U, (H, d, r), "U")
    _check("qwm_quantize_append", lib().qwm_quantize_append(
        ct.byref(cfg), cache.handle, _ptr(k), _ptr(v), N, _ptr(k_centroids), _ptr(v_centroids), _ptr(w),
        _ptr(U), _stream()))


def qwm_quantize_append_full(cfg: QwmConfig, cache: Cache, k, v, k_centroids, v_centroids, Mq, w=None, U=None):
    """qwm_quantize_append with the Keys' candidates by the full quadratic form
    (Mq: fp32 CUDA tensor [H][d][d])."""
    N = k.shape[0]
    H, d, C, r = cfg.num_heads, cfg.head_dim, cfg.num_centroids, cfg.psac_rank
    _bf16(k, (N, H, d), "k")
    _bf16(v, (N, H, d), "v")
    _bf16(k_centroids, (H, C, d), "k_centroids")
    _bf16(v_centroids, (H, C, d), "v_centroids")
    if not (Mq.is_cuda and Mq.dtype == torch.float32 and Mq.is_contiguous() and tuple(Mq.shape) == (H, d, d)):
        raise ValueError("Mq must be a contiguous fp32 CUDA tensor [H][d][d]")
    if w is not None:
        if not (w.is_cuda and w.dtype == torch.float32 and w.is_contiguous() and tuple(w.shape) == (H, d)):
            raise ValueError("w must be a contiguous fp32 CUDA tensor [H][d]")
    if U is not None:
        _bf16(U, (H, d, r), "U")
    _check("qwm_quantize_append_full", lib().qwm_quantize_append_full(
        ct.byref(cfg), cache.handle, _ptr(k), _ptr(v), N, _ptr(k_centroids), _ptr(v_centroids), _ptr(w),
        _ptr(U), _ptr(Mq), _stream()))


def qwm_attend_workspace_bytes(cfg: QwmConfig, cache: Cache, Nq: int, Ncur: int = 0) -> int:
    """Bytes of the scratch buffer qwm_attend can use to balance a launch (0: none needed)."""
    return int(lib().qwm_attend_workspace_bytes(ct.byref(cfg), cache.handle, int(Nq), int(Ncur)))


def attend_workspace(cfg: QwmConfig, cache: Cache, Nq: int, Ncur: int = 0, device=None):
    """A torch-allocated scratch buffer for qwm_attend(..., workspace=), or None when none is needed."""
    n = qwm_attend_workspace_bytes(cfg, cache, Nq, Ncur)
    if n == 0:
        return None
    dev = torch.device(device) if device is not None else torch.device("cuda", torch.cuda.current_device())
    raw = torch.empty(n + 256, dtype=torch.uint8, device=dev)
    off = (-raw.data_ptr()) % 256
    return raw[off:off + n]


def qwm_attend(cfg: QwmConfig, cache: Cache, q, k_cur=None, v_cur=None, sm_scale=None, out=None,
               lse=None, want_lse=False, workspace=None):
    Nq = q.shape[0]
    H, d = cfg.num_heads, cfg.head_dim
    _bf16(q, (Nq, H, d), "q")
    Ncur = 0 if k_cur is None else k_cur.shape[0]
    if Ncur:
        _bf16(k_cur, (Ncur, H, d), "k_cur")
        _bf16(v_cur, (Ncur, H, d), "v_cur")
    if out is None:
        out = torch.empty(Nq, H, d, dtype=torch.bfloat16, device=q.device)
    _bf16(out, (Nq, H, d), "out")
    if want_lse and lse is None:
        lse = torch.empty(H, Nq, dtype=torch.float32, device=q.device)
    scale = 1.0 / math.sqrt(d) if sm_scale is None else float(sm_scale)
    if workspace is None:
        _check("qwm_attend", lib().qwm_attend(ct.byref(cfg), cache.handle, _ptr(q), Nq,
                                              _ptr(k_cur) if Ncur else None, _ptr(v_cur) if Ncur else None, Ncur,
                                              scale, _ptr(out), _ptr(lse), _stream()))
    else:
        _check("qwm_attend_ws", lib().qwm_attend_ws(ct.byref(cfg), cache.handle, _ptr(q), Nq,
                                                    _ptr(k_cur) if Ncur else None, _ptr(v_cur) if Ncur else None,
                                                    Ncur, scale, _ptr(out), _ptr(lse), _ptr(workspace),
                                                    workspace.numel() * workspace.element_size(), _stream()))
    return (out, lse) if (want_lse or lse is not None) else out


# ------------------------------------------------------------------ Query statistics
class QueryStats:
    """Running per-head Query statistics in a torch-allocated device buffer
    (qwm_query_stats_bytes bytes: a 256-byte header, then fp32 sums [H][d][d])."""

    HEADER = 256

    def __init__(self, cfg: QwmConfig, device=None):
        self.cfg = cfg
        nbytes = int(lib().qwm_query_stats_bytes(ct.byref(cfg)))
        if nbytes == 0:
            raise QwmError("qwm_query_stats_bytes", 2)
        dev = torch.device(device) if device is not None else torch.device("cuda", torch.cuda.current_device())
        self._raw = torch.empty(nbytes + 256, dtype=torch.uint8, device=dev)
        off = (-self._raw.data_ptr()) % 256
        self.buffer = self._raw[off:off + nbytes]
        self.nbytes = nbytes
        self.reset()

    def reset(self):
        _check("qwm_query_stats_reset", lib().qwm_query_stats_reset(ct.byref(self.cfg), _ptr(self.buffer),
                                                                    _stream()))

    @property
    def sums(self) -> torch.Tensor:
        """View of the fp32 sums S_h = sum q q^T, [H][d][d] (no copy)."""
        H, d = self.cfg.num_heads, self.cfg.head_dim
        return self.buffer[self.HEADER:].view(torch.float32).view(H, d, d)

    def update(self, q):
        """qwm_query_stats_update: fold one chunk's Queries q [N][H][d] (bf16) in."""
        N = q.shape[0]
        _bf16(q, (N, self.cfg.num_heads, self.cfg.head_dim), "q")
        _check("qwm_query_stats_update", lib().qwm_query_stats_update(ct.byref(self.cfg), _ptr(self.buffer),
                                                                      _ptr(q) if N else None, N, _stream()))

    def basis(self, w=True, U=True, eigenvalues=False):
        """qwm_query_basis: returns (w [H][d] fp32, U [H][d][r] bf16, eigenvalues
        [H][d] fp32), each None when not requested (U also when r = 0)."""
        H, d, r = self.cfg.num_heads, self.cfg.head_dim, self.cfg.psac_rank
        dev = self.buffer.device
        tw = torch.empty(H, d, dtype=torch.float32, device=dev) if w else None
        tU = torch.empty(H, d, r, dtype=torch.bfloat16, device=dev) if (U and r > 0) else None
        te = torch.empty(H, d, dtype=torch.float32, device=dev) if eigenvalues else None
        _check("qwm_query_basis", lib().qwm_query_basis(ct.byref(self.cfg), _ptr(self.buffer), _ptr(tw),
                                                        _ptr(tU), _ptr(te), _stream()))
        return tw, tU, te

    def read(self):
        """(status, count): synchronises the stream and clears the status word."""
        st, cnt = ct.c_int32(), ct.c_int64()
        _check("qwm_query_stats_read", lib().qwm_query_stats_read(_ptr(self.buffer), ct.byref(st), ct.byref(cnt),
                                                                  _stream()))
        return st.value, cnt.value

    def sweeps(self) -> int:
        """Jacobi sweeps of the last basis computation (maximum over heads)."""
        return int(self.buffer[16:20].view(torch.int32).item())


# ------------------------------------------------------------------ token-selection shift
def qwm_dequant_chunk(cfg: QwmConfig, cache: Cache, i: int, keys=True, values=False):
    """fp32 reconstruction of cached chunk i: (k_hat, v_hat), each [N][H][d] or None."""
    _, N = cache.chunk_info(i)
    H, d = cfg.num_heads, cfg.head_dim
    dev = cache.buffer.device
    k = torch.empty(N, H, d, dtype=torch.float32, device=dev) if keys else None
    v = torch.empty(N, H, d, dtype=torch.float32, device=dev) if values else None
    _check("qwm_dequant_chunk", lib().qwm_dequant_chunk(ct.byref(cfg), cache.handle, i, _ptr(k), _ptr(v),
                                                        _stream()))
    return k, v


def qwm_top1_keys(cfg: QwmConfig, q, keys, idx=None):
    """Index of the highest-logit key for every query and head, int32 [H][Nq]."""
    Nq, Nk = q.shape[0], keys.shape[0]
    H, d = cfg.num_heads, cfg.head_dim
    _bf16(q, (Nq, H, d), "q")
    if not (keys.is_cuda and keys.dtype == torch.float32 and keys.is_contiguous() and tuple(keys.shape) == (Nk, H, d)):
        raise ValueError("keys must be a contiguous fp32 CUDA tensor [Nk][H][d]")
    if idx is None:
        idx = torch.empty(H, Nq, dtype=torch.int32, device=q.device)
    _check("qwm_top1_keys", lib().qwm_top1_keys(ct.byref(cfg), _ptr(q), Nq, _ptr(keys), Nk, _ptr(idx), _stream()))
    return idx
