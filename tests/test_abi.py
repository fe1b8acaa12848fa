"""Host-only checks of the C ABI: the library builds, loads without a GPU,
exports every function include/qwm.h declares, and sizes the packed cache as
the paper's packed storage (App. D.1) implies."""
import ctypes as ct
import os
import re

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def qlib():
    from paper_2609_26425_gb300 import build
    build.build()
    import paper_2609_26425_gb300 as qwm
    return qwm


def declared_functions():
    src = open(os.path.join(ROOT, "include", "qwm.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(qwm_[a-z0-9_]+)\s*\(", src)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for n in ("qwm_fit_centroids", "qwm_quantize_append", "qwm_attend", "qwm_cache_bytes"):
        assert n in names


def test_library_exports_every_declared_symbol(qlib):
    L = ct.CDLL(qlib.LIB_PATH)
    missing = [n for n in declared_functions() if not hasattr(L, n)]
    assert not missing, missing


def test_cache_bytes_matches_packed_format(qlib):
    """Per token-head: d/4 code bytes, d/G binary16 scales, 1 id byte, the zero-point
    byte; Keys add r INT8 codes + a binary16 row scale; per chunk-head two
    binary16 centroid tables, U_r^T and a 16-byte PSAC keep mask per tile.
    Tiles hold 128 tokens."""
    for (H, C, G, r, T, n) in [(40, 256, 32, 16, 4680, 6), (4, 64, 32, 16, 880, 3), (12, 64, 64, 8, 880, 15),
                               (2, 16, 32, 0, 100, 1)]:
        cfg = qlib.config(H, C, group_size=G, psac_rank=r)
        b = qlib.qwm_cache_bytes(cfg, T, n)
        d, ng = 128, 128 // G
        k_tok = d // 4 + 2 * ng + 1 + 1 + (r + 2 if r else 0)
        v_tok = d // 4 + 2 * ng + 1 + 1
        tiles = -(-T // 128)
        per_head = 2 * C * d * 2 + r * d * 2 + (16 * tiles if r else 0)   # + a PSAC keep mask per tile
        per_head = -(-per_head // 1024) * 1024 + tiles * 128 * (k_tok + v_tok)
        per_head = -(-per_head // 1024) * 1024
        assert b == 256 + n * (256 + H * per_head)


def test_compression_ratio_of_wan14b_layer(qlib):
    """The packed format against bf16 K+V for the Wan-14B-shaped layer (H=40,
    C=256, G=32, r=16, 6 chunks of 4680 tokens): per token-head 60 + 42 bytes
    vs 512 (5.02x); with the per-chunk tables ~3.9x (the paper's 6.20x
    assumes G=64, r=8, INT8 scale codes and amortised tables)."""
    cfg = qlib.config(40, 256, group_size=32, psac_rank=16)
    b = qlib.qwm_cache_bytes(cfg, 4680, 6)
    bf16 = 2 * 6 * 4680 * 40 * 128 * 2
    ratio = bf16 / b
    assert 3.7 < ratio < 4.0
    assert 512 / (60 + 42) == pytest.approx(5.02, abs=0.01)


def test_unsupported_shapes_size_to_zero(qlib):
    assert qlib.qwm_cache_bytes(qlib.config(4, 64, group_size=16), 100, 2) == 0
    assert qlib.qwm_cache_bytes(qlib.config(4, 300), 100, 2) == 0
    assert qlib.qwm_cache_bytes(qlib.config(4, 64, psac_rank=12), 100, 2) == 0
    assert qlib.qwm_cache_bytes(qlib.config(4, 64), 100, 257) == 0
    assert qlib.qwm_fit_workspace_bytes(qlib.config(4, 64), 0) == 0
    # centroids H*C*d*4, operand images H*P*512 (P = C rounded to 16), assignment and lists H*N*5
    assert qlib.qwm_fit_workspace_bytes(qlib.config(4, 64), 10) >= 4 * 64 * 128 * 4 + 4 * 64 * 512 + 4 * 10 * 5
    assert qlib.qwm_fit_workspace_bytes(qlib.config(4, 64), 20000) >= 4 * 64 * 128 * 4 + 4 * 64 * 512 + 4 * 20000 * 5


def test_query_statistics_and_measurement_host_errors(qlib):
    """Argument errors of the Query-statistics and measurement entry points come
    back before anything touches a device (these calls never reach CUDA)."""
    L = qlib.lib()
    cfg = qlib.config(4, 64, psac_rank=16)
    bad = qlib.config(4, 64, psac_rank=12)
    fake = ct.c_void_p(1 << 20)            # 256-byte aligned, never dereferenced
    unaligned = ct.c_void_p((1 << 20) + 8)
    assert L.qwm_query_stats_bytes(ct.byref(cfg)) == 256 + 4 * 128 * 128 * 4
    assert L.qwm_query_stats_bytes(ct.byref(bad)) == 0
    assert L.qwm_query_stats_update(ct.byref(bad), fake, fake, 10, None) == 2
    assert L.qwm_query_stats_update(ct.byref(cfg), None, fake, 10, None) == 1
    assert L.qwm_query_stats_update(ct.byref(cfg), unaligned, fake, 10, None) == 1
    assert L.qwm_query_stats_update(ct.byref(cfg), fake, fake, -1, None) == 1
    assert L.qwm_query_stats_update(ct.byref(cfg), fake, None, 0, None) == 0     # N = 0: nothing to do
    assert L.qwm_query_stats_update(ct.byref(cfg), fake, None, 5, None) == 1
    assert L.qwm_query_basis(ct.byref(cfg), fake, None, None, None, None) == 0   # nothing requested
    assert L.qwm_query_basis(ct.byref(bad), fake, None, None, None, None) == 2
    assert L.qwm_query_basis(ct.byref(cfg), fake, ct.c_void_p((1 << 20) + 2), None, None, None) == 1
    assert L.qwm_query_stats_read(None, None, None, None) == 1
    assert L.qwm_top1_keys(ct.byref(cfg), fake, 0, fake, 10, fake, None) == 1
    assert L.qwm_top1_keys(ct.byref(cfg), fake, 10, fake, 0, fake, None) == 1
    assert L.qwm_top1_keys(ct.byref(bad), fake, 10, fake, 10, fake, None) == 2
    assert L.qwm_top1_keys(ct.byref(cfg), fake, 10, ct.c_void_p((1 << 20) + 4), 10, fake, None) == 1
    assert L.qwm_dequant_chunk(ct.byref(cfg), None, 0, fake, None, None) == 1


def test_cache_bytes_two_level_scales(qlib):
    """Scale format 1 (App. D.1): per token-head d/G uint8 scale codes and one
    binary16 secondary scale replace the d/G binary16 scales, for Keys and
    Values alike (58 + 40 bytes instead of 60 + 42 at G = 32, r = 16)."""
    for (H, C, G, r, T, n) in [(40, 256, 32, 16, 4680, 6), (4, 64, 64, 8, 880, 3), (2, 16, 32, 0, 100, 1)]:
        cfg = qlib.config(H, C, group_size=G, psac_rank=r, scale_format=1)
        b = qlib.qwm_cache_bytes(cfg, T, n)
        d, ng = 128, 128 // G
        k_tok = d // 4 + ng + 2 + 1 + 1 + (r + 2 if r else 0)
        v_tok = d // 4 + ng + 2 + 1 + 1
        tiles = -(-T // 128)
        per_head = 2 * C * d * 2 + r * d * 2 + (16 * tiles if r else 0)
        per_head = -(-per_head // 1024) * 1024 + tiles * 128 * (k_tok + v_tok)
        per_head = -(-per_head // 1024) * 1024
        assert b == 256 + n * (256 + H * per_head)
    assert qlib.qwm_cache_bytes(qlib.config(4, 64, scale_format=2), 100, 2) == 0


def test_fit_entry_points_accept_the_same_configurations(qlib):
    """The allocation-free k-means entry point rejects exactly what the
    workspace entry point rejects (an unsupported scale format, rank or
    group size) before anything reaches CUDA."""
    L = qlib.lib()
    fn = L.qwm_fit_centroids_noalloc
    fn.argtypes = [ct.c_void_p, ct.c_void_p, ct.c_int64, ct.c_void_p, ct.c_void_p]
    fn.restype = ct.c_int
    fake = ct.c_void_p(1 << 20)
    for bad in (qlib.config(4, 64, scale_format=2), qlib.config(4, 64, psac_rank=12),
                qlib.config(4, 64, group_size=16), qlib.config(4, 300)):
        assert L.qwm_fit_centroids(ct.byref(bad), fake, 10, fake, fake, 1 << 30, None) == 2
        assert fn(ct.byref(bad), fake, 10, fake, None) == 2
    assert fn(ct.byref(qlib.config(4, 64)), fake, 0, fake, None) == 1


def test_wait_limit_and_idle_role_argument_checks(qlib):
    """The timeout-path settings reject a missing cache and values out of range
    without touching a device."""
    L = qlib.lib()
    assert L.qwm_cache_set_wait_limit(None, 1_000_000) == 1
    assert L.qwm_cache_set_idle_role(None, 0) == 1
