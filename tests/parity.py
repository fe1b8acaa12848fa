"""Shared helpers for the GPU-vs-oracle parity tests (test infrastructure).

The comparison rules for the packed output:
  * centroid ids, INT2 codes, zero-points and binary16 group scales must be
    bit-exact;
  * an id may differ only where the oracle's own decision margin is below
    1e-5 (relative gap between the M-th and (M+1)-th Query-aware distance, or
    between the best and second-best QSAC score); such tokens are requantised
    by the oracle with the GPU's id and must then match bit-exactly;
  * PSAC INT8 codes and binary16 row scales must be bit-exact except where
    the oracle's PSAC margin (rounding boundaries, keep test) is below 1e-5.
Attention: bf16 output against the oracle's fp64 result, max-abs <= 2e-2 and
mean-abs <= 2e-3.
"""
from __future__ import annotations

import numpy as np

from oracle import oracle as orc

ID_MARGIN = 1e-5
PSAC_MARGIN = 1e-5
ATT_MAX_ABS = 2e-2
ATT_MEAN_ABS = 2e-3


def oracle_append(k_bits, v_bits, kc_bits, vc_bits, *, G, r, M, w=None, U_bits=None, nthreads=0,
                  two_level=False):
    """Oracle packed Keys and Values of one chunk (token-major dicts)."""
    ko = orc.quantize(k_bits, kc_bits, G=G, r=r, M=M, is_key=True, w=w, U_bits=U_bits, nthreads=nthreads,
                      two_level_scales=two_level)
    vo = orc.quantize(v_bits, vc_bits, G=G, r=r, M=M, is_key=False, nthreads=nthreads, two_level_scales=two_level)
    return ko, vo


def compare_packed(gpu: dict, ref: dict, x_bits, cent_bits, *, G, r, M, is_key, w=None, U_bits=None,
                   prefix="", two_level=False):
    """Assert bit-exact parity of one side (Keys: prefix '', Values: prefix 'v_').
    two_level: the slot stores uint8 group codes and a binary16 secondary scale
    (scale format 1) instead of binary16 group scales."""
    g_ids = gpu[prefix + "ids"]
    diff = g_ids != ref["ids"]
    stats = {"tokens": int(g_ids.size), "id_flips": int(diff.sum())}
    if diff.any():
        margin = np.minimum(ref["m_topm"], ref["m_sel"])
        bad = diff & (margin >= ID_MARGIN)
        assert not bad.any(), f"{int(bad.sum())} id mismatches with oracle margin >= {ID_MARGIN}"
        ref = orc.quantize(x_bits, cent_bits, G=G, r=r, M=M, is_key=is_key, w=w, U_bits=U_bits,
                           force_ids=g_ids, two_level_scales=two_level)
    for key in ("codes", "zeros") + (("scode", "s2") if two_level else ("scales",)):
        a, b = gpu[prefix + key], ref[key]
        assert a.shape == b.shape, (key, a.shape, b.shape)
        nbad = int((a != b).sum())
        assert nbad == 0, f"{prefix}{key}: {nbad} mismatching entries"
    if is_key and r > 0:
        row_bad = (gpu["coef"] != ref["coef"]).any(-1) | (gpu["sigma"] != ref["sigma"])
        stats["psac_flips"] = int(row_bad.sum())
        if row_bad.any():
            assert np.all(ref["m_psac"][row_bad] < PSAC_MARGIN), \
                f"{int((row_bad & (ref['m_psac'] >= PSAC_MARGIN)).sum())} PSAC rows differ beyond the margin"
    return stats


def compare_attention(out_gpu: np.ndarray, ref: np.ndarray):
    err = np.abs(out_gpu.astype(np.float64) - ref)
    mx, mean = float(err.max()), float(err.mean())
    assert mx <= ATT_MAX_ABS, f"attention max-abs error {mx:.3e} > {ATT_MAX_ABS}"
    assert mean <= ATT_MEAN_ABS, f"attention mean-abs error {mean:.3e} > {ATT_MEAN_ABS}"
    return mx, mean


def oracle_kv(ko: dict, vo: dict, kc_bits, vc_bits, *, G, r, U_bits=None):
    """fp64 K_hat, V_hat of one chunk from the ORACLE's own packed arrays
    (Keys with the PSAC term when U is given, Values without)."""
    K = orc.dequant(ko, kc_bits, G=G, r=r, U_bits=U_bits if r > 0 else None)
    V = orc.dequant(vo, vc_bits, G=G, r=0)
    return K, V


def strided_centroids(x_bits, C):
    """Generator-side centroid table: tokens floor(j*N/C) of the chunk (no arithmetic)."""
    N = x_bits.shape[0]
    idx = (np.arange(C) * N) // C
    return np.ascontiguousarray(x_bits[idx].transpose(1, 0, 2))
