"""GPU: values beyond the binary16 range.

The cache and the attention tensor cores hold binary16 operands (binary16
group scales and centroid tables, App. D.1's FP16 storage; f16 MMAs with fp32
accumulation).  A bf16 input of magnitude above 65504, or one that is not a
number, cannot be represented there.  The library reports it in the device
status word as QWM_ERR_NONFINITE and keeps its outputs finite; inputs inside
the range are unaffected (every other GPU test checks that the status stays
QWM_OK).  Finite values beyond the range saturate to +-65504, so outputs stay
finite; a NaN input is reported and propagates.  Nothing here faults a GPU: the values are ordinary bf16 numbers.
"""
import math

import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2609_26425_gb300 import synth
import paper_2609_26425_gb300 as qwm

from parity import compare_attention, compare_packed, oracle_append, oracle_kv, strided_centroids

pytestmark = pytest.mark.gpu
NONFINITE = 6


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    qwm.lib()


def dev(t):
    return t.to("cuda").contiguous()


def chunk(seed, N, H):
    q = synth.gaussian_bf16(seed * 3 + 1, N, H, 128)
    k = synth.gaussian_bf16(seed * 3 + 2, N, H, 128)
    v = synth.gaussian_bf16(seed * 3 + 3, N, H, 128)
    return q, k, v


def small_cache(H=2, N=300, C=16, G=32, r=16, M=4, seed=3):
    q, k, v = chunk(seed, N, H)
    kb, vb = synth.bits(k), synth.bits(v)
    kc, vc = strided_centroids(kb, C), strided_centroids(vb, C)
    Ub = synth.bits(synth.random_orthonormal(seed + 9, H, 128, r))
    cfg = qwm.config(H, C, group_size=G, psac_rank=r, candidates=M)
    cache = qwm.Cache(cfg, N, 1)
    qwm.qwm_quantize_append(cfg, cache, dev(k), dev(v), dev(synth.from_bits(kc)), dev(synth.from_bits(vc)),
                            U=dev(synth.from_bits(Ub)))
    assert cache.status() == 0
    ko, vo = oracle_append(kb, vb, kc, vc, G=G, r=r, M=M, U_bits=Ub)
    K, V = oracle_kv(ko, vo, kc, vc, G=G, r=r, U_bits=Ub)
    return cfg, cache, q, K, V


def test_attend_query_beyond_binary16_is_reported_and_output_stays_finite():
    """A query value of 7e4 (above 65504) sets QWM_ERR_NONFINITE; the output
    stays finite; the next call with ordinary queries is exact again."""
    cfg, cache, q, K, V = small_cache()
    qbad = q.clone()
    qbad[7, 1, 3] = 7.0e4
    out = qwm.qwm_attend(cfg, cache, dev(qbad))
    torch.cuda.synchronize()
    assert cache.status() == NONFINITE
    assert torch.isfinite(out.float()).all()
    out = qwm.qwm_attend(cfg, cache, dev(q))
    assert cache.status() == 0       # the status word was cleared by the read before
    ref, _ = orc.attend(synth.bits(q), K, V, 1 / math.sqrt(128))
    compare_attention(out.float().cpu().numpy(), ref)


@pytest.mark.parametrize("which", ["k", "v", "nan"])
def test_attend_active_chunk_beyond_binary16_is_reported(which):
    """Active-chunk Keys or Values of 1e5 set QWM_ERR_NONFINITE and the output
    stays finite (they saturate to +-65504); a NaN is reported the same way
    (it reaches the output of its head)."""
    cfg, cache, q, K, V = small_cache(seed=4)
    _, kcur, vcur = chunk(11, 200, 2)
    if which == "k":
        kcur[5, 0, 17] = 1.0e5
    elif which == "v":
        vcur[150, 1, 99] = -1.0e5
    else:
        kcur[9, 1, 2] = float("nan")
    out = qwm.qwm_attend(cfg, cache, dev(q), dev(kcur), dev(vcur))
    torch.cuda.synchronize()
    assert cache.status() == NONFINITE
    if which != "nan":
        assert torch.isfinite(out.float()).all()


def test_append_keys_beyond_binary16_take_exact_rescoring():
    """Keys with single channels at +-9e4 (beyond binary16, so their rows
    cannot enter the f16 candidate filter) fall back to the exact rescoring of
    every centroid: the packed records still equal the oracle's bit for bit,
    and the append reports QWM_ERR_NONFINITE (attention cannot hold them)."""
    H, N, C, G, r, M = 2, 300, 64, 32, 16, 4
    _, k, v = chunk(21, N, H)
    k = k.float()
    g = torch.Generator().manual_seed(5)
    rows = torch.randperm(N, generator=g)[:12]
    for i, t in enumerate(rows.tolist()):
        k[t, i % H, (7 * i) % 128] = 9.0e4 if i % 2 else -9.0e4
    k = k.to(torch.bfloat16)
    kb, vb = synth.bits(k), synth.bits(v)
    kc, vc = strided_centroids(kb, C), strided_centroids(vb, C)
    w = synth.random_weights(31, H, 128).numpy()
    Ub = synth.bits(synth.random_orthonormal(32, H, 128, r))
    cfg = qwm.config(H, C, group_size=G, psac_rank=r, candidates=M)
    cache = qwm.Cache(cfg, N, 1)
    qwm.qwm_quantize_append(cfg, cache, dev(k), dev(v), dev(synth.from_bits(kc)), dev(synth.from_bits(vc)),
                            w=torch.from_numpy(w).cuda(), U=dev(synth.from_bits(Ub)))
    torch.cuda.synchronize()
    assert cache.status() == NONFINITE
    dec = cache.decode_chunk(0)
    ko, vo = oracle_append(kb, vb, kc, vc, G=G, r=r, M=M, w=w, U_bits=Ub)
    compare_packed(dec, ko, kb, kc, G=G, r=r, M=M, is_key=True, w=w, U_bits=Ub)
    compare_packed(dec, vo, vb, vc, G=G, r=r, M=M, is_key=False, prefix="v_")
    # the large channels really are beyond binary16 (and their groups' scales are finite)
    assert np.abs(orc.bf16_to_f32(kb)).max() > 65504
    assert np.isfinite(dec["scales"].view(np.float16).astype(np.float32)).all()


def test_append_table_beyond_binary16_is_reported():
    """A centroid value beyond binary16 cannot be stored in the slot's
    binary16 table: QWM_ERR_NONFINITE."""
    H, N, C = 2, 200, 16
    _, k, v = chunk(41, N, H)
    kb, vb = synth.bits(k), synth.bits(v)
    kc, vc = strided_centroids(kb, C), strided_centroids(vb, C)
    vct = synth.from_bits(vc).clone()
    vct[1, 3, 64] = 2.0e5
    cfg = qwm.config(H, C, psac_rank=0)
    cache = qwm.Cache(cfg, N, 1)
    qwm.qwm_quantize_append(cfg, cache, dev(k), dev(v), dev(synth.from_bits(kc)), dev(vct))
    torch.cuda.synchronize()
    assert cache.status() == NONFINITE
