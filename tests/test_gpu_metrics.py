"""GPU parity of the token-selection shift measurement: the reconstruction
of a cached chunk (qwm_dequant_chunk) and the top-1 key of each query
(qwm_top1_keys) against the oracle's dequant and top1.

Reconstruction: fp32 against the oracle's fp64 of its own packing, within
2^-20 of |mu| + 3 s + |U t sigma| per entry.  Top-1 keys: equal wherever the
oracle's best logit leads the second by more than 2e-5 |q| max|k| (the fp32
channel-order sum's rounding bound, with margin); elsewhere the GPU's pick is
within that bound of the best logit.
"""
import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2609_26425_gb300 import synth
import paper_2609_26425_gb300 as qwm

pytestmark = pytest.mark.gpu

MARGIN = 2e-5


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    qwm.lib()


def check_top1(idx_gpu, q_bits, keys64):
    idx, margin, scale = orc.top1(q_bits, keys64)
    decided = margin > MARGIN * scale
    assert np.array_equal(idx_gpu[decided], idx[decided]), f"{int((idx_gpu != idx)[decided].sum())} decided mismatches"
    # undecided rows: the GPU's key is within the bound of the best logit
    qf = orc.bf16_to_f32(q_bits).astype(np.float64)
    for h, n in zip(*np.nonzero(~decided)):
        lg = qf[n, h] @ keys64[idx_gpu[h, n], h]
        lb = qf[n, h] @ keys64[idx[h, n], h]
        assert lg >= lb - MARGIN * scale[h, n]
    return idx


@pytest.mark.parametrize("Nq,Nk,H", [(1, 1, 1), (70, 300, 2), (130, 1000, 3), (64, 4097, 1)])
def test_top1_keys_parity(Nq, Nk, H):
    q = synth.gaussian_bf16(31 + Nq, Nq, H, 128)
    k = torch.randn(Nk, H, 128, generator=torch.Generator().manual_seed(Nk)).float()
    k[Nk // 2] = k[Nk // 3]          # duplicated keys: the lower index must win on equal logits
    cfg = qwm.config(H, 16)
    idx = qwm.qwm_top1_keys(cfg, q.cuda(), k.cuda()).cpu().numpy()
    check_top1(idx, synth.bits(q), k.double().numpy())


def test_dequant_and_shift_ratio_single_layer():
    """The single-layer workload's two cached chunks appended three ways — QVG
    (w = 1, nearest centroid, no PSAC), QSAC (w, top-M) and QSAC + PSAC — then
    the share of the new chunk's queries whose top-1 cached key moves away from
    the bf16 keys' top-1, on the GPU and in the oracle."""
    wl = synth.WORKLOADS["single_layer_h4"]
    H, N, C, G, r = wl.heads, wl.chunk_tokens, wl.centroids, wl.group_size, wl.psac_rank
    src = synth.ChunkSource(wl)
    q_new, _, _ = src.chunk(wl.past_chunks)
    q_bits = synth.bits(q_new)
    past = [src.chunk(t) for t in range(wl.past_chunks)]
    w = synth.population_w(src.log_scale0)
    U = synth.population_U(src.log_scale0, r)
    k_ref = np.concatenate([orc.bf16_to_f32(synth.bits(k)).astype(np.float64) for _, k, _ in past])
    idx_ref_gpu = qwm.qwm_top1_keys(qwm.config(H, C), q_new.cuda(), torch.from_numpy(k_ref).float().cuda())
    idx_ref = check_top1(idx_ref_gpu.cpu().numpy(), q_bits, k_ref)
    ratios = {}
    for name, M, use_w, use_U in (("qvg", 1, False, False), ("qsac", 4, True, False), ("qsac_psac", 4, True, True)):
        rr = r if use_U else 0
        cfg = qwm.config(H, C, group_size=G, psac_rank=rr, candidates=M)
        cache = qwm.Cache(cfg, N, wl.past_chunks)
        k_hat_oracle, k_hat_gpu = [], []
        for t, (_, k, v) in enumerate(past):
            kb = synth.bits(k)
            kc = orc.fit_centroids(kb, C, 4)["centroids"]
            vc = orc.fit_centroids(synth.bits(v), C, 4)["centroids"]
            wv = w.numpy() if use_w else None
            Ub = synth.bits(U) if use_U else None
            qwm.qwm_quantize_append(cfg, cache, k.cuda(), v.cuda(), synth.from_bits(kc).cuda(),
                                    synth.from_bits(vc).cuda(), w=w.cuda() if use_w else None,
                                    U=U.cuda() if use_U else None)
            ko = orc.quantize(kb, kc, G=G, r=rr, M=M, is_key=True, w=wv, U_bits=Ub)
            k_hat_oracle.append(orc.dequant(ko, kc, G=G, r=rr, U_bits=Ub))
            kg, _ = qwm.qwm_dequant_chunk(cfg, cache, t)
            kg = kg.cpu().double().numpy()
            same = (cache.decode_chunk(t)["ids"] == ko["ids"])
            err = np.abs(kg - k_hat_oracle[-1])[same]
            scale = np.abs(k_hat_oracle[-1])[same] + 1.0
            assert np.all(err <= 2.0 ** -18 * scale), f"{name}: reconstruction error {err.max():.3e}"
            k_hat_gpu.append(kg)
        torch.cuda.synchronize()
        assert cache.status() == 0
        kh_o = np.concatenate(k_hat_oracle)
        idx_gpu = qwm.qwm_top1_keys(cfg, q_new.cuda(), torch.from_numpy(np.concatenate(k_hat_gpu)).float().cuda())
        idx_o = check_top1(idx_gpu.cpu().numpy(), q_bits, kh_o)
        ratio_gpu = orc.top1_shift(idx_ref_gpu.cpu().numpy(), idx_gpu.cpu().numpy())
        ratio_o = orc.top1_shift(idx_ref, idx_o)
        assert abs(ratio_gpu - ratio_o) <= 0.01, (name, ratio_gpu, ratio_o)
        ratios[name] = ratio_gpu
    print("top-1 shift ratios:", ratios)
