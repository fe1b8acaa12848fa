"""GPU parity at the workloads' full sizes, in the launch configuration bench.py times.

The oracle cannot quantize and attend a whole Wan-14B-shaped layer in seconds, so these
tests run the full-size GPU path and check sampled outputs that the oracle computes one
by one:
  * the packed records of sampled tokens of every appended chunk, all heads, bit-exact
    under the margin rule of ``parity.compare_packed``;
  * attention rows of sampled queries on sampled heads, against the oracle's fp64
    softmax over its own reconstruction of every cached key of those heads plus the
    active bf16 chunk (max-abs 2e-2, mean-abs 2e-3), and the log-sum-exp.
Inputs are the workloads' seeded generators (``synth.ChunkSource``: LogNormal query
channel scales with AR(1) drift, outlier Key channels, population w and U_r); the
centroid tables are the generator's strided tokens (k-means with zero iterations), so no
oracle input comes from the GPU.  The token and row samples always include the first and
last rows of the 128-row tiles at both ends and the ragged tail.
"""
import math

import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2609_26425_gb300 import synth
import paper_2609_26425_gb300 as qwm

from parity import compare_attention, compare_packed, oracle_append, oracle_kv

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    qwm.lib()


def dev(t):
    return t.to("cuda").contiguous()


def strided_centroids(x_bits, C):
    """Tokens floor(j*N/C) of the chunk as the table (k-means initial centroids, no arithmetic)."""
    N = x_bits.shape[0]
    idx = (np.arange(C) * N) // C
    return np.ascontiguousarray(x_bits[idx].transpose(1, 0, 2))


def sample_rows(N, n, seed):
    """Sorted sample of [0, N): tile edges at both ends, the ragged tail, n random rows."""
    edge = [0, 1, 63, 64, 127, 128, 129, 255, 256]
    last = (N - 1) // 128 * 128
    edge += [last - 1, last, last + 1, N - 2, N - 1]
    rng = np.random.default_rng(seed)
    s = set(i for i in edge if 0 <= i < N) | set(rng.integers(0, N, size=n).tolist())
    return np.array(sorted(s), dtype=np.int64)


def subset(dec, idx):
    keys = ("ids", "codes", "scales", "zeros", "coef", "sigma", "v_ids", "v_codes", "v_scales", "v_zeros")
    return {k: dec[k][idx] for k in keys}


class Held:
    """Host copy of one appended chunk, restricted to the attention-check heads."""

    def __init__(self, kb, vb, kc, vc, w, Ub, heads):
        self.kb, self.vb = kb[:, heads], vb[:, heads]
        self.kc, self.vc = kc[heads], vc[heads]
        self.w = None if w is None else w[heads]
        self.Ub = None if Ub is None else Ub[heads]


def check_chunk(cfg, cache, kb, vb, kc, vc, w, Ub, *, G, r, M, n_tok, seed):
    """Sampled tokens of the newest chunk, all heads, against the oracle."""
    dec = cache.decode_chunk(cache.num_chunks - 1)
    N = kb.shape[0]
    assert dec["tokens"] == N
    idx = sample_rows(N, n_tok, seed)
    ko, vo = oracle_append(kb[idx], vb[idx], kc, vc, G=G, r=r, M=M, w=w, U_bits=Ub)
    g = subset(dec, idx)
    compare_packed(g, ko, kb[idx], kc, G=G, r=r, M=M, is_key=True, w=w, U_bits=Ub)
    compare_packed(g, vo, vb[idx], vc, G=G, r=r, M=M, is_key=False, prefix="v_")
    assert np.array_equal(dec["k_tab"], synth.from_bits(kc).to(torch.float16).view(torch.int16).numpy().view(np.uint16))


def run_workload(wl, *, layer=0, appended=None, r=None, n_tok=96, heads=(0, 1), n_rows=48):
    H, N, C, G, M = wl.heads, wl.chunk_tokens, wl.centroids, wl.group_size, wl.candidates
    r = wl.psac_rank if r is None else r
    slots = wl.window if wl.window else wl.past_chunks
    appended = wl.past_chunks if appended is None else appended
    heads = list(heads)
    cfg = qwm.config(H, C, group_size=G, psac_rank=r, candidates=M)
    src = synth.ChunkSource(wl, layer=layer)
    hist = qwm.Cache(cfg, N, slots, sliding_window=bool(wl.window))
    held = []
    for t in range(appended):
        _, k, v = src.chunk(t)
        a = src.query_log_scale(t)
        w = synth.population_w(a).numpy() if t > 0 else None
        Ub = synth.bits(synth.population_U(a, r)) if (t > 0 and r > 0) else None
        kb, vb = synth.bits(k), synth.bits(v)
        kc, vc = strided_centroids(kb, C), strided_centroids(vb, C)
        qwm.qwm_quantize_append(cfg, hist, dev(k), dev(v), dev(synth.from_bits(kc)), dev(synth.from_bits(vc)),
                                w=None if w is None else torch.from_numpy(w).cuda(),
                                U=None if Ub is None else dev(synth.from_bits(Ub)))
        torch.cuda.synchronize()
        assert hist.status() == 0
        check_chunk(cfg, hist, kb, vb, kc, vc, w, Ub, G=G, r=r, M=M, n_tok=n_tok, seed=1000 * layer + t)
        held.append(Held(kb, vb, kc, vc, w, Ub, heads))
        held = held[-slots:]
    assert hist.num_chunks == min(appended, slots)

    # the new chunk: its queries attend the cache plus its own bf16 K/V (the active chunk)
    q, k, v = src.chunk(appended)
    # in the launch configuration the bench times: the work units of the
    # last wave split along the key chunks (qwm_attend_ws)
    ws = qwm.attend_workspace(cfg, hist, q.shape[0], k.shape[0])
    out, lse = qwm.qwm_attend(cfg, hist, dev(q), dev(k), dev(v), want_lse=True, workspace=ws)
    torch.cuda.synchronize()
    assert hist.status() == 0
    Ks, Vs = [], []
    for hc in held:
        ko, vo = oracle_append(hc.kb, hc.vb, hc.kc, hc.vc, G=G, r=r, M=M, w=hc.w, U_bits=hc.Ub)
        K, V = oracle_kv(ko, vo, hc.kc, hc.vc, G=G, r=r, U_bits=hc.Ub)
        Ks.append(K)
        Vs.append(V)
    Ks.append(orc.bf16_to_f32(synth.bits(k)[:, heads]).astype(np.float64))
    Vs.append(orc.bf16_to_f32(synth.bits(v)[:, heads]).astype(np.float64))
    rows = sample_rows(q.shape[0], n_rows, 77 + layer)
    ref, ref_lse = orc.attend(synth.bits(q)[:, heads], np.concatenate(Ks, 0), np.concatenate(Vs, 0),
                              1 / math.sqrt(128), rows=rows)
    got = out.float().cpu().numpy()[rows][:, heads]
    compare_attention(got, ref)
    got_lse = lse.cpu().numpy()[heads][:, rows]
    assert np.abs(got_lse - ref_lse).max() < 2e-2


def test_wan14b_layer_full_size():
    """40 heads, C = 256, G = 32, r = 16; 6 cached chunks of 4680 tokens and the
    4680-token active chunk attended by its 4680 queries: the step bench.py times."""
    run_workload(synth.WORKLOADS["wan14b_layer"], heads=(0, 23, 39))


def test_wan14b_stack_longest_cache():
    """The long-horizon stack's largest per-layer step: 8 cached chunks (37440 tokens)
    of the last layer's seeds."""
    wl = synth.WORKLOADS["wan14b_stack"]
    run_workload(wl, layer=wl.layers - 1, n_tok=48, heads=(5, 31))


@pytest.mark.parametrize("r", [8, 32])
def test_dit1p3b_sliding_window(r):
    """12 heads, 1-frame chunks of 880 tokens with Student-t(3) outlier Keys, C = 64,
    a 15-chunk sliding window wrapped twice (17 appends), PSAC rank 8 and 32."""
    wl = synth.WORKLOADS["dit1p3b_window"]
    run_workload(wl, layer=7, appended=17, r=r, n_tok=64, heads=(0, 11))


@pytest.mark.parametrize("H,chunks,C,G,r,Nq,Ncur", [
    (40, [65536, 65536], 16, 64, 32, 1024, 1000),   # 64k appended per chunk, 128k cached keys
    (40, [65536], 256, 32, 8, 4096, 0),             # the largest table at the largest append
    (40, [16384, 4096], 64, 64, 0, 4000, 4096),     # PSAC off, G = 64, ragged query count
])
def test_microbench_sweep_extremes(H, chunks, C, G, r, Nq, Ncur):
    """End points of the one-layer sweep (appended tokens up to 64k, cache up to 128k
    tokens, C in {16, 64, 256}, r in {0, 8, 32}, G in {32, 64}); Gaussian inputs with
    8x outlier Key channels, random w and orthonormal U_r."""
    heads = [0, H - 1]
    cfg = qwm.config(H, C, group_size=G, psac_rank=r, candidates=4)
    cache = qwm.Cache(cfg, max(chunks), len(chunks))
    Ks, Vs = [], []
    for ci, N in enumerate(chunks):
        seed = 9000 + 10 * ci + C
        k = synth.gaussian_bf16(seed + 1, N, H, 128).float()
        k[:, :, [3, 50, 91, 126]] *= 8
        k = k.to(torch.bfloat16)
        v = synth.gaussian_bf16(seed + 2, N, H, 128)
        kb, vb = synth.bits(k), synth.bits(v)
        kc, vc = strided_centroids(kb, C), strided_centroids(vb, C)
        w = synth.random_weights(seed + 3, H, 128).numpy()
        Ub = synth.bits(synth.random_orthonormal(seed + 4, H, 128, r)) if r else None
        qwm.qwm_quantize_append(cfg, cache, dev(k), dev(v), dev(synth.from_bits(kc)), dev(synth.from_bits(vc)),
                                w=torch.from_numpy(w).cuda(), U=None if Ub is None else dev(synth.from_bits(Ub)))
        torch.cuda.synchronize()
        assert cache.status() == 0
        check_chunk(cfg, cache, kb, vb, kc, vc, w, Ub, G=G, r=r, M=4, n_tok=64, seed=seed)
        hc = Held(kb, vb, kc, vc, w, Ub, heads)
        del k, v, kb, vb
        ko, vo = oracle_append(hc.kb, hc.vb, hc.kc, hc.vc, G=G, r=r, M=4, w=hc.w, U_bits=hc.Ub)
        K, V = oracle_kv(ko, vo, hc.kc, hc.vc, G=G, r=r, U_bits=hc.Ub)
        Ks.append(K)
        Vs.append(V)
    q = synth.gaussian_bf16(9500 + C, Nq, H, 128)
    kcur = synth.gaussian_bf16(9501 + C, Ncur, H, 128) if Ncur else None
    vcur = synth.gaussian_bf16(9502 + C, Ncur, H, 128) if Ncur else None
    ws = qwm.attend_workspace(cfg, cache, Nq, Ncur)
    out, lse = qwm.qwm_attend(cfg, cache, dev(q), None if kcur is None else dev(kcur),
                              None if vcur is None else dev(vcur), want_lse=True, workspace=ws)
    torch.cuda.synchronize()
    assert cache.status() == 0
    if Ncur:
        Ks.append(orc.bf16_to_f32(synth.bits(kcur)[:, heads]).astype(np.float64))
        Vs.append(orc.bf16_to_f32(synth.bits(vcur)[:, heads]).astype(np.float64))
    rows = sample_rows(Nq, 32, C)
    ref, ref_lse = orc.attend(synth.bits(q)[:, heads], np.concatenate(Ks, 0), np.concatenate(Vs, 0),
                              1 / math.sqrt(128), rows=rows)
    compare_attention(out.float().cpu().numpy()[rows][:, heads], ref)
    assert np.abs(lse.cpu().numpy()[heads][:, rows] - ref_lse).max() < 2e-2


def test_wan14b_append_with_fitted_tables_sampled_heads():
    """The bench's append configuration with k-means tables: the Wan-14B chunk
    (40 heads, 4680 tokens, C = 256, 10 Lloyd iterations).  Three heads take
    the oracle's own fitted tables (many near ties between centroids, unlike
    strided tokens); the other heads take the GPU's fit, which the k-means
    parity tests prove equal to the oracle's.  Sampled tokens of the three
    heads are compared with the oracle bit for bit under the margin rule."""
    wl = synth.WORKLOADS["wan14b_layer"]
    H, N, C, G, r, M = wl.heads, wl.chunk_tokens, wl.centroids, wl.group_size, wl.psac_rank, wl.candidates
    heads = [0, 17, 39]
    cfg = qwm.config(H, C, group_size=G, psac_rank=r, candidates=M, kmeans_iters=wl.kmeans_iters)
    src = synth.ChunkSource(wl)
    _, k, v = src.chunk(wl.past_chunks)
    a = src.query_log_scale(wl.past_chunks)
    w = synth.population_w(a).numpy()
    Ub = synth.bits(synth.population_U(a, r))
    kb, vb = synth.bits(k), synth.bits(v)
    kd, vd = dev(k), dev(v)
    kc_g = synth.bits(qwm.qwm_fit_centroids(cfg, kd).cpu())
    vc_g = synth.bits(qwm.qwm_fit_centroids(cfg, vd).cpu())
    kc_o = orc.fit_centroids(np.ascontiguousarray(kb[:, heads]), C, wl.kmeans_iters)["centroids"]
    vc_o = orc.fit_centroids(np.ascontiguousarray(vb[:, heads]), C, wl.kmeans_iters)["centroids"]
    kc, vc = kc_g.copy(), vc_g.copy()
    kc[heads], vc[heads] = kc_o, vc_o
    cache = qwm.Cache(cfg, N, 1)
    qwm.qwm_quantize_append(cfg, cache, kd, vd, dev(synth.from_bits(kc)), dev(synth.from_bits(vc)),
                            w=torch.from_numpy(w).cuda(), U=dev(synth.from_bits(Ub)))
    torch.cuda.synchronize()
    assert cache.status() == 0
    dec = cache.decode_chunk(0)
    idx = sample_rows(N, 160, 77)
    hs = np.array(heads)
    g = {key: dec[key][idx][:, hs] for key in ("ids", "codes", "scales", "zeros", "coef", "sigma",
                                               "v_ids", "v_codes", "v_scales", "v_zeros")}
    kbs = np.ascontiguousarray(kb[idx][:, hs])
    vbs = np.ascontiguousarray(vb[idx][:, hs])
    ko, vo = oracle_append(kbs, vbs, kc_o, vc_o, G=G, r=r, M=M, w=w[hs], U_bits=Ub[hs])
    compare_packed(g, ko, kbs, kc_o, G=G, r=r, M=M, is_key=True, w=w[hs], U_bits=Ub[hs])
    compare_packed(g, vo, vbs, vc_o, G=G, r=r, M=M, is_key=False, prefix="v_")
