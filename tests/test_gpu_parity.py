"""GPU parity: the CUDA path (through the C ABI) against the CPU oracle.

Inputs are seeded synthetic tensors from paper_2609_26425_gb300.synth; the
centroid tables fed to both sides come from the oracle's k-means or from the
generator, never from the GPU.  Packed codes, zero-points, scales and ids are
compared bit-exactly (with the oracle-margin rule for near-ties), attention
against the oracle's fp64 softmax attention over the oracle's own
reconstruction.
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


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    qwm.lib()


def dev(t):
    return t.to("cuda").contiguous()


def f16_bits(bf16_bits):
    """bf16 bit patterns -> binary16 bit patterns of the same values (torch conversion)."""
    t = synth.from_bits(bf16_bits).to(torch.float16)
    return t.view(torch.int16).numpy().view(np.uint16)


def make_chunk(seed, N, H, *, outliers=True):
    q = synth.gaussian_bf16(seed * 3 + 1, N, H, 128)
    k = synth.gaussian_bf16(seed * 3 + 2, N, H, 128)
    if outliers:
        k = k.float()
        k[:, :, [5, 40, 77, 120]] *= 8
        k = k.to(torch.bfloat16)
    v = synth.gaussian_bf16(seed * 3 + 3, N, H, 128)
    return q, k, v


def run_append_case(H, N, C, G, r, M, use_w, use_U, seed, fit_iters=None, T=None, scale_format=0):
    _, k, v = make_chunk(seed, N, H)
    kb, vb = synth.bits(k), synth.bits(v)
    if fit_iters:
        kc = orc.fit_centroids(kb, C, fit_iters)["centroids"]
        vc = orc.fit_centroids(vb, C, fit_iters)["centroids"]
    else:
        kc, vc = strided_centroids(kb, C), strided_centroids(vb, C)
    w = synth.random_weights(seed + 100, H, 128).numpy() if use_w else None
    Ub = synth.bits(synth.random_orthonormal(seed + 200, H, 128, r)) if (use_U and r > 0) else None
    cfg = qwm.config(H, C, group_size=G, psac_rank=r, candidates=M, scale_format=scale_format)
    cache = qwm.Cache(cfg, T or N, 2)
    tl = scale_format == 1
    qwm.qwm_quantize_append(cfg, cache, dev(k), dev(v), dev(synth.from_bits(kc)), dev(synth.from_bits(vc)),
                            w=None if w is None else torch.from_numpy(w).cuda(),
                            U=None if Ub is None else dev(synth.from_bits(Ub)))
    torch.cuda.synchronize()
    assert cache.status() == 0
    dec = cache.decode_chunk(0)
    ko, vo = oracle_append(kb, vb, kc, vc, G=G, r=r, M=M, w=w, U_bits=Ub, two_level=tl)
    sk = compare_packed(dec, ko, kb, kc, G=G, r=r, M=M, is_key=True, w=w, U_bits=Ub, two_level=tl)
    sv = compare_packed(dec, vo, vb, vc, G=G, r=r, M=M, is_key=False, prefix="v_", two_level=tl)
    assert np.array_equal(dec["k_tab"], f16_bits(kc)) and np.array_equal(dec["v_tab"], f16_bits(vc))
    if Ub is not None:
        assert np.array_equal(dec["U"], Ub)
    return sk, sv


@pytest.mark.parametrize("H,N,C,G,r,M,use_w,use_U", [
    (4, 880, 64, 32, 16, 4, True, True),      # the single-layer workload's shape
    (2, 300, 16, 64, 8, 4, True, True),
    (2, 257, 256, 32, 32, 4, True, True),
    (3, 130, 64, 32, 16, 1, False, False),    # cold start: w = 1, no PSAC
    (2, 200, 8, 32, 16, 8, True, True),       # exhaustive QSAC (M = C)
    (2, 129, 64, 64, 0, 4, True, False),      # PSAC disabled by rank 0
    (1, 1, 4, 32, 8, 4, True, True),          # a single token
    (2, 150, 64, 32, 16, 12, True, True),     # 8 < M < C: the generic kernel
    (2, 300, 256, 64, 32, 2, True, True),     # G = 64 with the largest table
])
def test_append_parity(H, N, C, G, r, M, use_w, use_U):
    sk, sv = run_append_case(H, N, C, G, r, M, use_w, use_U, seed=H * 1000 + N)
    assert sk["id_flips"] <= max(1, N * H // 1000)


@pytest.mark.parametrize("H,N,C,G,r,M", [
    (4, 880, 64, 32, 16, 4),      # the single-layer workload's shape
    (2, 300, 256, 64, 32, 2),     # G = 64
    (2, 150, 64, 32, 16, 12),     # 8 < M < C: the generic kernel
    (1, 1, 4, 32, 8, 4),          # a single token
])
def test_append_parity_two_level_scales(H, N, C, G, r, M):
    """Scale format 1 (App. D.1): uint8 group codes with a binary16 secondary
    scale per token-head, bit-exact against the oracle's two-level scales."""
    sk, sv = run_append_case(H, N, C, G, r, M, True, True, seed=H * 1000 + N + 7, scale_format=1)
    assert sk["id_flips"] <= max(1, N * H // 1000)


@pytest.mark.parametrize("H,N,C,r,M,use_U", [
    (2, 300, 64, 16, 4, True),       # the fused kernel's candidate filter, ragged tail tile
    (2, 257, 16, 8, 4, True),        # r = 8: a tile needs two dropped rows to go sparse
    (3, 130, 64, 32, 1, True),
    (2, 200, 8, 16, 8, True),        # exhaustive QSAC (M = C)
    (2, 300, 64, 16, 4, False),      # cold start: no row kept, every tile sparse and empty
    (2, 150, 64, 16, 12, True),      # 8 < M < C: the exhaustive-distance kernel and its tile finish
    (2, 150, 64, 16, 12, False),     # the same, cold start: every tile sparse and empty
    (1, 333, 32, 32, 10, True),      # the same, r = 32, ragged tail tile
])
def test_psac_tile_layout_matches_oracle(H, N, C, r, M, use_U):
    """App. D.1 dense/sparse PSAC layouts per 128-token tile: the GPU stores
    the layout the oracle chooses (keep mask, byte count), and the rows read
    back through the mask equal the oracle's (compare_packed)."""
    _, k, v = make_chunk(H * 77 + N, N, H)
    kb, vb = synth.bits(k), synth.bits(v)
    kc, vc = strided_centroids(kb, C), strided_centroids(vb, C)
    w = synth.random_weights(N + 5, H, 128).numpy()
    Ub = synth.bits(synth.random_orthonormal(N + 6, H, 128, r)) if use_U else None
    cfg = qwm.config(H, C, psac_rank=r, candidates=M)
    cache = qwm.Cache(cfg, N, 1)
    qwm.qwm_quantize_append(cfg, cache, dev(k), dev(v), dev(synth.from_bits(kc)), dev(synth.from_bits(vc)),
                            w=torch.from_numpy(w).cuda(), U=None if Ub is None else dev(synth.from_bits(Ub)))
    assert cache.status() == 0
    dec = cache.decode_chunk(0)
    ko, vo = oracle_append(kb, vb, kc, vc, G=32, r=r, M=M, w=w, U_bits=Ub)
    compare_packed(dec, ko, kb, kc, G=32, r=r, M=M, is_key=True, w=w, U_bits=Ub)
    ntile = -(-N // 128)
    for h in range(H):
        pm = dec["pmask"][h]
        full = np.zeros((ntile, 4), np.uint32)
        for t in range(ntile):
            nt = min(128, N - 128 * t)
            for wd in range(4):
                nb = nt - 32 * wd
                full[t, wd] = 0xFFFFFFFF if nb >= 32 else ((1 << nb) - 1 if nb > 0 else 0)
        gpu_sparse = (pm != full).any(-1)
        kept_bits = np.array([[bin(int(x)).count("1") for x in row] for row in pm]).sum(-1)
        sp, nb = orc.psac_tile_layout(ko["kept"][:, h], r)
        assert np.array_equal(gpu_sparse, sp), (h, gpu_sparse, sp)
        gpu_bytes = np.where(gpu_sparse, 16 + kept_bits * (r + 2),
                             np.minimum(128, N - 128 * np.arange(ntile)) * (r + 2))
        assert np.array_equal(gpu_bytes, nb)
        # a sparse tile's mask is the oracle's keep set
        for t in np.nonzero(sp)[0]:
            kt = ko["kept"][128 * t: 128 * t + 128, h].astype(bool)
            bits = ((pm[t][np.arange(kt.size) // 32] >> (np.arange(kt.size) % 32).astype(np.uint32)) & 1).astype(bool)
            assert np.array_equal(bits, kt)


@pytest.mark.parametrize("kind,H,N,C,M", [
    ("diag", 2, 300, 64, 4),       # M = diag(w): the full form evaluated on a diagonal matrix
    ("dense", 2, 300, 64, 4),      # a dense symmetric positive M
    ("dense", 2, 257, 256, 2),     # the largest table, ragged tile
    ("dense", 1, 130, 16, 1),
    ("dense", 2, 200, 8, 8),       # M = C: every centroid a candidate (the matrix plays no part)
])
def test_append_full_matrix_distance_parity(kind, H, N, C, M):
    """App. C.4 ablation: the Keys' top-M candidates by the full quadratic form
    (k - mu)^T M (k - mu), bit-exact against the oracle's full-form path
    under the margin rule (the QSAC score and everything after keep w)."""
    _, k, v = make_chunk(H * 31 + N, N, H)
    kb, vb = synth.bits(k), synth.bits(v)
    kc, vc = strided_centroids(kb, C), strided_centroids(vb, C)
    w = synth.random_weights(N + 11, H, 128).numpy()
    r = 16
    Ub = synth.bits(synth.random_orthonormal(N + 12, H, 128, r))
    if kind == "diag":
        Mq = np.stack([np.diag(w[h]) for h in range(H)]).astype(np.float32)
    else:
        R = np.random.default_rng(N).standard_normal((H, 128, 128))
        Mq = (np.einsum("hij,hkj->hik", R, R) / 128).astype(np.float32)
    cfg = qwm.config(H, C, psac_rank=r, candidates=M)
    cache = qwm.Cache(cfg, N, 1)
    qwm.qwm_quantize_append_full(cfg, cache, dev(k), dev(v), dev(synth.from_bits(kc)), dev(synth.from_bits(vc)),
                                 torch.from_numpy(Mq).cuda(), w=torch.from_numpy(w).cuda(), U=dev(synth.from_bits(Ub)))
    assert cache.status() == 0
    dec = cache.decode_chunk(0)
    ko = orc.quantize(kb, kc, G=32, r=r, M=M, is_key=True, w=w, U_bits=Ub, M_full=Mq)
    vo = orc.quantize(vb, vc, G=32, r=r, M=M, is_key=False)
    # margin-rule requantisation keeps the full form: compare ids through the oracle with M_full
    diff = dec["ids"] != ko["ids"]
    if diff.any():
        margin = np.minimum(ko["m_topm"], ko["m_sel"])
        assert not (diff & (margin >= 1e-5)).any()
        ko = orc.quantize(kb, kc, G=32, r=r, M=M, is_key=True, w=w, U_bits=Ub, M_full=Mq, force_ids=dec["ids"])
    for key in ("codes", "scales", "zeros"):
        assert np.array_equal(dec[key], ko[key]), key
    row_bad = (dec["coef"] != ko["coef"]).any(-1) | (dec["sigma"] != ko["sigma"])
    assert np.all(ko["m_psac"][row_bad] < 1e-5)
    compare_packed(dec, vo, vb, vc, G=32, r=r, M=M, is_key=False, prefix="v_")


def test_append_full_matrix_rejects_the_exhaustive_kernel_range():
    cfg = qwm.config(2, 64, candidates=12)
    cache = qwm.Cache(cfg, 10, 1)
    z = torch.zeros(10, 2, 128, dtype=torch.bfloat16, device="cuda")
    t = torch.zeros(2, 64, 128, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(qwm.QwmError) as e:
        qwm.qwm_quantize_append_full(cfg, cache, z, z, t, t, torch.zeros(2, 128, 128, device="cuda"))
    assert e.value.status == 2


def test_append_parity_fitted_tables():
    """Tables from the oracle's k-means (the realistic case: many near ties)."""
    run_append_case(4, 880, 64, 32, 16, 4, True, True, seed=7, fit_iters=10)


@pytest.mark.parametrize("H,N,C,iters", [
    (4, 880, 64, 10),      # the single-layer workload's table
    (3, 130, 4, 5),        # fewer centroids than one MMA column block
    (2, 1000, 100, 4),     # C not a multiple of 16
    (2, 257, 256, 3),      # the largest table, ragged tile
    (1, 1, 1, 2),          # one token, one centroid
    (2, 5000, 255, 2),
    (2, 300, 64, 0),       # no iteration: the initial tokens
])
def test_fit_parity(H, N, C, iters):
    """Lloyd k-means on the GPU equals the oracle's bit for bit: the tensor
    cores only screen, every assignment is decided on the sequential fp32
    distance and every mean is the fp32 rounding of the exact mean."""
    _, k, _ = make_chunk(11 + N, N, H)
    kb = synth.bits(k)
    ref = orc.fit_centroids(kb, C, iters)
    cfg = qwm.config(H, C, kmeans_iters=iters)
    got = synth.bits(qwm.qwm_fit_centroids(cfg, dev(k)).cpu())
    nbad = int((got != ref["centroids"]).any(-1).sum())
    assert nbad == 0, f"{nbad} of {H * C} centroids differ"


def test_fit_parity_off_grid_members():
    """Entries of +-2^-45 among N(0, 1) values fall below the fixed-point grid
    of the exact member sums (its unit is 2^-43 here), so their clusters take
    the fp64 path; the fp64 sums stay exact (49 bits), and the fit must still
    equal the oracle bit for bit."""
    H, N, C, iters = 2, 300, 16, 3
    g = torch.Generator().manual_seed(5)
    x = torch.randn(N, H, 128, generator=g)
    tiny = torch.rand(N, H, 128, generator=g) < 0.01
    x = torch.where(tiny, torch.sign(x) * 2.0 ** -45, x).to(torch.bfloat16)
    xb = synth.bits(x)
    ref = orc.fit_centroids(xb, C, iters)
    got = synth.bits(qwm.qwm_fit_centroids(qwm.config(H, C, kmeans_iters=iters), dev(x)).cpu())
    assert np.array_equal(got, ref["centroids"])


@pytest.mark.parametrize("rows,C,iters", [
    ([(2.0, 0.0), (-2.0, 0.0), (0.0, 1.0)], 2, 1),                 # exact tie -> lower index
    ([(1.0, 0.0), (1.0, 0.5), (1.0, 0.0), (1.0, 1.5)], 2, 1),      # cluster 1 empty after step 1
    ([(1.0, 0.0), (1.0, 0.5), (1.0, 0.0), (1.0, 1.5)], 2, 2),
])
def test_fit_parity_ties_and_empty_clusters(rows, C, iters):
    """The hand fixtures of the oracle's k-means pins (exact distance ties,
    an empty cluster keeping its centroid) give the same centroids on the GPU."""
    x = np.zeros((len(rows), 1, 128), np.float32)
    for i, row in enumerate(rows):
        x[i, 0, : len(row)] = row
    xt = torch.from_numpy(x).to(torch.bfloat16)
    ref = orc.fit_centroids(synth.bits(xt), C, iters)
    got = synth.bits(qwm.qwm_fit_centroids(qwm.config(1, C, kmeans_iters=iters), dev(xt)).cpu())
    assert np.array_equal(got, ref["centroids"])


def test_fit_parity_full_size_sampled():
    """The Wan-14B-shaped Keys and Values (40 heads, 4680 tokens, 256
    centroids, 10 iterations); the oracle runs on three sampled heads."""
    wl = synth.WORKLOADS["wan14b_layer"]
    src = synth.ChunkSource(wl)
    _, k, v = src.chunk(0)
    cfg = qwm.config(wl.heads, wl.centroids, kmeans_iters=wl.kmeans_iters)
    heads = [0, 21, 39]
    for x in (k, v):
        got = synth.bits(qwm.qwm_fit_centroids(cfg, dev(x)).cpu())
        ref = orc.fit_centroids(synth.bits(x[:, heads].contiguous()), wl.centroids, wl.kmeans_iters)
        assert np.array_equal(got[heads], ref["centroids"])


def build_cache_and_reference(H, chunk_sizes, C, G, r, M, seed, *, Ncur, Nq, window=0, max_chunks=None,
                              psac_chunks=None, rows=None, scale_format=0):
    """Append chunks on the GPU and build the oracle's reference keys/values."""
    cfg = qwm.config(H, C, group_size=G, psac_rank=r, candidates=M, scale_format=scale_format)
    T = max(chunk_sizes)
    cache = qwm.Cache(cfg, T, max_chunks or len(chunk_sizes), sliding_window=bool(window))
    Ks, Vs = [], []
    for ci, N in enumerate(chunk_sizes):
        _, k, v = make_chunk(seed + ci, N, H)
        kb, vb = synth.bits(k), synth.bits(v)
        kc, vc = strided_centroids(kb, C), strided_centroids(vb, C)
        use_psac = r > 0 and (psac_chunks is None or ci in psac_chunks)
        w = synth.random_weights(seed + 50 + ci, H, 128).numpy() if ci > 0 else None
        Ub = synth.bits(synth.random_orthonormal(seed + 80 + ci, H, 128, r)) if use_psac else None
        qwm.qwm_quantize_append(cfg, cache, dev(k), dev(v), dev(synth.from_bits(kc)), dev(synth.from_bits(vc)),
                                w=None if w is None else torch.from_numpy(w).cuda(),
                                U=None if Ub is None else dev(synth.from_bits(Ub)))
        ko, vo = oracle_append(kb, vb, kc, vc, G=G, r=r, M=M, w=w, U_bits=Ub, two_level=scale_format == 1)
        K, V = oracle_kv(ko, vo, kc, vc, G=G, r=r, U_bits=Ub)
        Ks.append(K)
        Vs.append(V)
    n_keep = cache.num_chunks
    Ks, Vs = Ks[len(Ks) - n_keep:], Vs[len(Vs) - n_keep:]
    q, kcur, vcur = make_chunk(seed + 999, max(Nq, Ncur, 1), H, outliers=True)
    q = q[:Nq].contiguous()
    kcur, vcur = kcur[:Ncur].contiguous(), vcur[:Ncur].contiguous()
    if Ncur:
        Ks.append(orc.bf16_to_f32(synth.bits(kcur)).astype(np.float64))
        Vs.append(orc.bf16_to_f32(synth.bits(vcur)).astype(np.float64))
    Kall, Vall = np.concatenate(Ks, 0), np.concatenate(Vs, 0)
    scale = 1 / math.sqrt(128)
    ref, lse = orc.attend(synth.bits(q), Kall, Vall, scale, rows=rows)
    return cfg, cache, q, kcur, vcur, ref, lse


@pytest.mark.parametrize("split", [False, True])
@pytest.mark.parametrize("H,chunks,C,G,r,Ncur,Nq", [
    (4, [880, 880], 64, 32, 16, 880, 880),    # the single-layer workload
    (2, [300, 77], 16, 64, 8, 129, 200),
    (2, [256, 256], 256, 32, 32, 0, 130),     # no active chunk
    (2, [128], 64, 32, 0, 1, 1),              # r = 0, one query, one active key
    (1, [1, 5], 4, 32, 16, 0, 33),            # tiny chunks
    (3, [300, 200, 129, 77], 16, 32, 16, 50, 1100),  # four chunks and an active one, ragged query blocks
])
def test_attend_parity(H, chunks, C, G, r, Ncur, Nq, split):
    """Attention against the oracle's fp64 softmax; split: through
    qwm_attend_ws, whose work units are split along the key chunks (every unit
    here: they are fewer than the GPU's CTA pairs) and combined."""
    cfg, cache, q, kc, vc, ref, lse = build_cache_and_reference(H, chunks, C, G, r, 4, seed=31 * H + Nq,
                                                               Ncur=Ncur, Nq=Nq)
    ws = qwm.attend_workspace(cfg, cache, Nq, Ncur) if split else None
    if split:
        assert ws is not None and ws.numel() > 0  # more than one key unit: the parts are used
    out, lse_g = qwm.qwm_attend(cfg, cache, dev(q), dev(kc) if Ncur else None, dev(vc) if Ncur else None,
                                want_lse=True, workspace=ws)
    torch.cuda.synchronize()
    assert cache.status() == 0
    compare_attention(out.float().cpu().numpy(), ref)
    assert np.abs(lse_g.cpu().numpy() - lse).max() < 2e-2


def test_attend_workspace_sizing_and_small_buffer():
    """qwm_attend_ws needs no scratch over a single key unit; a buffer smaller
    than qwm_attend_workspace_bytes runs the unsplit launch (the same bits as
    qwm_attend); the split launch agrees with the oracle and with the unsplit
    output within the attention tolerance."""
    cfg, cache, q, _, _, _, _ = build_cache_and_reference(2, [300], 16, 32, 16, 4, seed=5, Ncur=0, Nq=200)
    assert qwm.qwm_attend_workspace_bytes(cfg, cache, 200, 0) == 0
    assert qwm.attend_workspace(cfg, cache, 200, 0) is None
    cfg, cache, q, kc, vc, ref, _ = build_cache_and_reference(2, [300, 77], 16, 32, 16, 4, seed=6, Ncur=129, Nq=200)
    need = qwm.qwm_attend_workspace_bytes(cfg, cache, 200, 129)
    assert need > 0
    plain = qwm.qwm_attend(cfg, cache, dev(q), dev(kc), dev(vc))
    small = torch.empty(256, dtype=torch.uint8, device="cuda")
    fallback = qwm.qwm_attend(cfg, cache, dev(q), dev(kc), dev(vc), workspace=small)
    split = qwm.qwm_attend(cfg, cache, dev(q), dev(kc), dev(vc), workspace=qwm.attend_workspace(cfg, cache, 200, 129))
    torch.cuda.synchronize()
    assert cache.status() == 0
    assert torch.equal(plain, fallback)
    compare_attention(split.float().cpu().numpy(), ref)
    assert (split.float() - plain.float()).abs().max().item() < 2e-2


@pytest.mark.parametrize("H,chunks,C,G,r,Ncur,Nq", [
    (4, [880, 880], 64, 32, 16, 880, 880),
    (2, [300, 77], 16, 64, 8, 129, 200),
])
def test_attend_parity_two_level_scales(H, chunks, C, G, r, Ncur, Nq):
    """Attention over a cache stored with scale format 1 (group scale = code *
    secondary scale, rebuilt in binary16) against the oracle's fp64 attention
    over its own two-level reconstruction."""
    cfg, cache, q, kc, vc, ref, lse = build_cache_and_reference(H, chunks, C, G, r, 4, seed=37 * H + Nq,
                                                               Ncur=Ncur, Nq=Nq, scale_format=1)
    out, lse_g = qwm.qwm_attend(cfg, cache, dev(q), dev(kc) if Ncur else None, dev(vc) if Ncur else None,
                                want_lse=True)
    torch.cuda.synchronize()
    assert cache.status() == 0
    compare_attention(out.float().cpu().numpy(), ref)
    assert np.abs(lse_g.cpu().numpy() - lse).max() < 2e-2


def test_attend_sliding_window_and_cold_chunk():
    """A ring of 2 slots after 4 appends holds the last two chunks; the first
    held chunk was appended without PSAC (cold start)."""
    cfg, cache, q, kc, vc, ref, _ = build_cache_and_reference(2, [200, 150, 180, 90], 16, 32, 16, 4, seed=5,
                                                             Ncur=64, Nq=100, window=1, max_chunks=2,
                                                             psac_chunks={3})
    assert cache.num_chunks == 2
    out = qwm.qwm_attend(cfg, cache, dev(q), dev(kc), dev(vc))
    torch.cuda.synchronize()
    compare_attention(out.float().cpu().numpy(), ref)


def test_attend_lossless_cache_equals_dense_attention():
    """Keys/values on the INT2 grid with a zero centroid reconstruct exactly, so
    attention over the cache equals attention over the raw bf16 tensors."""
    H, N, d, G = 2, 256, 128, 32
    rng = np.random.default_rng(9)
    s = 0.25
    def grid():
        m = rng.integers(-1, 3, size=(N, H, d)).astype(np.float32)
        m[..., ::G] = -1
        m[..., 1::G] = 2
        return torch.from_numpy(m * s).to(torch.bfloat16)
    k, v = grid(), grid()
    q = synth.gaussian_bf16(10, 77, H, d)
    cfg = qwm.config(H, 1, group_size=G, psac_rank=0, candidates=1)
    cache = qwm.Cache(cfg, N, 1)
    zc = torch.zeros(H, 1, d, dtype=torch.bfloat16)
    qwm.qwm_quantize_append(cfg, cache, dev(k), dev(v), dev(zc), dev(zc))
    out = qwm.qwm_attend(cfg, cache, dev(q))
    torch.cuda.synchronize()
    qf = q.double().permute(1, 0, 2)
    ref = torch.nn.functional.scaled_dot_product_attention(qf, k.double().permute(1, 0, 2),
                                                           v.double().permute(1, 0, 2)).permute(1, 0, 2)
    compare_attention(out.float().cpu().numpy(), ref.numpy())


def test_error_paths():
    H = 2
    cfg = qwm.config(H, 16, group_size=32, psac_rank=16)
    cache = qwm.Cache(cfg, 100, 1)
    _, k, v = make_chunk(3, 101, H)
    kc = dev(torch.zeros(H, 16, 128, dtype=torch.bfloat16))
    with pytest.raises(qwm.QwmError) as e:
        qwm.qwm_quantize_append(cfg, cache, dev(k), dev(v), kc, kc)
    assert e.value.status == 3  # capacity
    qwm.qwm_quantize_append(cfg, cache, dev(k[:100]), dev(v[:100]), kc, kc)
    with pytest.raises(qwm.QwmError) as e:  # full, no sliding window
        qwm.qwm_quantize_append(cfg, cache, dev(k[:10]), dev(v[:10]), kc, kc)
    assert e.value.status == 3
    bad = qwm.config(H, 16, group_size=16)
    assert qwm.qwm_cache_bytes(bad, 100, 1) == 0
    with pytest.raises(qwm.QwmError):
        qwm.qwm_attend(cfg, cache, dev(k[:4]), sm_scale=-1.0)
    empty = qwm.Cache(cfg, 100, 1)
    with pytest.raises(qwm.QwmError) as e:  # no keys at all
        qwm.qwm_attend(cfg, empty, dev(k[:4]))
    assert e.value.status == 1
    fresh = qwm.Cache(cfg, 100, 1)
    buf = torch.zeros(H * 16 * 128 + 8, dtype=torch.bfloat16, device="cuda")
    kc16 = buf[8:].view(H, 16, 128)  # 16-byte aligned, not 32: centroid rows are read as 32-byte sectors
    with pytest.raises(qwm.QwmError) as e:
        qwm.qwm_quantize_append(cfg, fresh, dev(k[:10]), dev(v[:10]), kc16, kc16)
    assert e.value.status == 1
    out = qwm.qwm_attend(cfg, cache, dev(k[:0]))  # Nq = 0 is a no-op
    assert out.shape[0] == 0
    torch.cuda.synchronize()
    assert cache.status() == 0
