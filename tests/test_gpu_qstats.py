"""GPU parity of the Query statistics and the principal Query basis
(qwm_query_stats_update, qwm_query_basis) against the oracle's query_stats
(Sec. 4.1 Eq. 6 and 8, Sec. 4.2 Eq. 15).

What is unique is compared: the sums S_h (fp32 tensor-core accumulation of
exact bf16 products, so within 2e-4 of sum |q_c q_e| of the exact value), the
count, w, every eigenvalue, each leading eigenvector whose eigenvalue is
separated from its neighbours (up to sign; the GPU's sign rule is checked on
its own), and the leading subspace where it is separated from the rest.
Everything else (near-equal eigenvalues) is checked for validity:
orthonormality and the eigen-equation residual.
"""
import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2609_26425_gb300 import synth
import paper_2609_26425_gb300 as qwm

pytestmark = pytest.mark.gpu

SUM_RTOL = 2e-4        # of sum_n |q_nc q_ne|
EIG_TOL = 5e-5         # of ||M||_F, eigenvalues and the eigen-solver's perturbation
U_ROUND = 4e-3         # bf16 rounding of a unit vector (2^-9 per entry, relative)


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    qwm.lib()


def workload_queries(name, chunk, tokens=None, heads=None):
    src = synth.ChunkSource(synth.WORKLOADS[name])
    q, _, _ = src.chunk(chunk, tokens=tokens)
    return q if heads is None else q[:, :heads].contiguous()


def check_sums(st: qwm.QueryStats, q_all: torch.Tensor, heads=None):
    """S_h against N * M_h of the oracle, per head in `heads` (default all)."""
    qb = synth.bits(q_all)
    N, H, d = qb.shape
    heads = range(H) if heads is None else heads
    S = st.sums.cpu().double().numpy()
    qf = orc.bf16_to_f32(qb).astype(np.float64)
    for h in heads:
        M, _, _, _ = orc.query_stats(np.ascontiguousarray(qb[:, h:h + 1]), 1)
        a = np.abs(qf[:, h])
        bound = SUM_RTOL * (a.T @ a) + 1e-30
        err = np.abs(S[h] - N * M[0])
        assert np.all(err <= bound), f"head {h}: sum error {float((err / bound).max()):.2f} x the bound"


def check_basis(st: qwm.QueryStats, q_all: torch.Tensor, r: int, heads=None):
    w, U, lam = st.basis(w=True, U=True, eigenvalues=True)
    status, _ = st.read()
    assert status == 0
    assert st.sweeps() < 30, "Jacobi did not converge"
    qb = synth.bits(q_all)
    H = qb.shape[1]
    heads = range(H) if heads is None else heads
    w, lam = w.cpu().numpy(), lam.cpu().numpy()
    Ug = U.float().cpu().double().numpy() if U is not None else None
    for h in heads:
        M, wo, Uo, lo = orc.query_stats(np.ascontiguousarray(qb[:, h:h + 1]), r)
        M, wo, Uo, lo = M[0], wo[0], Uo[0], lo[0]
        fro = np.linalg.norm(M)
        assert np.allclose(w[h], wo, rtol=1e-4, atol=1e-6), f"head {h}: w"
        assert np.all(np.abs(lam[h] - lo) <= EIG_TOL * fro), f"head {h}: eigenvalues"
        assert np.all(np.diff(lam[h]) <= 0), f"head {h}: eigenvalues not decreasing"
        if Ug is None:
            continue
        u = Ug[h]
        # validity: orthonormal columns, eigen-equation residual, sign rule
        assert np.abs(u.T @ u - np.eye(r)).max() <= 3 * U_ROUND
        res = np.linalg.norm(M @ u - u * lo[:r], axis=0)
        assert np.all(res <= 2 * U_ROUND * lo[0] + EIG_TOL * fro), f"head {h}: residual {res.max():.3e}"
        assert np.all(u.max(0) >= np.abs(u.min(0)) * (1 - 2 ** -7)), f"head {h}: sign rule"
        # uniqueness where the spectrum separates the vector
        ext = np.concatenate([[np.inf], lo, [-np.inf]])
        for j in range(r):
            gap = min(ext[j] - ext[j + 1], ext[j + 1] - ext[j + 2])
            tol = U_ROUND + 4 * EIG_TOL * fro / gap
            if tol < 0.5:
                s = np.sign(np.dot(u[:, j], Uo[:, j])) or 1.0
                assert np.linalg.norm(u[:, j] - s * Uo[:, j]) <= tol, f"head {h} vector {j}"
        gap_r = lo[r - 1] - lo[r]
        tol = U_ROUND * np.sqrt(2 * r) + 4 * EIG_TOL * fro / gap_r
        if tol < 0.5:
            assert np.linalg.norm(u @ u.T - Uo @ Uo.T) <= tol, f"head {h}: leading subspace"
    return w, U, lam


@pytest.mark.parametrize("H,chunks,r", [
    (4, [880], 16),               # the single-layer workload: one chunk of Queries
    (4, [1, 63, 64, 65], 8),      # ragged tails, a single token, exact tile multiples
    (3, [1000, 880], 32),         # two chunks folded into one running sum
    (2, [4680], 16),              # one split per CTA pair of the cluster
])
def test_query_stats_parity(H, chunks, r):
    cfg = qwm.config(H, 64, psac_rank=r)
    st = qwm.QueryStats(cfg)
    qs = []
    for t, n in enumerate(chunks):
        q = workload_queries("single_layer_h4", t, tokens=n, heads=H)
        qs.append(q)
        st.update(q.cuda())
    torch.cuda.synchronize()
    status, count = st.read()
    assert status == 0 and count == sum(chunks)
    q_all = torch.cat(qs, 0)
    check_sums(st, q_all)
    check_basis(st, q_all, r)


def test_query_stats_hadamard_closed_form():
    """Orthogonal +-1 rows scaled by n + 1 (and d - n): the sums are integers
    below 2^24 (exact in fp32), the eigenvalues are the squared scales and the
    eigenvectors the rows; the diagonal is constant, so w = 1 exactly."""
    H, d, r = 2, 128, 16
    q = synth.hadamard_queries(H, d)
    cfg = qwm.config(H, 64, psac_rank=r)
    st = qwm.QueryStats(cfg)
    st.update(q.cuda())
    w, U, lam = st.basis(w=True, U=True, eigenvalues=True)
    assert st.read()[0] == 0
    qf = q.float().numpy().astype(np.float64)
    assert np.array_equal(st.sums.cpu().double().numpy(), np.einsum("nhc,nhe->hce", qf, qf))
    assert torch.all(w == 1.0)
    had = q[:, 0].double().numpy() / (np.arange(d) + 1.0)[:, None]
    lam, U = lam.cpu().double().numpy(), U.float().cpu().double().numpy()
    for h in range(H):
        s = np.arange(1, d + 1.0) if h % 2 == 0 else np.arange(d, 0, -1.0)
        ref = np.sort(s ** 2)[::-1]
        assert np.all(np.abs(lam[h] - ref) <= 1e-5 * ref[0])
        top = np.argsort(-s, kind="stable")[:r]
        for j in range(r):
            v = had[top[j]] / np.sqrt(d)
            sg = np.sign(np.dot(U[h][:, j], v))
            assert np.linalg.norm(U[h][:, j] - sg * v) <= U_ROUND


def test_query_stats_cold_start_and_zero_queries():
    """No Query yet: w = 1, U = 0, eigenvalues 0 (App. C.3).  Zero Queries:
    w = 1 and eigenvalues 0; U is then the unit channels 0..r-1."""
    H, r = 3, 8
    cfg = qwm.config(H, 64, psac_rank=r)
    st = qwm.QueryStats(cfg)
    w, U, lam = st.basis(w=True, U=True, eigenvalues=True)
    assert st.read() == (0, 0)
    assert torch.all(w == 1.0) and torch.all(U.float() == 0.0) and torch.all(lam == 0.0)
    st.update(torch.zeros(70, H, 128, dtype=torch.bfloat16, device="cuda"))
    w, U, lam = st.basis(w=True, U=True, eigenvalues=True)
    assert st.read() == (0, 70)
    assert torch.all(w == 1.0) and torch.all(lam == 0.0)
    assert torch.equal(U.float().cpu(), torch.eye(128)[:, :r].expand(H, 128, r))


def test_query_stats_deterministic_and_noop():
    """The same Queries give the same bits; N = 0 changes nothing."""
    H = 4
    q = workload_queries("single_layer_h4", 0, tokens=2000).cuda()
    cfg = qwm.config(H, 64, psac_rank=16)
    outs = []
    for _ in range(2):
        st = qwm.QueryStats(cfg)
        st.update(q)
        st.update(q[:0])
        w, U, lam = st.basis(w=True, U=True, eigenvalues=True)
        torch.cuda.synchronize()
        outs.append((st.sums.clone(), w, U, lam, st.read()))
    for a, b in zip(outs[0], outs[1]):
        if isinstance(a, torch.Tensor):
            assert torch.equal(a.view(torch.uint8) if a.dtype != torch.uint8 else a,
                               b.view(torch.uint8) if b.dtype != torch.uint8 else b)
        else:
            assert a == b == (0, 2000)


def test_causal_loop_on_gpu():
    """The loop of App. C.3 / D.1 on the GPU alone: chunk t is appended with
    the weights and basis of the Queries of chunks < t (none for t = 0), then
    its own Queries are folded in.  The statistics track the oracle's over
    all past Queries, and the cache stores the basis it was given."""
    wl = synth.WORKLOADS["single_layer_h4"]
    H, N, C, r = wl.heads, wl.chunk_tokens, wl.centroids, wl.psac_rank
    cfg = qwm.config(H, C, group_size=wl.group_size, psac_rank=r, candidates=wl.candidates)
    src = synth.ChunkSource(wl)
    st = qwm.QueryStats(cfg)
    cache = qwm.Cache(cfg, N, 3)
    ws = torch.empty(qwm.qwm_fit_workspace_bytes(cfg, N), dtype=torch.uint8, device="cuda")
    qs = []
    for t in range(3):
        q, k, v = (x.cuda() for x in src.chunk(t))
        w, U = (None, None)
        if t > 0:
            w, U, _ = st.basis(w=True, U=True)
        kc = qwm.qwm_fit_centroids(cfg, k, workspace=ws)
        vc = qwm.qwm_fit_centroids(cfg, v, workspace=ws)
        qwm.qwm_quantize_append(cfg, cache, k, v, kc, vc, w=w, U=U)
        st.update(q)
        qs.append(q.cpu())
        if U is not None:
            torch.cuda.synchronize()
            assert np.array_equal(cache.decode_chunk(t)["U"], synth.bits(U))
    torch.cuda.synchronize()
    assert cache.status() == 0 and st.read() == (0, 3 * N)
    q_all = torch.cat(qs, 0)
    check_sums(st, q_all)
    check_basis(st, q_all, r)


def test_query_stats_full_size_sampled():
    """The Wan-14B-shaped layer (40 heads, chunks of 4680 Queries drifting
    AR(1) across chunks): two chunks folded in on the GPU; sums and basis
    compared on sampled heads."""
    wl = synth.WORKLOADS["wan14b_layer"]
    H, N, r = wl.heads, wl.chunk_tokens, wl.psac_rank
    cfg = qwm.config(H, wl.centroids, psac_rank=r)
    src = synth.ChunkSource(wl)
    st = qwm.QueryStats(cfg)
    qs = []
    for t in range(2):
        q, _, _ = src.chunk(t)
        st.update(q.cuda())
        qs.append(q)
    torch.cuda.synchronize()
    assert st.read() == (0, 2 * N)
    q_all = torch.cat(qs, 0)
    heads = [0, 17, 39]
    check_sums(st, q_all, heads)
    check_basis(st, q_all, r, heads)
