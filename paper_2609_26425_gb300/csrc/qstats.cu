// qstats.cu -- historical Query statistics and the principal Query basis on
// the GPU (Sec. 4.1 Eq. 6 and 8, Sec. 4.2 Eq. 15, App. C.3 cold start,
// App. D.1: per-head statistics kept incrementally, the basis recomputed at
// chunk boundaries, no past Query kept).
//
//   gram_kernel   S_h += Q_h^T Q_h for one chunk of Queries.  A tile of 64
//                 tokens x 128 channels is staged by TMA (128-byte swizzle,
//                 token rows) and serves as both MMA operands read MN-major:
//                 M = N = 128 channels, K = 16 tokens per tcgen05.mma, the
//                 fp32 accumulator in TMEM.  A cluster of S CTAs splits the
//                 tokens of one head; the S partial sums meet in distributed
//                 shared memory and are added to S_h in rank order, so the
//                 result does not depend on timing.
//   basis_kernel  w from the diagonal of S (Eq. 8) and the eigenvectors of
//                 M = S / count by cyclic Jacobi in fp32 (Eq. 15).  A holds
//                 its upper triangle in shared memory; each round rotates 64
//                 disjoint index pairs (round-robin schedule) and updates each
//                 2 x 2 block of A once, in place.  The CTAs of a cluster run
//                 the same rotations on their own copy of A (same arithmetic,
//                 same bits) and each accumulates its share of the rows of the
//                 eigenvector matrix V.
#include "qwm_internal.cuh"
#include "ptx_sm103.cuh"

namespace qwm {
namespace {
using namespace ptx;

constexpr int kStatsHeader = 256;   // status word, count, sweeps; then the sums

// ------------------------------------------------------------------ Gram sums
constexpr int kGTok = 64;                        // tokens per stage
constexpr int kGStages = 6;
constexpr int kGStage = kGTok * 256;             // two 8 KB boxes: channels [0,64) and [64,128)
constexpr int kGThreads = 128;
constexpr int kGBarOff = kGStages * kGStage;     // the [128][128] fp32 partial reuses the stages
constexpr int kGBarBytes = (2 * kGStages + 1) * 8;
constexpr int kGSmem = kGBarOff + kGBarBytes + 8 + 1024;   // barriers, TMEM slot, flag, alignment slack
static_assert(kGStages * kGStage >= 128 * 128 * 4, "partial sum buffer");

__global__ void __launch_bounds__(kGThreads) gram_kernel(const __grid_constant__ CUtensorMap tm, uint8_t* stats,
                                                         int64_t N, int S) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const uint32_t base = smem_u32(sm);
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + kGBarOff);  // full[kGStages], empty[kGStages], done
  uint32_t* tslot = reinterpret_cast<uint32_t*>(sm + kGBarOff + kGBarBytes);
  volatile int* s_err = reinterpret_cast<volatile int*>(sm + kGBarOff + kGBarBytes + 4);
  auto bar = [&](int i) { return smem_u32(bars + i); };

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int h = blockIdx.y;
  const int rank = (int)cluster_rank();
  const int64_t ntile = (N + kGTok - 1) / kGTok;
  const int my = (int)((ntile - rank + S - 1) / S);  // tiles rank, rank + S, ...; >= 1 as S <= ntile

  if (tid == 0) {
    for (int i = 0; i < 2 * kGStages + 1; ++i) mbar_init(bar(i), 1);
    *s_err = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tslot), 128);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tD = *tslot;

  // rows [rank R, rank R + R) of the running sum S_h, which this CTA updates
  // at the end: loaded now, while the tiles stream in
  const int R = 128 / S;                                  // S in {1, 2, 4, 8}
  float4* gS = reinterpret_cast<float4*>(stats + kStatsHeader) + (size_t)h * (128 * 32);
  float4 acc[32];                                         // R * 32 / 128 <= 32 items per thread
  const int nit = R / 4;
#pragma unroll
  for (int m = 0; m < 32; ++m)
    if (m < nit) acc[m] = gS[rank * R * 32 + tid + 128 * m];

  if (warp == 0) {
    if (lane == 0) {  // TMA producer
      prefetch_tmap(&tm);
      for (int k = 0; k < my; ++k) {
        const int s = k % kGStages;
        if (k >= kGStages && !mbar_wait(bar(kGStages + s), ((k / kGStages) - 1) & 1)) {
          *s_err = 1;
          break;
        }
        const int n0 = (int)(((int64_t)rank + (int64_t)k * S) * kGTok);
        const uint32_t dst = base + s * kGStage;
        mbar_arrive_expect_tx(bar(s), kGStage);
        tma_load_3d(dst, &tm, 0, h, n0, bar(s));
        tma_load_3d(dst + kGStage / 2, &tm, 64, h, n0, bar(s));
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {  // MMA issuer: D[c][e] += sum over the tile's tokens of q_c q_e
      constexpr uint32_t id = idesc_f16_mn(128, 128, true);
      for (int k = 0; k < my; ++k) {
        const int s = k % kGStages;
        if (!mbar_wait(bar(s), (k / kGStages) & 1)) {
          *s_err = 1;
          break;
        }
        tc_fence_after();
        const uint32_t a = base + s * kGStage;
#pragma unroll
        for (int ks = 0; ks < kGTok / 16; ++ks) {
          const uint64_t dsc = desc_sw128_mn(a + ks * 2048, kGStage / 2);
          umma_ss(tD, dsc, dsc, id, (k | ks) != 0);
        }
        umma_commit(bar(kGStages + s));
      }
      umma_commit(bar(2 * kGStages));  // every MMA issued above has completed
    }
    __syncwarp();
  }

  // ---- this CTA's partial sum: TMEM -> shared memory, row c = TMEM lane c,
  // float4 chunks XOR-swizzled by c % 8 (conflict-free stores and loads)
  bool ok = mbar_wait(bar(2 * kGStages), 0);
  ok = __all_sync(0xFFFFFFFFu, ok);
  tc_fence_after();
  float4* red = reinterpret_cast<float4*>(sm);
  const int row = warp * 32 + lane;
#pragma unroll 1
  for (int cb = 0; cb < 4; ++cb) {
    float v[32];
    if (ok) {
      tmem_ld32(tD + ((uint32_t)(warp * 32) << 16) + (uint32_t)(cb * 32), v);
    } else {
#pragma unroll
      for (int e = 0; e < 32; ++e) v[e] = 0.0f;
    }
#pragma unroll
    for (int e4 = 0; e4 < 8; ++e4) {
      const int c4 = cb * 8 + e4;
      red[row * 32 + (c4 ^ (row & 7))] = make_float4(v[4 * e4], v[4 * e4 + 1], v[4 * e4 + 2], v[4 * e4 + 3]);
    }
  }
  if (!ok && lane == 0) *s_err = 1;
  tc_fence_before();
  cluster_sync();
  tc_fence_after();

  // ---- the running sum plus the partials of ranks 0, 1, ..., S-1, in that
  // order; the loads of all ranks for a row are issued before the adds
  const uint32_t red_s = smem_u32(red);
#pragma unroll
  for (int m = 0; m < 32; ++m) {
    if (m < nit) {
      const int i = tid + 128 * m;
      const int r = rank * R + (i >> 5), c4 = i & 31;
      const uint32_t off = red_s + (uint32_t)((r * 32 + (c4 ^ (r & 7))) * 16);
      float4 p[8];
#pragma unroll
      for (int src = 0; src < 8; ++src)
        if (src < S) p[src] = ld_dsmem_f4(mapa(off, (uint32_t)src));
#pragma unroll
      for (int src = 0; src < 8; ++src)
        if (src < S) {
          acc[m].x += p[src].x;
          acc[m].y += p[src].y;
          acc[m].z += p[src].z;
          acc[m].w += p[src].w;
        }
      gS[rank * R * 32 + i] = acc[m];
    }
  }
  cluster_sync();  // no CTA leaves while its partial is still being read
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tD, 128);
  if (tid == 0) {
    if (*s_err) atomicCAS(reinterpret_cast<int*>(stats), 0, (int)QWM_ERR_TIMEOUT);
    if (h == 0 && rank == 0) *reinterpret_cast<unsigned long long*>(stats + 8) += (unsigned long long)N;
  }
}

// ------------------------------------------------------------------ Jacobi basis
constexpr int kJs = 129;          // padded row stride: entry (i, j) in bank (i + j) % 32
constexpr int kJThreads = 512;
constexpr int kMaxSweeps = 30;

__host__ __device__ constexpr int basis_smem_bytes(int vrows) {
  return (128 + vrows) * kJs * 4   // A, V rows
         + 4 * 64 * 4              // pair tables
         + 32 * 4 + 128 * 4        // reductions, eigenvalue order
         + 32 * 16 + 32 * 4;       // sign candidates, signs
}

__global__ void __launch_bounds__(kJThreads, 1) basis_kernel(uint8_t* stats, float* w, __nv_bfloat16* U,
                                                             float* evals, int r, int eig) {
  extern __shared__ __align__(16) float js[];
  const int SJ = (int)gridDim.x;   // CTAs of this head's cluster
  const int rank = (int)cluster_rank();
  const int VR = 128 / SJ;         // rows of V kept by this CTA: rank * VR + [0, VR)
  float* A = js;                   // [128][kJs], entry (i, j) at min(i,j) * kJs + max(i,j)
  float* V = A + 128 * kJs;        // [VR][kJs]
  float* pc = V + VR * kJs;        // per pair: cos, sin, new a_ff, new a_gg
  float* psn = pc + 64;
  float* paf = psn + 64;
  float* pag = paf + 64;
  float* red = pag + 64;
  int* order = reinterpret_cast<int*>(red + 32);
  float4* cand = reinterpret_cast<float4*>(order + 128);
  float* sgn = reinterpret_cast<float*>(cand + 32);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int h = blockIdx.y;
  const unsigned long long cnt = *reinterpret_cast<const unsigned long long*>(stats + 8);
  const float* S = reinterpret_cast<const float*>(stats + kStatsHeader) + (size_t)h * 128 * 128;
  auto ut = [](int i, int j) { return i <= j ? i * kJs + j : j * kJs + i; };

  // ---- Eq. 8: w_c = S_cc / mean_c' S_c'c' (the 1/count of M cancels)
  if (tid < 128) {
    const float dg = S[tid * 129];
    float t = dg;
#pragma unroll
    for (int o = 16; o; o >>= 1) t += __shfl_xor_sync(0xFFFFFFFFu, t, o);
    if (lane == 0) red[warp] = t;
    named_bar_sync(1, 128);
    const float sum = (red[0] + red[1]) + (red[2] + red[3]);
    if (w && rank == 0) w[h * 128 + tid] = (cnt > 0 && sum > 0.0f) ? dg * 128.0f / sum : 1.0f;
  }
  if (!eig) return;
  __syncthreads();

  // ---- M = S / count into A (upper triangle), V = identity rows, ||M||_F
  const float inv = cnt ? (float)(1.0 / (double)cnt) : 0.0f;
  float ss = 0.0f;
  for (int e = tid; e < 128 * 128; e += kJThreads) {
    const int i = e >> 7, j = e & 127;
    const float a = S[e] * inv;
    if (i <= j) A[i * kJs + j] = a;
    ss = fmaf(a, a, ss);
  }
  for (int e = tid; e < VR * 128; e += kJThreads) {
    const int i = e >> 7, j = e & 127;
    V[i * kJs + j] = (rank * VR + i == j) ? 1.0f : 0.0f;
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) ss += __shfl_xor_sync(0xFFFFFFFFu, ss, o);
  if (lane == 0) red[warp] = ss;
  __syncthreads();
  float fro2 = 0.0f;
  for (int i = 0; i < kJThreads / 32; ++i) fro2 += red[i];
  const float thr = ldexpf(sqrtf(fro2), -20);   // rotate pairs whose |a_fg| exceeds this

  // ---- cyclic Jacobi sweeps; round rr pairs index 0 with 1 + rr and
  // 1 + (rr + k) % 127 with 1 + (rr - k) % 127 for k = 1..63, so each sweep
  // (127 rounds) meets every index pair once
  auto wrap = [](int x) { return x >= 127 ? x - 127 : x; };   // x < 254
  auto pair_f = [&](int rr, int k) { return k == 0 ? 0 : 1 + wrap(rr + k); };
  auto pair_g = [&](int rr, int k) { return k == 0 ? 1 + rr : 1 + wrap(rr + 127 - k); };
  int sweeps = 0;
  for (; sweeps < kMaxSweeps; ++sweeps) {
    int any = 0;
#pragma unroll 1
    for (int rr = 0; rr < 127; ++rr) {
      int rot = 0;
      if (tid < 64) {
        const int f = pair_f(rr, tid), g = pair_g(rr, tid);
        const float aff = A[f * kJs + f], agg = A[g * kJs + g], afg = A[ut(f, g)];
        float c = 1.0f, s = 0.0f, nf = aff, ng = agg;
        if (fabsf(afg) > thr) {
          // the rotation that zeroes a_fg: tan = sign(tau) / (|tau| + sqrt(1 + tau^2)),
          // |tau| <= 2^20 here; fast reciprocals: any (c, s) with c^2 + s^2 = 1
          // to rounding is an orthogonal step, and a_fg is set to zero below
          const float tau = __fdividef(agg - aff, 2.0f * afg);
          const float q = fmaf(tau, tau, 1.0f);
          const float t = __fdividef(copysignf(1.0f, tau), fabsf(tau) + q * rsqrtf(q));
          c = rsqrtf(fmaf(t, t, 1.0f));
          s = t * c;
          nf = aff - t * afg;
          ng = agg + t * afg;
          rot = 1;
        }
        pc[tid] = c;
        psn[tid] = s;
        paf[tid] = nf;
        pag[tid] = ng;
      }
      if (!__syncthreads_or(rot)) continue;
      any = 1;
      // A <- J^T A J.  Off-diagonal 2 x 2 blocks {a, b}: warp-iteration b,
      // lanes a = (b + 1 + lane) % 64 (lane 31 only for b < 32), so each
      // unordered pair of pairs is updated exactly once.  The four blocks of
      // a thread are disjoint: all loads first, then the rotations.
      {
        int ix[4][4];
        float cs[4][4], x[4][4];
        bool act[4];
#pragma unroll
        for (int it = 0; it < 4; ++it) {
          const int b = warp + 16 * it;
          const int a = (b + 1 + lane) & 63;
          cs[it][0] = pc[a];
          cs[it][1] = psn[a];
          cs[it][2] = pc[b];
          cs[it][3] = psn[b];
          act[it] = !(lane == 31 && b >= 32) && (cs[it][1] != 0.0f || cs[it][3] != 0.0f);
          const int fa = pair_f(rr, a), ga = pair_g(rr, a), fb = pair_f(rr, b), gb = pair_g(rr, b);
          ix[it][0] = ut(fa, fb);
          ix[it][1] = ut(fa, gb);
          ix[it][2] = ut(ga, fb);
          ix[it][3] = ut(ga, gb);
        }
#pragma unroll
        for (int it = 0; it < 4; ++it)
          if (act[it])
#pragma unroll
            for (int e = 0; e < 4; ++e) x[it][e] = A[ix[it][e]];
#pragma unroll
        for (int it = 0; it < 4; ++it) {
          if (!act[it]) continue;
          const float ca = cs[it][0], sa = cs[it][1], cb = cs[it][2], sb = cs[it][3];
          // columns of pair b, then rows of pair a
          const float y00 = cb * x[it][0] - sb * x[it][1], y01 = sb * x[it][0] + cb * x[it][1];
          const float y10 = cb * x[it][2] - sb * x[it][3], y11 = sb * x[it][2] + cb * x[it][3];
          A[ix[it][0]] = ca * y00 - sa * y10;
          A[ix[it][2]] = sa * y00 + ca * y10;
          A[ix[it][1]] = ca * y01 - sa * y11;
          A[ix[it][3]] = sa * y01 + ca * y11;
        }
      }
      // the diagonal block of each rotated pair in closed form
      if (tid < 64 && psn[tid] != 0.0f) {
        const int f = pair_f(rr, tid), g = pair_g(rr, tid);
        A[f * kJs + f] = paf[tid];
        A[g * kJs + g] = pag[tid];
        A[ut(f, g)] = 0.0f;
      }
      // V <- V J on this CTA's rows (columns of four disjoint pairs per warp)
      {
        int vf[4], vg[4];
        float vc[4], vs[4];
#pragma unroll
        for (int it = 0; it < 4; ++it) {
          const int b = warp + 16 * it;
          vc[it] = pc[b];
          vs[it] = psn[b];
          vf[it] = pair_f(rr, b);
          vg[it] = pair_g(rr, b);
        }
        for (int i = lane; i < VR; i += 32) {
          float x[4], y[4];
#pragma unroll
          for (int it = 0; it < 4; ++it)
            if (vs[it] != 0.0f) {
              x[it] = V[i * kJs + vf[it]];
              y[it] = V[i * kJs + vg[it]];
            }
#pragma unroll
          for (int it = 0; it < 4; ++it)
            if (vs[it] != 0.0f) {
              V[i * kJs + vf[it]] = vc[it] * x[it] - vs[it] * y[it];
              V[i * kJs + vg[it]] = vs[it] * x[it] + vc[it] * y[it];
            }
        }
      }
      __syncthreads();
    }
    if (!any) break;
  }
  const int nsweeps = sweeps < kMaxSweeps ? sweeps + 1 : kMaxSweeps;

  // ---- eigenvalues in decreasing order (equal values by increasing index;
  // NaN last)
  __syncthreads();
  if (tid < 128) {
    float ki = A[tid * kJs + tid];
    if (ki != ki) ki = -INFINITY;
    int rk = 0;
    for (int j = 0; j < 128; ++j) {
      float kj = A[j * kJs + j];
      if (kj != kj) kj = -INFINITY;
      rk += (kj > ki) || (kj == ki && j < tid);
    }
    order[rk] = tid;
  }
  __syncthreads();
  if (rank == 0) {
    if (evals && tid < 128) evals[h * 128 + tid] = A[order[tid] * kJs + order[tid]];
    if (tid == 0) atomicMax(reinterpret_cast<int*>(stats + 16), nsweeps);
  }
  if (!U || r == 0) return;

  // ---- U_r: column j = eigenvector order[j], signed so that its largest
  // |entry| (the first one on ties) is positive; the candidates of the
  // cluster's row blocks meet through distributed shared memory
  if (tid < r) {
    const int col = order[tid];
    float best = -1.0f, val = 0.0f;
    int brow = 0;
    for (int i = 0; i < VR; ++i) {
      const float v = V[i * kJs + col];
      if (fabsf(v) > best) {
        best = fabsf(v);
        brow = rank * VR + i;
        val = v;
      }
    }
    cand[tid] = make_float4(best, __int_as_float(brow), val, 0.0f);
  }
  cluster_sync();
  if (tid < r) {
    float best = -1.0f, val = 0.0f;
    for (int src = 0; src < SJ; ++src) {
      const float4 c = ld_dsmem_f4(mapa(smem_u32(cand + tid), (uint32_t)src));
      if (c.x > best) {
        best = c.x;
        val = c.z;
      }
    }
    sgn[tid] = val < 0.0f ? -1.0f : 1.0f;
  }
  cluster_sync();  // candidates read by every CTA before any leaves
  for (int e = tid; e < VR * r; e += kJThreads) {
    const int i = e / r, j = e - i * r;
    const float v = cnt ? sgn[j] * V[i * kJs + order[j]] : 0.0f;
    U[((size_t)h * 128 + rank * VR + i) * r + j] = __float2bfloat16_rn(v);
  }
}

int sm_count() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) !=
                                                 cudaSuccess || n < 1)
    return 1;
  return n;
}

bool stats_ok(const qwm_config* cfg, const void* stats) {
  return cfg && stats && config_supported(cfg) && (reinterpret_cast<uintptr_t>(stats) & 255u) == 0;
}

}  // namespace
}  // namespace qwm

extern "C" {

QWM_API size_t qwm_query_stats_bytes(const qwm_config* cfg) {
  if (!cfg || !qwm::config_supported(cfg)) return 0;
  return (size_t)qwm::kStatsHeader + (size_t)cfg->num_heads * 128 * 128 * 4;
}

QWM_API qwm_status qwm_query_stats_reset(const qwm_config* cfg, void* stats, void* stream) {
  if (!cfg || !stats) return QWM_ERR_INVALID_ARG;
  if (!qwm::config_supported(cfg)) return QWM_ERR_UNSUPPORTED;
  if (!qwm::stats_ok(cfg, stats)) return QWM_ERR_INVALID_ARG;
  return cudaMemsetAsync(stats, 0, qwm_query_stats_bytes(cfg), static_cast<cudaStream_t>(stream)) == cudaSuccess
             ? QWM_OK
             : QWM_ERR_CUDA;
}

QWM_API qwm_status qwm_query_stats_update(const qwm_config* cfg, void* stats, const void* q, int64_t N,
                                          void* stream) {
  using namespace qwm;
  if (!cfg || !stats || N < 0) return QWM_ERR_INVALID_ARG;
  if (!config_supported(cfg)) return QWM_ERR_UNSUPPORTED;
  if (!stats_ok(cfg, stats)) return QWM_ERR_INVALID_ARG;
  if (N == 0) return QWM_OK;
  if (!q || (reinterpret_cast<uintptr_t>(q) & 15u)) return QWM_ERR_INVALID_ARG;
  if (N > ((int64_t)1 << 31) - kGTok) return QWM_ERR_UNSUPPORTED;
  const int H = cfg->num_heads;
  CUtensorMap tm;
  if (!make_token_map(&tm, q, N, H, kGTok)) return QWM_ERR_CUDA;
  // S CTAs per head (a power of two <= 8, at most one per token tile), as
  // many as keep the grid within two CTAs per SM
  const int64_t ntile = (N + kGTok - 1) / kGTok;
  const int slots = 2 * sm_count();
  int S = 1;
  while (S < 8 && 2 * S <= ntile && (int64_t)H * 2 * S <= slots) S *= 2;
  if (cudaFuncSetAttribute(gram_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kGSmem) != cudaSuccess)
    return QWM_ERR_CUDA;
  cudaLaunchConfig_t lc{};
  lc.gridDim = dim3((unsigned)S, (unsigned)H);
  lc.blockDim = dim3(kGThreads);
  lc.dynamicSmemBytes = kGSmem;
  lc.stream = static_cast<cudaStream_t>(stream);
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeClusterDimension;
  at[0].val.clusterDim.x = (unsigned)S;
  at[0].val.clusterDim.y = 1;
  at[0].val.clusterDim.z = 1;
  lc.attrs = at;
  lc.numAttrs = 1;
  uint8_t* st = static_cast<uint8_t*>(stats);
  if (cudaLaunchKernelEx(&lc, gram_kernel, tm, st, N, S) != cudaSuccess) return QWM_ERR_CUDA;
  return cudaGetLastError() == cudaSuccess ? QWM_OK : QWM_ERR_CUDA;
}

QWM_API qwm_status qwm_query_basis(const qwm_config* cfg, const void* stats, float* w, void* U, float* eigenvalues,
                                   void* stream) {
  using namespace qwm;
  if (!cfg || !stats) return QWM_ERR_INVALID_ARG;
  if (!config_supported(cfg)) return QWM_ERR_UNSUPPORTED;
  if (!stats_ok(cfg, stats)) return QWM_ERR_INVALID_ARG;
  if ((w && (reinterpret_cast<uintptr_t>(w) & 3u)) || (eigenvalues && (reinterpret_cast<uintptr_t>(eigenvalues) & 3u)) ||
      (U && (reinterpret_cast<uintptr_t>(U) & 1u)))
    return QWM_ERR_INVALID_ARG;
  const int H = cfg->num_heads, r = cfg->psac_rank;
  __nv_bfloat16* Ub = (U && r > 0) ? static_cast<__nv_bfloat16*>(U) : nullptr;
  const int eig = (Ub || eigenvalues) ? 1 : 0;
  if (!w && !eig) return QWM_OK;
  // CTAs per head share the rows of V: 4, 2 or 1, one CTA per SM
  const int sms = sm_count();
  int SJ = 4;
  while (SJ > 1 && (int64_t)H * SJ > sms) SJ /= 2;
  if (!eig) SJ = 1;
  const int smem = basis_smem_bytes(128 / SJ);
  if (cudaFuncSetAttribute(basis_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess)
    return QWM_ERR_CUDA;
  cudaLaunchConfig_t lc{};
  lc.gridDim = dim3((unsigned)SJ, (unsigned)H);
  lc.blockDim = dim3(kJThreads);
  lc.dynamicSmemBytes = (size_t)smem;
  lc.stream = static_cast<cudaStream_t>(stream);
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeClusterDimension;
  at[0].val.clusterDim.x = (unsigned)SJ;
  at[0].val.clusterDim.y = 1;
  at[0].val.clusterDim.z = 1;
  lc.attrs = at;
  lc.numAttrs = 1;
  uint8_t* st = static_cast<uint8_t*>(const_cast<void*>(stats));
  if (cudaLaunchKernelEx(&lc, basis_kernel, st, w, Ub, eigenvalues, r, eig) != cudaSuccess) return QWM_ERR_CUDA;
  return cudaGetLastError() == cudaSuccess ? QWM_OK : QWM_ERR_CUDA;
}

QWM_API qwm_status qwm_query_stats_read(void* stats, int32_t* status, int64_t* count, void* stream) {
  if (!stats || !status) return QWM_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int64_t hdr[2] = {0, 0};
  if (cudaMemcpyAsync(hdr, stats, sizeof hdr, cudaMemcpyDeviceToHost, s) != cudaSuccess) return QWM_ERR_CUDA;
  if (cudaStreamSynchronize(s) != cudaSuccess) return QWM_ERR_CUDA;
  const int32_t v = (int32_t)(hdr[0] & 0xFFFFFFFF);
  if (v != 0 && cudaMemsetAsync(stats, 0, sizeof(int32_t), s) != cudaSuccess) return QWM_ERR_CUDA;
  *status = v;
  if (count) *count = hdr[1];
  return QWM_OK;
}

}  // extern "C"
