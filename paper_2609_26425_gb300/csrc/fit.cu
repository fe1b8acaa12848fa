// fit.cu -- k-means centroids of one chunk per head (Sec. 2: the
// centroid-residual form of QVG with centroids kept in BF16, App. D.1).
//
// Lloyd's algorithm with the arithmetic of its plain definition: initial
// centroid j = token floor(j*N/C); each iteration assigns every token to its
// Euclidean-nearest centroid, the distance being the fp32 sum in channel order
// of the rounded squares of the rounded differences (ties to the lower
// index), then replaces each non-empty cluster by the fp32 rounding of its
// fp64 member mean; the result is rounded to bf16.  Per iteration:
//
//   fit_assign  (persistent, one CTA per SM, tcgen05).  A 128-token tile
//     arrives by TMA and two MMAs per K step accumulate
//     P = X mu_hi^T + X mu_lo^T in TMEM (mu_hi = bf16(mu), mu_lo =
//     bf16(mu - mu_hi): mu to 2^-18 relative; bf16 x bf16 products are exact).
//     With dt_j = |mu_j|^2 - 2 P_j, |dt_j + |x|^2 - d_j| stays below
//     E = 2^-11 (|x|^2 + max_j |mu_j|^2) for the sequential fp32 distance d_j
//     (operand split 2^-18, fp32 accumulation of 256 products 2^-15, the
//     norms and the sequential sum's own rounding (d + 2) 2^-24, each relative
//     to |x|^2 + |mu_j|^2, with margin).  Every centroid within 2E of the
//     smallest dt is therefore a candidate for the exact argmin; a row with a
//     single candidate is decided, the others (a few percent) are rescored
//     with the sequential fp32 distance.
//   fit_scatter (one CTA per head): counting sort of the tokens by cluster.
//   fit_means   (one warp per centroid): exact fp64 member sums (bf16 values
//     of ordinary range add exactly, so the order does not matter), the mean,
//     and the next iteration's operand images and norm.
#include <mutex>

#include "ptx_sm103.cuh"
#include "qwm_internal.cuh"

namespace qwm {
namespace {

using namespace ptx;

constexpr int AT = 128;                       // tokens per tile
constexpr int AEW = 16;                       // epilogue warps: rows 32 (w & 3) + lane, column quarter w >> 2
constexpr int ANT = (AEW + 1) * 32;           // + one producer / MMA warp
constexpr int kPairCap = 1024;                // (row, centroid) pairs rescored per tile
constexpr int kRowCap = 8;                    // candidates per row
constexpr int A_X = 0;                        // 2 token tiles, each 2 x [128 rows][128 B] bf16
constexpr int A_IMG = 65536;                  // operand images hi, lo: 2 x 2 x [Npad][128 B]
constexpr int A_NRM = A_IMG + 131072;         // |mu_j|^2 [256] for each TMEM buffer
constexpr int A_PJ = A_NRM + 2048;            // pair (row << 16 | j) [kPairCap]
constexpr int A_PD = A_PJ + kPairCap * 4;     // pair distance [kPairCap]
constexpr int A_ROW = A_PD + kPairCap * 4;    // row: first slot << 16 | count (0xFFFF: full scan)
constexpr int A_MIN = A_ROW + AT * 4;         // [4 quarters][128] partial minima
constexpr int A_CNT = A_MIN + 4 * AT * 4;     // [4 quarters][128] candidate counts
constexpr int A_CND = A_CNT + 4 * AT * 4;     // [128][4 quarters][kRowCap] candidates (u8)
constexpr int A_BAR = A_CND + AT * 4 * kRowCap;   // mbarriers, pair counter, flag, TMEM slot
constexpr int A_SMEM = A_BAR + 128 + 1024;

// Byte offset of 16-byte chunk `ch` (channels 8ch..8ch+7) of row `row` in two
// 128-byte-swizzled blocks of `rows` rows x 64 two-byte elements.
__device__ __forceinline__ int sw_off(int rows, int row, int ch) {
  return (ch >> 3) * rows * 128 + row * 128 + (((ch & 7) ^ (row & 7)) << 4);
}

// The sequential fp32 distance of the definition: channel order, the
// difference, its square and the running sum each rounded on its own.  The
// centroid row is fetched whole first (one memory round trip), then summed.
__device__ float exact_dist(const uint8_t* sX, int row, const float* mu) {
  float4 mv[32];
#pragma unroll
  for (int i = 0; i < 32; ++i) mv[i] = __ldg(reinterpret_cast<const float4*>(mu) + i);
  float acc = 0.0f;
#pragma unroll
  for (int ch = 0; ch < 16; ++ch) {
    const uint4 xv = *reinterpret_cast<const uint4*>(sX + sw_off(128, row, ch));
    const uint32_t xw[4] = {xv.x, xv.y, xv.z, xv.w};
    const float ms[8] = {mv[2 * ch].x, mv[2 * ch].y, mv[2 * ch].z, mv[2 * ch].w,
                         mv[2 * ch + 1].x, mv[2 * ch + 1].y, mv[2 * ch + 1].z, mv[2 * ch + 1].w};
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      const float xe = (e & 1) ? __uint_as_float(xw[e >> 1] & 0xFFFF0000u) : __uint_as_float(xw[e >> 1] << 16);
      const float t = __fsub_rn(xe, ms[e]);
      acc = __fadd_rn(acc, __fmul_rn(t, t));
    }
  }
  return acc;
}

// Operand images and norm of centroid j of head h from its fp32 row (one
// warp, lane = channels 4 lane .. 4 lane + 3).
__device__ __forceinline__ void emit_row(const FitArgs& a, int h, int j, float4 m, int lane) {
  const int c0 = 4 * lane;
  const __nv_bfloat162 h01 = __floats2bfloat162_rn(m.x, m.y), h23 = __floats2bfloat162_rn(m.z, m.w);
  const float2 f01 = __bfloat1622float2(h01), f23 = __bfloat1622float2(h23);
  const __nv_bfloat162 l01 = __floats2bfloat162_rn(m.x - f01.x, m.y - f01.y);
  const __nv_bfloat162 l23 = __floats2bfloat162_rn(m.z - f23.x, m.w - f23.y);
  const size_t off = (size_t)sw_off(a.Npad, j, c0 >> 3) + (size_t)(c0 & 7) * 2;
  uint8_t* hi = a.img + (size_t)h * 2 * a.Npad * 256;
  uint8_t* lo = hi + (size_t)a.Npad * 256;
  *reinterpret_cast<uint2*>(hi + off) =
      make_uint2(*reinterpret_cast<const uint32_t*>(&h01), *reinterpret_cast<const uint32_t*>(&h23));
  *reinterpret_cast<uint2*>(lo + off) =
      make_uint2(*reinterpret_cast<const uint32_t*>(&l01), *reinterpret_cast<const uint32_t*>(&l23));
  float n2 = fmaf(m.x, m.x, fmaf(m.y, m.y, fmaf(m.z, m.z, m.w * m.w)));
#pragma unroll
  for (int o = 16; o; o >>= 1) n2 += __shfl_xor_sync(0xFFFFFFFFu, n2, o);
  if (lane == 0) {
    a.nrm[(size_t)h * a.Npad + j] = n2;
    atomicMax(a.nmax + h, __float_as_uint(n2));  // n2 >= 0: the bits order like the values
  }
}

// Initial centroids (token floor(j N / C)) and their images; padding rows
// j in [C, Npad) get zero images and norm.  One warp per (head, row).
__global__ void __launch_bounds__(512) fit_prep(const FitArgs a) {
  const int lane = threadIdx.x & 31;
  const int64_t w = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  if (w >= (int64_t)a.H * a.Npad) return;
  const int h = (int)(w / a.Npad), j = (int)(w % a.Npad);
  if (j >= a.C) {
    const size_t off = (size_t)sw_off(a.Npad, j, lane >> 1) + (size_t)(lane & 1) * 8;
    uint8_t* hi = a.img + (size_t)h * 2 * a.Npad * 256;
    *reinterpret_cast<uint2*>(hi + off) = make_uint2(0, 0);
    *reinterpret_cast<uint2*>(hi + (size_t)a.Npad * 256 + off) = make_uint2(0, 0);
    if (lane == 0) a.nrm[(size_t)h * a.Npad + j] = INFINITY;  // padding columns never win
    return;
  }
  const int64_t src = ((int64_t)j * a.N) / a.C;
  const uint2 xv = __ldg(reinterpret_cast<const uint2*>(a.x + ((size_t)src * a.H + h) * 128 + 4 * lane));
  const float4 m = make_float4(__uint_as_float(xv.x << 16), __uint_as_float(xv.x & 0xFFFF0000u),
                               __uint_as_float(xv.y << 16), __uint_as_float(xv.y & 0xFFFF0000u));
  reinterpret_cast<float4*>(a.cent + ((size_t)h * a.C + j) * 128)[lane] = m;
  emit_row(a, h, j, m, lane);
}

// Assignment of every token (see the file comment).  Units are (head, tile)
// in head-major order, split into contiguous runs over the CTAs.  Warp 8 loads
// (TMA) and multiplies (tcgen05) tile t + 1 into the second token buffer and
// TMEM accumulator while warps 0-7 finish tile t: two warps per row, one per
// column half of the accumulator, meeting in shared memory.
__global__ void __launch_bounds__(ANT, 1)
    fit_assign(const FitArgs a, const __grid_constant__ CUtensorMap tm, int tiles, int units) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int C = a.C, Npad = a.Npad;
  uint32_t* sPJ = reinterpret_cast<uint32_t*>(sm + A_PJ);
  float* sPD = reinterpret_cast<float*>(sm + A_PD);
  uint32_t* sRow = reinterpret_cast<uint32_t*>(sm + A_ROW);
  float* sMin = reinterpret_cast<float*>(sm + A_MIN);
  int* sCnt = reinterpret_cast<int*>(sm + A_CNT);
  uint8_t* sCnd = sm + A_CND;
  const uint32_t bars = smem_u32(sm + A_BAR);
  auto bar_tma = [&](int b) { return bars + 8 * b; };          // token tile b landed
  auto bar_mma = [&](int b) { return bars + 16 + 8 * b; };     // accumulator b complete
  auto bar_free = [&](int b) { return bars + 32 + 8 * b; };    // tile b and accumulator b consumed
  const uint32_t bar_img = bars + 48;
  int* s_np = reinterpret_cast<int*>(sm + A_BAR + 64);
  volatile int* s_err = reinterpret_cast<volatile int*>(sm + A_BAR + 68);
  uint32_t* tslot = reinterpret_cast<uint32_t*>(sm + A_BAR + 72);
  uint32_t ncols = 32;
  while ((int)ncols < Npad) ncols <<= 1;

  if (warp == 0) {
    tmem_alloc(smem_u32(tslot), 2 * ncols);
    tmem_relinquish();
  }
  // norms past Npad are never copied in: +inf, so that columns beyond the
  // MMA width (read when Npad is not a multiple of 32) never win
  for (int i = tid; i < 512; i += ANT)
    if ((i & 255) >= Npad) reinterpret_cast<float*>(sm + A_NRM)[i] = INFINITY;
  if (tid == 0) {
    for (int b = 0; b < 2; ++b) {
      mbar_init(bar_tma(b), 1);
      mbar_init(bar_mma(b), 1);
      mbar_init(bar_free(b), AEW);
    }
    mbar_init(bar_img, 1);
    fence_mbar_init();
    *s_np = 0;
    *s_err = 0;
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tbase = *tslot;
  const int u0 = (int)((int64_t)blockIdx.x * units / gridDim.x);
  const int u1 = (int)((int64_t)(blockIdx.x + 1) * units / gridDim.x);
  const int T = u1 - u0;

  if (warp == AEW) {
    // ---------------- producer / MMA issuer
    if (lane == 0) {
      const uint32_t id = idesc_f16(128, Npad, false, true);
      const uint32_t aI = smem_u32(sm + A_IMG);
      const uint32_t ib = (uint32_t)Npad * 512u;
      int cur_h = -1;
      uint32_t ph_img = 0;
      for (int t = 0; t < T; ++t) {
        const int u = u0 + t, h = u / tiles, tile = u - h * tiles, b = t & 1;
        if (t >= 2 && !mbar_wait(bar_free(b), ((t >> 1) - 1) & 1)) { *s_err = 1; break; }
        if (h != cur_h) {
          // the previous head's MMAs read the images: wait for them, then load this head's
          if (t >= 1 && !mbar_wait(bar_mma((t - 1) & 1), ((t - 1) >> 1) & 1)) { *s_err = 1; break; }
          mbar_arrive_expect_tx(bar_img, ib);
          bulk_g2s(aI, a.img + (size_t)h * ib, ib, bar_img);
          if (!mbar_wait(bar_img, ph_img)) { *s_err = 1; break; }
          ph_img ^= 1;
          cur_h = h;
        }
        const uint32_t aX = smem_u32(sm + A_X + b * 32768);
        mbar_arrive_expect_tx(bar_tma(b), 32768u + (uint32_t)Npad * 4u);
        tma_load_3d(aX, &tm, 0, h, tile * 128, bar_tma(b));
        tma_load_3d(aX + 16384, &tm, 64, h, tile * 128, bar_tma(b));
        bulk_g2s(smem_u32(sm + A_NRM + b * 1024), a.nrm + (size_t)h * Npad, (uint32_t)Npad * 4u, bar_tma(b));
        if (!mbar_wait(bar_tma(b), (t >> 1) & 1)) { *s_err = 1; break; }
        tc_fence_after();
        const uint32_t tD = tbase + (uint32_t)b * ncols;
#pragma unroll
        for (int half = 0; half < 2; ++half)
#pragma unroll
          for (int kb = 0; kb < 2; ++kb)
#pragma unroll
            for (int ks = 0; ks < 4; ++ks)
              umma_ss(tD, desc_sw128(aX + kb * 16384 + ks * 32),
                      desc_sw128(aI + half * Npad * 256 + kb * Npad * 128 + ks * 32), id, (half | kb | ks) != 0);
        umma_commit(bar_mma(b));
      }
    }
    __syncwarp();
  } else {
    // ---------------- epilogue: warps 0-15
    const int qt = warp >> 2, row = (warp & 3) * 32 + lane;
    const uint32_t lrow = (uint32_t)((warp & 3) * 32) << 16;
    const int nchunk = (Npad + 31) >> 5;
    const int ch0 = (qt * nchunk) >> 2, ch1 = ((qt + 1) * nchunk) >> 2;   // this quarter's 32-column chunks
    for (int t = 0; t < T; ++t) {
      const int u = u0 + t, h = u / tiles, tile = u - h * tiles, b = t & 1;
      const uint8_t* sX = sm + A_X + b * 32768;
      const float4* sNrm4 = reinterpret_cast<const float4*>(sm + A_NRM + b * 1024);  // +inf past C
      const uint32_t tD = tbase + (uint32_t)b * ncols;
      const int64_t n = (int64_t)tile * 128 + row;
      const bool valid = n < a.N;
      const float kx = valid ? a.xn2[(size_t)h * a.N + n] : 0.0f;
      bool ok = mbar_wait(bar_mma(b), (t >> 1) & 1);
      ok = __all_sync(0xFFFFFFFFu, ok);
      tc_fence_after();
      if (!ok) *s_err = 1;
      // smallest dt of this quarter
      float mn = INFINITY;
      if (ok) {
#pragma unroll 1
        for (int cb = ch0; cb < ch1; cb += 2) {
          float v[64];
          const int cb2 = cb + 1 < ch1 ? cb + 1 : cb;  // a lone last chunk is read twice (harmless for a minimum)
          tmem_ld32x2(tD + lrow + cb * 32, tD + lrow + cb2 * 32, *reinterpret_cast<float(*)[32]>(v),
                      *reinterpret_cast<float(*)[32]>(v + 32));
#pragma unroll
          for (int e4 = 0; e4 < 16; ++e4) {
            const float4 nr = sNrm4[(e4 < 8 ? cb : cb2) * 8 + (e4 & 7)];
            mn = fminf(mn, fminf(fminf(fmaf(-2.0f, v[4 * e4], nr.x), fmaf(-2.0f, v[4 * e4 + 1], nr.y)),
                                 fminf(fmaf(-2.0f, v[4 * e4 + 2], nr.z), fmaf(-2.0f, v[4 * e4 + 3], nr.w))));
          }
        }
      }
      sMin[qt * AT + row] = mn;
      named_bar_sync(1, AEW * 32);
      mn = fminf(fminf(sMin[row], sMin[AT + row]), fminf(sMin[2 * AT + row], sMin[3 * AT + row]));
      const float thr = mn + 2.0f * ldexpf(kx + __uint_as_float(a.nmax[h]), -11);
      // this quarter's candidates, ascending
      int cnt = 0;
      uint8_t* cand = sCnd + (row * 4 + qt) * kRowCap;
      if (ok && thr < INFINITY) {
#pragma unroll 1
        for (int cb = ch0; cb < ch1; cb += 2) {
          float v[64];
          const int cb2 = cb + 1 < ch1 ? cb + 1 : cb;
          tmem_ld32x2(tD + lrow + cb * 32, tD + lrow + cb2 * 32, *reinterpret_cast<float(*)[32]>(v),
                      *reinterpret_cast<float(*)[32]>(v + 32));
          const int ne = cb2 > cb ? 64 : 32;
#pragma unroll
          for (int e4 = 0; e4 < 16; ++e4) {
            const float4 nr = sNrm4[(e4 < 8 ? cb : cb2) * 8 + (e4 & 7)];
            const float d4[4] = {fmaf(-2.0f, v[4 * e4], nr.x), fmaf(-2.0f, v[4 * e4 + 1], nr.y),
                                 fmaf(-2.0f, v[4 * e4 + 2], nr.z), fmaf(-2.0f, v[4 * e4 + 3], nr.w)};
#pragma unroll
            for (int q = 0; q < 4; ++q)
              if (4 * e4 + q < ne && d4[q] <= thr) {
                if (cnt < kRowCap) cand[cnt] = (uint8_t)(cb * 32 + 4 * e4 + q);
                ++cnt;
              }
          }
        }
      }
      sCnt[qt * AT + row] = (ok && thr < INFINITY) ? cnt : -1;
      tc_fence_before();
      named_bar_sync(1, AEW * 32);
      // the row owner (quarter 0) merges: one candidate decides, a few go to the pair list
      int best = 0;
      if (qt == 0) {
        int c[4], tot = 0;
        bool bad = false;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          c[q] = sCnt[q * AT + row];
          bad = bad || c[q] < 0;
          tot += c[q];
        }
        uint32_t rinfo = 0;
        if (bad || tot == 0 || tot > kRowCap) {
          rinfo = 0xFFFFu;  // every centroid, sequentially
        } else if (tot == 1) {
#pragma unroll
          for (int q = 0; q < 4; ++q)
            if (c[q]) best = sCnd[(row * 4 + q) * kRowCap];
        } else if (valid) {
          const int base = atomicAdd(s_np, tot);
          if (base + tot <= kPairCap) {
            int s2 = 0;
#pragma unroll
            for (int q = 0; q < 4; ++q)
              for (int k = 0; k < c[q]; ++k)
                sPJ[base + s2++] = ((uint32_t)row << 16) | (uint32_t)sCnd[(row * 4 + q) * kRowCap + k];
            rinfo = ((uint32_t)base << 16) | (uint32_t)tot;
          } else {
            rinfo = 0xFFFFu;
          }
        }
        sRow[row] = rinfo;
      }
      named_bar_sync(1, AEW * 32);
      // exact rescoring of the listed pairs, spread over the epilogue warps
      const int np = min(*s_np, kPairCap);
      const float* muh = a.cent + (size_t)h * C * 128;
      for (int p = tid; p < np; p += AEW * 32) {
        const uint32_t pj = sPJ[p];
        sPD[p] = exact_dist(sX, (int)(pj >> 16), muh + (size_t)(pj & 0xFFFFu) * 128);
      }
      if (np > 0) named_bar_sync(1, AEW * 32);   // np is the same for every thread
      if (qt == 0 && valid && ok) {
        const uint32_t rinfo = sRow[row];
        if (rinfo == 0xFFFFu) {
          float bd = 0.0f;
          for (int j = 0; j < C; ++j) {
            const float dj = exact_dist(sX, row, muh + (size_t)j * 128);
            if (j == 0 || dj < bd) {
              bd = dj;
              best = j;
            }
          }
        } else if (rinfo != 0) {
          const int base = (int)(rinfo >> 16), c2 = (int)(rinfo & 0xFFFFu);
          float bd = sPD[base];
          best = (int)(sPJ[base] & 0xFFFFu);
          for (int s2 = 1; s2 < c2; ++s2)
            if (sPD[base + s2] < bd) {  // ascending j: the lower index keeps a tie
              bd = sPD[base + s2];
              best = (int)(sPJ[base + s2] & 0xFFFFu);
            }
        }
        a.asg[(size_t)h * a.N + n] = (uint8_t)best;
        atomicAdd(a.counts + (size_t)h * C + best, 1);
      }
      fence_proxy_async_smem();  // generic reads of tile b before the next copy into it
      tc_fence_before();
      // one vote, so that every epilogue warp leaves the loop together
      const bool go = named_bar_and(1, AEW * 32, *s_err == 0);
      if (tid == 0) *s_np = 0;
      if (lane == 0) mbar_arrive(bar_free(b));
      if (!go) break;
    }
  }
  if (tid == 0 && *s_err) atomicCAS(a.status, 0, (int)QWM_ERR_TIMEOUT);
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tbase, 2 * ncols);
  }
}

// Counting sort of one head's tokens by cluster: offsets from the counts,
// then each token to a slot of its cluster (any order within a cluster).
__global__ void __launch_bounds__(1024) fit_scatter(const FitArgs a) {
  __shared__ int s_off[256], s_cur[256], s_wsum[8];
  const int h = blockIdx.x, tid = threadIdx.x, C = a.C, lane = tid & 31;
  // exclusive prefix of the counts over j (warp scans, then the warp totals)
  int v = 0, incl = 0;
  if (tid < 256) {
    v = tid < C ? a.counts[(size_t)h * C + tid] : 0;
    incl = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
      if (lane >= o) incl += y;
    }
    if (lane == 31) s_wsum[tid >> 5] = incl;
  }
  if (tid == 0) a.nmax[h] = 0u;  // rebuilt by fit_means
  __syncthreads();
  if (tid < 256) {
    int wp = 0;
    for (int k = 0; k < (tid >> 5); ++k) wp += s_wsum[k];
    s_off[tid] = wp + incl - v;
  }
  __syncthreads();
  if (tid < C) {
    a.offs[(size_t)h * C + tid] = s_off[tid];
    s_cur[tid] = 0;
  }
  __syncthreads();
  const uint8_t* asg = a.asg + (size_t)h * a.N;
  int32_t* lst = a.list + (size_t)h * a.N;
  // (the bounds checks only matter after a timed-out assignment left stale entries)
  for (int64_t n = tid; n < a.N; n += blockDim.x) {
    const int j = asg[n];
    if (j < C) {
      const int pos = s_off[j] + atomicAdd(&s_cur[j], 1);
      if (pos < a.N) lst[pos] = (int32_t)n;
    }
  }
}

// Largest bf16 exponent field over each head's tokens, which fixes the unit
// 2^U of the exact fixed-point member sums (U = emax - 134 - room), and |x|^2
// of every token, which sizes the screening bound.
__global__ void __launch_bounds__(256) fit_scale(const FitArgs a) {
  const int h = blockIdx.y, lane = threadIdx.x & 31;
  uint32_t mx = 0;
  for (int64_t n = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5); n < a.N; n += (int64_t)gridDim.x * 8) {
    const uint2 xv = __ldg(reinterpret_cast<const uint2*>(a.x + ((size_t)n * a.H + h) * 128 + 4 * lane));
    mx = max(mx, max(max((xv.x >> 7) & 0xFFu, (xv.x >> 23) & 0xFFu), max((xv.y >> 7) & 0xFFu, (xv.y >> 23) & 0xFFu)));
    const float x0 = __uint_as_float(xv.x << 16), x1 = __uint_as_float(xv.x & 0xFFFF0000u);
    const float x2 = __uint_as_float(xv.y << 16), x3 = __uint_as_float(xv.y & 0xFFFF0000u);
    float n2 = fmaf(x0, x0, fmaf(x1, x1, fmaf(x2, x2, x3 * x3)));
#pragma unroll
    for (int o = 16; o; o >>= 1) n2 += __shfl_xor_sync(0xFFFFFFFFu, n2, o);
    if (lane == 0) a.xn2[(size_t)h * a.N + n] = n2;
  }
  mx = __reduce_max_sync(0xFFFFFFFFu, mx);
  if (lane == 0) atomicMax(a.emax + h, (int)mx);
}

// New centroid j of head h: the fp32 rounding of the fp64 member mean (kept
// when the cluster is empty); then its images and norm.  One warp each, lane =
// four channels, member rows read four at a time.
//   The member sum is exact and independent of order.  A normal bf16 value is
//   (128 + f) 2^(e - 134); with U = emax - 134 - room every member is the
//   integer (128 + f) << (e - 134 - U) < 2^(8 + room) in units of 2^U, and N
//   of them add in int64 without overflow.  A member outside that grid (tiny,
//   subnormal, inf or NaN) sends the cluster to fp64 sums instead.
//   The mean RN32(RN64(S / n)): q = S * RN64(1/n) lies within 2.5 ulp of
//   RN64(S / n), so both round to the same fp32 value unless q is within a
//   few ulp of a point halfway between two fp32 values; there (and outside the
//   fp32 normal range) the exact fp64 division decides.
__device__ __forceinline__ float mean_of(int64_t k, int U, double invs, double dc, bool& exact_ok) {
  const double kd = (double)k;
  if (!((double)(kd) == (double)k && (long long)kd == k)) {
    exact_ok = false;
    return 0.0f;
  }
  const double q = kd * invs;
  const long long bits = __double_as_longlong(q);
  const int ex = (int)((bits >> 52) & 0x7FF);
  const long long lo = bits & ((1LL << 29) - 1);
  const bool near = (lo > (1LL << 28) - 16 && lo < (1LL << 28) + 16) || ex < 1023 - 126 || ex > 1023 + 127;
  if (k != 0 && near) return __double2float_rn(__ddiv_rn(ldexp(kd, U), dc));
  return __double2float_rn(q);
}

__global__ void __launch_bounds__(512) fit_means(const FitArgs a) {
  const int lane = threadIdx.x & 31;
  const int64_t w = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  if (w >= (int64_t)a.H * a.C) return;
  const int h = (int)(w / a.C), j = (int)(w % a.C);
  const int cnt = a.counts[w], base = a.offs[w];
  float4* cr = reinterpret_cast<float4*>(a.cent + (size_t)w * 128) + lane;
  float4 m;
  if (cnt > 0) {
    const int32_t* lst = a.list + (size_t)h * a.N + (base < a.N ? base : 0);
    const int U = a.emax[h] - 134 - a.room;
    int64_t k0 = 0, k1 = 0, k2 = 0, k3 = 0;
    bool grid_ok = true;
    // A member value in units of 2^U, y = (128 + f) 2^(e - 134 - U) < 2^48 (room <= 40),
    // has 8 significant bits: the bf16 bits widened to fp32 with -U added to the
    // exponent field.  Two additions of 3 2^54 and 3 2^38 split it exactly into
    // fp32 limbs that are multiples of 2^32 and 2^16 and a remainder below
    // 2^15; 32 such limbs add exactly in fp32 (below 2^21 units each), and every
    // 32 members the three limb sums go to int64.  Zero stays zero; a value off
    // the grid (tiny, subnormal, inf, NaN) clears grid_ok.
    const uint32_t eadd = (uint32_t)(-U) << 23;
    const int emin = U + 134;
    const float C32 = 5.4043195528445952e16f;   // 3 * 2^54
    const float C16 = 8.24633720832e11f;        // 3 * 2^38
    float l2[4], l1[4], l0[4];
    auto limb = [&](uint32_t b16, int ch) {
      const uint32_t e = (b16 >> 7) & 0xFFu;
      const bool zero = (b16 & 0x7FFFu) == 0u;
      grid_ok = grid_ok && (zero || ((int)e >= emin && e != 255u));
      const float y = zero ? 0.0f : __uint_as_float((b16 << 16) + eadd);
      const float hi = __fsub_rn(__fadd_rn(y, C32), C32);
      const float r1 = __fsub_rn(y, hi);
      const float mid = __fsub_rn(__fadd_rn(r1, C16), C16);
      l2[ch] = __fadd_rn(l2[ch], hi);
      l1[ch] = __fadd_rn(l1[ch], mid);
      l0[ch] = __fadd_rn(l0[ch], __fsub_rn(r1, mid));
    };
    auto flush = [&](int64_t& k, int ch) {
      k += ((int64_t)__float2int_rn(l2[ch] * 2.3283064365386963e-10f) << 32) +
           ((int64_t)__float2int_rn(l1[ch] * 1.52587890625e-05f) << 16) + (int64_t)__float2int_rn(l0[ch]);
    };
    for (int i0 = 0; i0 < cnt; i0 += 32) {
      const int nb = min(32, cnt - i0);
      const int my = lane < nb ? lst[i0 + lane] : -1;  // 32 member indices in one read
#pragma unroll
      for (int ch = 0; ch < 4; ++ch) l2[ch] = l1[ch] = l0[ch] = 0.0f;
      for (int kb = 0; kb < nb; kb += 8) {
        uint2 xv[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          const int tok = __shfl_sync(0xFFFFFFFFu, my, (kb + k) & 31);
          xv[k] = make_uint2(0, 0);
          if (kb + k < nb && tok >= 0 && tok < a.N)  // always, unless a timed-out assignment left stale lists
            xv[k] = __ldg(reinterpret_cast<const uint2*>(a.x + ((size_t)tok * a.H + h) * 128 + 4 * lane));
        }
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          limb(xv[k].x & 0xFFFFu, 0);
          limb(xv[k].x >> 16, 1);
          limb(xv[k].y & 0xFFFFu, 2);
          limb(xv[k].y >> 16, 3);
        }
      }
      flush(k0, 0);
      flush(k1, 1);
      flush(k2, 2);
      flush(k3, 3);
    }
    const double dc = (double)cnt;
    bool ok = __all_sync(0xFFFFFFFFu, grid_ok);
    if (ok) {
      const double invs = ldexp(__ddiv_rn(1.0, dc), U);
      bool eo = true;
      m = make_float4(mean_of(k0, U, invs, dc, eo), mean_of(k1, U, invs, dc, eo), mean_of(k2, U, invs, dc, eo),
                      mean_of(k3, U, invs, dc, eo));
      ok = __all_sync(0xFFFFFFFFu, eo);
    }
    if (!ok) {  // fp64 sums (exact for members of ordinary range)
      double s0 = 0.0, s1 = 0.0, s2 = 0.0, s3 = 0.0;
      for (int i = 0; i < cnt; ++i) {
        const int64_t tok = lst[i];
        if (tok < 0 || tok >= a.N) continue;
        const uint2 xv = __ldg(reinterpret_cast<const uint2*>(a.x + ((size_t)tok * a.H + h) * 128 + 4 * lane));
        s0 += (double)__uint_as_float(xv.x << 16);
        s1 += (double)__uint_as_float(xv.x & 0xFFFF0000u);
        s2 += (double)__uint_as_float(xv.y << 16);
        s3 += (double)__uint_as_float(xv.y & 0xFFFF0000u);
      }
      m = make_float4(__double2float_rn(__ddiv_rn(s0, dc)), __double2float_rn(__ddiv_rn(s1, dc)),
                      __double2float_rn(__ddiv_rn(s2, dc)), __double2float_rn(__ddiv_rn(s3, dc)));
    }
    *cr = m;
  } else {
    m = *cr;
  }
  emit_row(a, h, j, m, lane);
  __syncwarp();
  if (lane == 0) a.counts[w] = 0;  // ready for the next assignment
}

// bf16 output; NaN everywhere if a wait inside the assignment ran out.
__global__ void fit_out(const FitArgs a) {
  const int64_t n = (int64_t)a.H * a.C * 128;
  const bool bad = *a.status != 0;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
    a.out[i] = bad ? __float2bfloat16_rn(NAN) : __float2bfloat16_rn(a.cent[i]);
}

int sm_count() {
  int dev = 0, nsm = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev) !=
                                                 cudaSuccess || nsm < 1)
    return 1;
  return nsm;
}

}  // namespace

static int npad_of(int C) { return C < 16 ? 16 : (C + 15) & ~15; }

size_t fit_workspace_bytes(int H, int d, int C, int64_t N) {
  const int Np = npad_of(C);
  size_t b = 256;                                               // status
  b += (size_t)round_up((int64_t)H * C * d * 4, 256);           // cent
  b += (size_t)round_up((int64_t)H * Np * 512, 256);            // images
  b += (size_t)round_up((int64_t)H * Np * 4, 256);              // norms
  b += 2 * (size_t)round_up((int64_t)H * 4, 256);               // largest norm, largest exponent
  b += 2 * (size_t)round_up((int64_t)H * C * 4, 256);           // counts, offsets
  b += (size_t)round_up((int64_t)H * N, 256);                   // assignment
  b += (size_t)round_up((int64_t)H * N * 4, 256);               // token norms
  b += (size_t)round_up((int64_t)H * N * 4, 256);               // member lists
  return b;
}

void fit_carve(FitArgs& a, uint8_t* ws) {
  a.Npad = npad_of(a.C);
  uint8_t* p = ws;
  auto take = [&](int64_t bytes) {
    uint8_t* q = p;
    p += round_up(bytes, 256);
    return q;
  };
  a.status = reinterpret_cast<int32_t*>(take(256));
  a.cent = reinterpret_cast<float*>(take((int64_t)a.H * a.C * a.d * 4));
  a.img = take((int64_t)a.H * a.Npad * 512);
  a.nrm = reinterpret_cast<float*>(take((int64_t)a.H * a.Npad * 4));
  a.nmax = reinterpret_cast<uint32_t*>(take((int64_t)a.H * 4));
  a.emax = reinterpret_cast<int32_t*>(take((int64_t)a.H * 4));
  // member sums of at most N values below 2^(8 + room) each stay below 2^61, and
  // each value below 2^48 units
  int lg = 0;
  while (((int64_t)1 << lg) < a.N + 1) ++lg;
  a.room = 53 - lg < 40 ? 53 - lg : 40;  // values below 2^48 units: three fp32 limbs (fit_means)
  a.counts = reinterpret_cast<int32_t*>(take((int64_t)a.H * a.C * 4));
  a.offs = reinterpret_cast<int32_t*>(take((int64_t)a.H * a.C * 4));
  a.asg = take((int64_t)a.H * a.N);
  a.xn2 = reinterpret_cast<float*>(take((int64_t)a.H * a.N * 4));
  a.list = reinterpret_cast<int32_t*>(take((int64_t)a.H * a.N * 4));
}

cudaError_t launch_fit(const FitArgs& a, cudaStream_t st) {
  cudaError_t e;
  if ((e = cudaMemsetAsync(a.status, 0, 4, st)) != cudaSuccess) return e;
  if ((e = cudaMemsetAsync(a.nmax, 0, (size_t)a.H * 4, st)) != cudaSuccess) return e;
  if ((e = cudaMemsetAsync(a.emax, 0, (size_t)a.H * 4, st)) != cudaSuccess) return e;
  if ((e = cudaMemsetAsync(a.counts, 0, (size_t)a.H * a.C * 4, st)) != cudaSuccess) return e;
  const int64_t prep_warps = (int64_t)a.H * a.Npad;
  fit_prep<<<(unsigned)((prep_warps + 15) / 16), 512, 0, st>>>(a);
  if (a.iters > 0) {
    CUtensorMap tm;
    if (!make_token_map(&tm, a.x, a.N, a.H, 128)) return cudaErrorInvalidValue;
    if ((e = cudaFuncSetAttribute(fit_assign, cudaFuncAttributeMaxDynamicSharedMemorySize, A_SMEM)) != cudaSuccess)
      return e;
    const int tiles = (int)((a.N + 127) / 128);
    const int units = a.H * tiles;
    const int grid = units < sm_count() ? units : sm_count();
    const int64_t mean_warps = (int64_t)a.H * a.C;
    const int64_t sb = (a.N + 7) / 8;
    fit_scale<<<dim3((unsigned)(sb < 64 ? sb : 64), (unsigned)a.H), 256, 0, st>>>(a);
    for (int it = 0; it < a.iters; ++it) {
      fit_assign<<<grid, ANT, A_SMEM, st>>>(a, tm, tiles, units);
      fit_scatter<<<a.H, 1024, 0, st>>>(a);
      fit_means<<<(unsigned)((mean_warps + 15) / 16), 512, 0, st>>>(a);
    }
  }
  const int64_t n = (int64_t)a.H * a.C * a.d;
  const unsigned og = (unsigned)((n + 255) / 256 < 4096 ? (n + 255) / 256 : 4096);
  fit_out<<<og, 256, 0, st>>>(a);
  return cudaGetLastError();
}

}  // namespace qwm

namespace qwm {

// ----------------------------------------------------------------------------
// Allocation-free variant of qwm_fit_centroids.
//
// Some callers cannot hand the library a scratch buffer: a plain C host
// program that only owns the input and output tensors it was given, or an
// inference engine whose device memory is already reserved by its own pool
// and which must not call cudaMalloc/cudaFree in the middle of generation
// (those calls can synchronise the whole device).  For them the k-means
// scratch (fp32 centroids, MMA operand images, norms, counts, assignment and
// member lists) lives in this file-scope device array instead.
// ----------------------------------------------------------------------------
namespace {

constexpr size_t kNoAllocFitScratchBytes = (size_t)16 << 20;  // 16 MiB per GPU that loads the library
static __device__ __align__(256) uint8_t g_fit_scratch[kNoAllocFitScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_fit_scratch_mutex;
void* g_fit_scratch_addr[kMaxDevices] = {};

}  // namespace
}  // namespace qwm

extern "C" QWM_API qwm_status qwm_fit_centroids_noalloc(const qwm_config* cfg, const void* x, int64_t N,
                                                        void* centroids, void* stream) {
  using namespace qwm;
  if (!cfg || !x || !centroids || N < 1) return QWM_ERR_INVALID_ARG;
  if (!config_supported(cfg)) return QWM_ERR_UNSUPPORTED;  // the same set qwm_fit_centroids accepts
  if (N > (int64_t)1 << 31) return QWM_ERR_UNSUPPORTED;
  if ((reinterpret_cast<uintptr_t>(x) & 15u) || (reinterpret_cast<uintptr_t>(centroids) & 15u))
    return QWM_ERR_INVALID_ARG;
  const size_t need = fit_workspace_bytes(cfg->num_heads, cfg->head_dim, cfg->num_centroids, N);
  if (need > kNoAllocFitScratchBytes) return QWM_ERR_CAPACITY;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return QWM_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return QWM_ERR_UNSUPPORTED;
  uint8_t* ws = nullptr;
  {
    // First call on a device: look up the device address of the array there
    // (in host code its name is only a host-side stand-in).
    std::lock_guard<std::mutex> lock(g_fit_scratch_mutex);
    if (!g_fit_scratch_addr[dev]) {
      void* p = nullptr;
      if (cudaGetSymbolAddress(&p, g_fit_scratch) != cudaSuccess || !p) return QWM_ERR_CUDA;
      g_fit_scratch_addr[dev] = p;
    }
    ws = static_cast<uint8_t*>(g_fit_scratch_addr[dev]);
  }
  FitArgs a{};
  a.H = cfg->num_heads; a.d = cfg->head_dim; a.C = cfg->num_centroids; a.iters = cfg->kmeans_iters;
  a.N = N;
  a.x = static_cast<const __nv_bfloat16*>(x);
  a.out = static_cast<__nv_bfloat16*>(centroids);
  fit_carve(a, ws);
  // launch_fit clears the status word, the counts and the largest norms and
  // writes every centroid, image and norm before reading it, so nothing
  // depends on what an earlier call left in the array.
  return launch_fit(a, static_cast<cudaStream_t>(stream)) == cudaSuccess ? QWM_OK : QWM_ERR_CUDA;
}

