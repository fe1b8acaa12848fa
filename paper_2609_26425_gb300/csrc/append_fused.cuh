// append_fused.cuh -- quantize-on-append in one persistent kernel: each
// 128-token tile of one (head, K/V side) is read from HBM once, screened for
// its top-M QSAC candidates on the tensor cores, and quantised from registers.
//
// A CTA (one per SM) holds the run's centroid table mu [C][128] (bf16, the
// 128-byte swizzled MMA operand layout, loaded by TMA once per (head, side))
// and two groups of 128 threads; a group owns one tile at a time, thread =
// token row, and the groups alternate over the CTA's contiguous run of tiles.
// Per tile of a group:
//   1. the bf16 rows arrive by TMA; each thread loads its row into registers;
//      for Keys with sensitivity weights the row becomes the MMA operand
//      a = w o k, split into two bf16 parts (a_hi in place, a_lo beside it:
//      a_hi + a_lo carries the fp32 product to 2^-17), so that
//      D = a mu^T = sum_c w_c k_c mu_jc and the Query-aware distance
//      (Sec. 4.1, Eq. 9) expands as dQ_j = sum_c w_c k_c^2 - 2 D_j + A_j with
//      A_j = sum_c w_c mu_jc^2; Values and unweighted Keys use the bf16 row
//      itself (exact, one MMA);
//   2. tcgen05 MMAs (bf16, fp32 accumulation, 128 x C) write D into the
//      group's TMEM columns; the tile buffer is then free and the copy of the
//      group's next tile is issued;
//   3. each thread keeps the M+1 smallest dt_j = A_j - 2 D_j of its row.
//      With the error bound B of dt against the oracle's sequential fp32
//      distance (less their common term), every centroid of the exact top-M
//      lies within 2B of the M-th smallest dt: when the (M+1)-th lies beyond
//      that band the top-M is decided, otherwise the band members are
//      rescored exactly: their rows are parked in shared memory and the
//      group evaluates the (row, centroid) pairs together with the oracle's
//      sequential fp32 distance;
//   4. QSAC (Eq. 10, 12) over the M candidates, the INT2 residual
//      quantisation with packing (Eq. 1-2) and, for Keys, the PSAC
//      projection c = U_r^T E with its INT8 codes and keep rule (Eq. 13, 16),
//      all in fp32 with every rounding explicit (one fused multiply-add per
//      term of a sum of products, channel order), from the register row and
//      the shared-memory table; the packed record is stored, the tile's PSAC
//      rows in the smaller of the dense and sparse layouts (App. D.1).
// The selection of the full quadratic form (App. C.4) and the exhaustive
// range 8 < M < C use the other append kernels.
#pragma once
#include "ptx_sm103.cuh"
#include "qwm_internal.cuh"
#include "append_common.cuh"

namespace qwm {
namespace {

using namespace ptx;

constexpr int XG = 2;               // token groups per CTA
constexpr int XNT = XG * 128;
constexpr int kXRsCap = 512;        // (row, centroid) pairs rescored together per group and tile

template <int R>
struct XSmem {
  static constexpr int MU = 0;                                  // [2][256 rows][128 B] bf16, swizzled
  static constexpr int BUF = 65536;                             // [XG] token tiles [2][128][128 B]
  static constexpr int LO = BUF + XG * 32768;                   // [XG] a_lo tiles; then the rows (256 B each)
  static constexpr int U = LO + XG * 32768;                     // U [128][R] fp32
  static constexpr int G = U + (R > 0 ? 128 * R * 4 : 0);       // U^T W U [R][R] fp32
  static constexpr int W = G + (R > 0 ? R * R * 4 : 0);         // w [128] fp32
  static constexpr int AJ = W + 512;                            // A_j [256] fp32
  static constexpr int MISC = AJ + 1024;                        // 64 floats (see the kernel)
  static constexpr int RSP = MISC + 256;                        // [XG][kXRsCap] (row, centroid) u16
  static constexpr int RSD = RSP + XG * kXRsCap * 2;            // [XG][kXRsCap] their distances
  static constexpr int CNT = RSD + XG * kXRsCap * 4;            // [XG][8] ints
  static constexpr int BAR = CNT + XG * 32;                     // mbarriers, flags, TMEM slot
  static constexpr int BYTES = BAR + 64 + 1024;
};
static_assert(XSmem<32>::BYTES <= 232448, "shared memory of the fused append kernel");

// A token row parked in shared memory: 256 bytes, its 16-byte chunk ch (bf16
// channels 8 ch .. 8 ch + 7) at position ch ^ (row % 16), so that a warp's
// rows spread over the banks.
__device__ __forceinline__ uint4 row_chunk(const uint8_t* rowp, int key, int ch) {
  return lds16(rowp + ((ch ^ key) << 4));
}

// The Query-aware distance of the oracle (Eq. 9): sum over c in channel order
// of w_c (k_c - mu_c)^2, the difference and its square each rounded, one fused
// multiply-add per term.  Row from its shared-memory copy (row index r),
// centroid row j from the swizzled table.
__device__ __forceinline__ float dq_smem(const uint8_t* rows, int r, const uint8_t* mu, int Npad, int j,
                                         const float* sW) {
  const uint8_t* rowp = rows + r * 256;
  const int key = r & 15;
  float acc = 0.0f;
#pragma unroll 2
  for (int cc = 0; cc < 8; ++cc) {
    const uint4 ka = row_chunk(rowp, key, 2 * cc), kb = row_chunk(rowp, key, 2 * cc + 1);
    const uint4 ma = lds16(mu + sw_off(Npad, j, 2 * cc)), mb = lds16(mu + sw_off(Npad, j, 2 * cc + 1));
    const uint32_t kw[8] = {ka.x, ka.y, ka.z, ka.w, kb.x, kb.y, kb.z, kb.w};
    const uint32_t mw[8] = {ma.x, ma.y, ma.z, ma.w, mb.x, mb.y, mb.z, mb.w};
#pragma unroll
    for (int p = 0; p < 8; ++p) {
      uint64_t t2 = sub2(bf2_to_f2(kw[p]), bf2_to_f2(mw[p]));
      t2 = mul2(t2, t2);
      float lo, hi;
      f2unpack(t2, lo, hi);
      acc = __fmaf_rn(sW[cc * 16 + 2 * p], lo, acc);
      acc = __fmaf_rn(sW[cc * 16 + 2 * p + 1], hi, acc);
    }
  }
  return acc;
}

// CAPT = M + 1 (the ranked list of a row; kMaxFilterM + 1 for the candidate
// counts without their own instance), R = PSAC rank.
template <int CAPT, int R>
__global__ void __launch_bounds__(XNT, 1)
    append_fused(const AppendArgs a, const __grid_constant__ CUtensorMap tm_k,
                 const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ CUtensorMap tm_kc,
                 const __grid_constant__ CUtensorMap tm_vc, int tiles, int units) {
  using S = XSmem<R>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  const Layout& L = a.L;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = tid >> 7, row = tid & 127, gw = warp & 3;
  const int C = L.C, H = L.H, Mc = a.M;
  const bool all_cand = Mc >= C;
  const int Npad = (C + 15) & ~15;
  const int GS = L.G, ng = 128 / GS;
  const bool gs32 = GS == 32;
  constexpr int RP = R > 0 ? R / 2 : 1;

  uint8_t* sMU = sm + S::MU;
  uint8_t* sBuf = sm + S::BUF + g * 32768;
  uint8_t* sLo = sm + S::LO + g * 32768;
  float* sU = reinterpret_cast<float*>(sm + S::U);
  float* sG = reinterpret_cast<float*>(sm + S::G);
  float* sW = reinterpret_cast<float*>(sm + S::W);
  float* sAj = reinterpret_cast<float*>(sm + S::AJ);
  // sMisc: [0, 4) W_g; [8, 12) |U|_F^2 and [12, 16) max w of warps 0-3;
  // [16, 24) max |mu_j|^2 and [24, 32) max A_j of each warp
  float* sMisc = reinterpret_cast<float*>(sm + S::MISC);
  uint16_t* sRsPair = reinterpret_cast<uint16_t*>(sm + S::RSP) + g * kXRsCap;
  float* sRsDq = reinterpret_cast<float*>(sm + S::RSD) + g * kXRsCap;
  // sCnt: [0] pairs reserved, [2] end of the listed pairs,
  // [4, 8) the tile's PSAC keep bits per warp
  int* sCnt = reinterpret_cast<int*>(sm + S::CNT) + g * 8;
  volatile int* sFlag = reinterpret_cast<volatile int*>(sm + S::BAR + 48);  // [XG] a wait of the group ran out
  uint32_t* tslot = reinterpret_cast<uint32_t*>(sm + S::BAR + 56);
  const uint32_t bar_tma = smem_u32(sm + S::BAR + 8 * g);
  const uint32_t bar_mma = smem_u32(sm + S::BAR + 16 + 8 * g);
  const uint32_t bar_mu = smem_u32(sm + S::BAR + 32);

  if (warp == 0) {
    tmem_alloc(smem_u32(tslot), 512);
    tmem_relinquish();
  }
  if (tid == 0) {
    for (int i = 0; i < 5; ++i) mbar_init(smem_u32(sm + S::BAR + 8 * i), 1);
    fence_mbar_init();
    sFlag[0] = sFlag[1] = 0;
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tbase = *tslot;
  const uint32_t tD = tbase + (uint32_t)(g * 256);
  const uint32_t lrow = (uint32_t)(gw * 32) << 16;

  // Work unit u = (side * H + h) * tiles + tile; this CTA takes [u0, u1), a
  // run per (head, side); group g takes the units u0 + g, u0 + g + 2, ...
  const int nb = gridDim.x;
  const int u0 = (int)((int64_t)blockIdx.x * units / nb);
  const int u1 = (int)((int64_t)(blockIdx.x + 1) * units / nb);
  auto issue_tile = [&](int u) {
    const int pr = u / tiles, tl = u - pr * tiles;
    const CUtensorMap* tm = pr < H ? &tm_k : &tm_v;
    mbar_arrive_expect_tx(bar_tma, 32768);
    tma_load_3d(smem_u32(sBuf), tm, 0, pr % H, tl * 128, bar_tma);
    tma_load_3d(smem_u32(sBuf + 16384), tm, 64, pr % H, tl * 128, bar_tma);
  };
  bool tma_pending = false, mma_pending = false;  // row 0 of the group: an issued copy / MMA not yet waited for
  if (row == 0 && u0 + g < u1) {
    issue_tile(u0 + g);
    tma_pending = true;
  }
  uint32_t ph_tma = 0, ph_mma = 0, ph_mu = 0;
  // A Key or Value or a table value beyond the binary16 range (or not a
  // number) cannot be held by the cache's binary16 operands: reported in the
  // cache's status word as QWM_ERR_NONFINITE once this CTA is done.
  bool nbad = false;
  bool stop = false;

  for (int s0 = u0; s0 < u1;) {
    const int pair = s0 / tiles;
    const int s1 = min(u1, (pair + 1) * tiles);
    const bool is_key = pair < H;
    const int h = pair % H;
    const bool use_w = is_key && a.w != nullptr;
    const bool psac = R > 0 && is_key && a.U != nullptr;
    const __nv_bfloat16* tab = (is_key ? a.kc : a.vc) + (size_t)h * C * 128;
    uint8_t* head = a.base + head_offset(L, a.slot, h);

    // ---- run setup: the table by TMA; w, U (fp32), U^T W U, W_g, A_j
    __syncthreads();  // the previous run's readers of the table and the per-run arrays are done
    if (sFlag[0] | sFlag[1]) {
      stop = true;
      break;
    }
    if (tid == 0) {
      const CUtensorMap* tmc = is_key ? &tm_kc : &tm_vc;
      mbar_arrive_expect_tx(bar_mu, (uint32_t)(2 * Npad * 128));
      tma_load_3d(smem_u32(sMU), tmc, 0, 0, h, bar_mu);
      tma_load_3d(smem_u32(sMU + Npad * 128), tmc, 64, 0, h, bar_mu);
    }
    if (tid < 128) sW[tid] = use_w ? a.w[(size_t)h * 128 + tid] : 1.0f;
    if constexpr (R > 0) {
      if (psac) {
        const __nv_bfloat16* Uh = a.U + (size_t)h * 128 * R;
        for (int i = tid; i < 128 * R; i += XNT) sU[i] = __bfloat162float(Uh[i]);  // [d][r]
      }
    }
    // The chunk's own tables travel with the slot, stored as binary16 (exact
    // for bf16 values in the binary16 range), the operand type of the
    // attention kernel's tensor-core path; the run holding tile 0 writes them.
    if (s0 == pair * tiles) {
      const uint32_t* src = reinterpret_cast<const uint32_t*>(tab);
      __half2* dst = reinterpret_cast<__half2*>(head + (is_key ? L.ktab : L.vtab));
      for (int i = tid; i < C * 64; i += XNT) {
        const uint32_t pr = src[i];
        nbad |= bf16x2_out_of_f16(pr);
        dst[i] = __floats2half2_rn(__uint_as_float(pr << 16), __uint_as_float(pr & 0xFFFF0000u));
      }
      if (psac) {
        __nv_bfloat16* ut = reinterpret_cast<__nv_bfloat16*>(head + L.ut);
        const __nv_bfloat16* Uh = a.U + (size_t)h * 128 * R;
        for (int i = tid; i < R * 128; i += XNT) ut[i] = Uh[(size_t)(i % 128) * R + i / 128];  // U_r^T [r][d]
      }
    }
    const bool mu_ok = mbar_wait(bar_mu, ph_mu);
    ph_mu ^= 1;
    if (__syncthreads_or(!mu_ok)) {
      stop = true;
      break;
    }
    {
      // A_j = sum_c w_c mu_jc^2 (fp32; it enters the selection with its
      // error bound) and |mu_j|^2, thread j
      const int j = tid;
      float A = INFINITY, m2 = 0.0f;
      if (j < C) {
        A = 0.0f;
#pragma unroll 4
        for (int ch = 0; ch < 16; ++ch) {
          const uint4 m = lds16(sMU + sw_off(Npad, j, ch));
          const uint32_t mw[4] = {m.x, m.y, m.z, m.w};
#pragma unroll
          for (int p = 0; p < 4; ++p) {
            const float m0 = __uint_as_float(mw[p] << 16), m1 = __uint_as_float(mw[p] & 0xFFFF0000u);
            A = fmaf(__fmul_rn(sW[ch * 8 + 2 * p], m0), m0, fmaf(__fmul_rn(sW[ch * 8 + 2 * p + 1], m1), m1, A));
            m2 = fmaf(m0, m0, fmaf(m1, m1, m2));
          }
        }
      }
      sAj[j] = A;  // j in [C, 256): never selected
      float am = j < C ? A : 0.0f;
#pragma unroll
      for (int off = 16; off; off >>= 1) {
        m2 = fmaxf(m2, __shfl_xor_sync(0xFFFFFFFFu, m2, off));
        am = fmaxf(am, __shfl_xor_sync(0xFFFFFFFFu, am, off));
      }
      if (lane == 0) {
        sMisc[16 + warp] = m2;
        sMisc[24 + warp] = am;
      }
    }
    if (tid < ng) {
      float Wg = 0.0f;
      for (int c = tid * GS; c < (tid + 1) * GS; ++c) Wg = __fadd_rn(Wg, sW[c]);
      sMisc[tid] = Wg;
    }
    if constexpr (R > 0) {
      if (psac) {
        // U^T W U (any order; it enters only with its error bound): thread
        // (j, k pair) accumulates two entries over the channels
        for (int e = tid; e < R * RP; e += XNT) {
          const int j = e / RP, kp = e % RP;
          uint64_t acc = 0;
          for (int c = 0; c < 128; ++c) {
            const float uw = sU[c * R + j] * sW[c];
            acc = fma2(f2pack(uw, uw), *reinterpret_cast<const uint64_t*>(sU + c * R + 2 * kp), acc);
          }
          *reinterpret_cast<uint64_t*>(sG + j * R + 2 * kp) = acc;
        }
        if (tid < 128) {
          float u2 = 0.0f;
#pragma unroll
          for (int j = 0; j < R; ++j) u2 = fmaf(sU[tid * R + j], sU[tid * R + j], u2);
          float wm = sW[tid];
#pragma unroll
          for (int off = 16; off; off >>= 1) {
            u2 += __shfl_xor_sync(0xFFFFFFFFu, u2, off);
            wm = fmaxf(wm, __shfl_xor_sync(0xFFFFFFFFu, wm, off));
          }
          if (lane == 0) {
            sMisc[8 + warp] = u2;
            sMisc[12 + warp] = wm;
          }
        }
      }
    }
    __syncthreads();
    float Mu2 = 0.0f, Am = 0.0f;
#pragma unroll
    for (int i = 0; i < XNT / 32; ++i) {
      Mu2 = fmaxf(Mu2, sMisc[16 + i]);
      Am = fmaxf(Am, sMisc[24 + i]);
    }
    const float Mn = sqrtf(Mu2) * 1.0001f;
    float Wg[4];
#pragma unroll
    for (int gi = 0; gi < 4; ++gi) Wg[gi] = gi < ng ? sMisc[gi] : 0.0f;

    // ---- this group's tiles of the run
    for (int u = s0 + ((((s0 - u0) & 1) != g) ? 1 : 0); u < s1; u += 2) {
      const int tile = u - pair * tiles;
      const int64_t t = (int64_t)tile * 128 + row;
      const bool valid = t < a.N;
      uint8_t* tb = head + L.tiles_off + (int64_t)tile * L.tile_bytes;
      if (row == 0) {
        sCnt[0] = 0;
        sCnt[2] = 0;
      }
      const bool tok = mbar_wait(bar_tma, ph_tma);
      ph_tma ^= 1;
      if (row == 0) tma_pending = false;

      // ---- 1. the row into registers; the MMA operand
      uint32_t kr[64];
#pragma unroll
      for (int ch = 0; ch < 16; ++ch) {
        const uint4 v = lds16(sBuf + sw_off(128, row, ch));
        kr[4 * ch] = v.x; kr[4 * ch + 1] = v.y; kr[4 * ch + 2] = v.z; kr[4 * ch + 3] = v.w;
      }
      float an2 = 0.0f, K0 = 0.0f;  // |w o k|^2 and sum_c w_c k_c^2 (fp32, any order: bound terms)
      if (!all_cand) {
        if (use_w) {
          uint64_t an2p = 0, K0p = 0;
#pragma unroll
          for (int ch = 0; ch < 16; ++ch) {
            const float4 wa = *reinterpret_cast<const float4*>(sW + ch * 8);
            const float4 wb = *reinterpret_cast<const float4*>(sW + ch * 8 + 4);
            const float wv[8] = {wa.x, wa.y, wa.z, wa.w, wb.x, wb.y, wb.z, wb.w};
            uint32_t hw[4], lw[4];
#pragma unroll
            for (int p = 0; p < 4; ++p) {
              const uint64_t k2 = bf2_to_f2(kr[4 * ch + p]);
              const uint64_t a2 = mul2(f2pack(wv[2 * p], wv[2 * p + 1]), k2);
              an2p = fma2(a2, a2, an2p);
              K0p = fma2(a2, k2, K0p);
              float a0, a1;
              f2unpack(a2, a0, a1);
              hw[p] = pack_bf16(a0, a1);
              float d0, d1;
              f2unpack(sub2(a2, bf2_to_f2(hw[p])), d0, d1);
              lw[p] = pack_bf16(d0, d1);
            }
            const int off = sw_off(128, row, ch);
            *reinterpret_cast<uint4*>(sBuf + off) = make_uint4(hw[0], hw[1], hw[2], hw[3]);
            *reinterpret_cast<uint4*>(sLo + off) = make_uint4(lw[0], lw[1], lw[2], lw[3]);
          }
          float x0, x1;
          f2unpack(an2p, x0, x1);
          an2 = x0 + x1;
          f2unpack(K0p, x0, x1);
          K0 = x0 + x1;
        } else {
          uint64_t p2 = 0;
#pragma unroll
          for (int i = 0; i < 64; ++i) {
            const uint64_t k2 = bf2_to_f2(kr[i]);
            p2 = fma2(k2, k2, p2);
          }
          float x0, x1;
          f2unpack(p2, x0, x1);
          an2 = x0 + x1;
          K0 = an2;
        }
      }
      fence_proxy_async_smem();
      tc_fence_before();
      const bool gok = named_bar_and(1 + g, 128, tok);
      tc_fence_after();
      if (!gok) {
        if (row == 0) sFlag[g] = 1;
        break;
      }

      // ---- 2. D = a mu^T on the tensor cores
      if (!all_cand) {
        if (row == 0) {
          const uint32_t id = idesc_f16(128, Npad, false, true);
          const uint32_t aB = smem_u32(sMU);
          const int parts = use_w ? 2 : 1;
          for (int part = 0; part < parts; ++part) {
            const uint32_t aA = smem_u32(part ? sLo : sBuf);
#pragma unroll
            for (int kb = 0; kb < 2; ++kb)
#pragma unroll
              for (int ks = 0; ks < 4; ++ks)
                umma_ss(tD, desc_sw128(aA + kb * 16384 + ks * 32), desc_sw128(aB + kb * Npad * 128 + ks * 32), id,
                        (part | kb | ks) != 0);
          }
          umma_commit(bar_mma);
          mma_pending = true;
        }
        const bool mok = mbar_wait(bar_mma, ph_mma);
        ph_mma ^= 1;
        tc_fence_after();
        if (!named_bar_and(1 + g, 128, mok)) {
          if (row == 0) sFlag[g] = 1;
          break;
        }
        if (row == 0) mma_pending = false;
      }
      // The MMA has read both operand buffers: the row goes to its 256 bytes of
      // the a_lo buffer for the rest of the tile (any thread of the group can
      // read any row there), and the tile buffer holds the selection scratch
      // until the group's next tile is copied into it.
      uint8_t* myrow = sLo + row * 256;
      const int rkey = row & 15;
#pragma unroll
      for (int ch = 0; ch < 16; ++ch)
        *reinterpret_cast<uint4*>(myrow + ((ch ^ rkey) << 4)) =
            make_uint4(kr[4 * ch], kr[4 * ch + 1], kr[4 * ch + 2], kr[4 * ch + 3]);

      // ---- 3. selection over dt_j = A_j - 2 D_j (the TMEM reads are
      // warp-collective, every other step is per row).
      //   a. the minima of 16 interleaved column groups (column j in group
      //      j % 16); their (M+1)-th smallest, T, bounds the (M+1)-th
      //      smallest dt from above;
      //   b. a second pass marks the columns with dt <= T in a bit mask per
      //      32 columns (usually a handful per row); only those are ranked
      //      (the M+1 smallest, ties to the lower j) and listed, in ascending
      //      j, in this row's 256 bytes of the consumed tile buffer, with the
      //      values of a 32-column block stashed there when the block has one.
      // The row's record (count byte + up to 16 centroid ids) is then left
      // in the first 32 of those bytes.
      uint8_t* rowbuf = sBuf + row * 256;
      uint32_t rec[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) rec[i] = 0;
      if (!all_cand) {
        uint8_t* myl = rowbuf;
        constexpr int kList = 16;
        const int npair = (Npad + 63) >> 6;  // pairs of 32-column blocks (at most 256 columns)
        // dt of 32 consecutive columns from their D values, two at a time with
        // packed fused multiply-adds (each lane rounds once, as fmaf(-2, D, A))
        auto dt32 = [&](int cb, float (&v)[32]) {
          const float4* aj4 = reinterpret_cast<const float4*>(sAj + cb * 32);
          const uint64_t M2 = f2pack(-2.0f, -2.0f);
#pragma unroll
          for (int e = 0; e < 32; e += 4) {
            const float4 A4 = aj4[e >> 2];
            const uint64_t r0 = fma2(f2pack(v[e], v[e + 1]), M2, f2pack(A4.x, A4.y));
            const uint64_t r1 = fma2(f2pack(v[e + 2], v[e + 3]), M2, f2pack(A4.z, A4.w));
            f2unpack(r0, v[e], v[e + 1]);
            f2unpack(r1, v[e + 2], v[e + 3]);
          }
        };
        float gm[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) gm[i] = INFINITY;
#pragma unroll 1
        for (int cp = 0; cp < npair; ++cp) {
          float va[32], vb[32];
          __syncwarp();
          tmem_ld32x2(tD + lrow + cp * 64, tD + lrow + cp * 64 + 32, va, vb);
          dt32(2 * cp, va);
          dt32(2 * cp + 1, vb);
#pragma unroll
          for (int e = 0; e < 16; ++e) gm[e] = fmin3(fmin3(gm[e], va[e], va[e + 16]), vb[e], vb[e + 16]);
        }
        float tq[CAPT];
#pragma unroll
        for (int i = 0; i < CAPT; ++i) tq[i] = INFINITY;
#pragma unroll
        for (int gi = 0; gi < 16; ++gi) {  // sorted insertion, every slot from the old values
          const float x = gm[gi];
#pragma unroll
          for (int i = CAPT - 1; i > 0; --i) tq[i] = fmaxf(tq[i - 1], fminf(tq[i], x));
          tq[0] = fminf(tq[0], x);
        }
        const float T = sel_at(tq, Mc);
        // The band of step c (every j with dt_j <= kth + 2 B) lies at or below
        // T2 = T + 2 Bmax: kth (the M-th smallest dt) is at most T and at least
        // the smallest dt, tq[0], so the bound B below is at most Bmax.  The
        // second pass lists every column at or below T2, which holds the M + 1
        // smallest and the whole band.
        const float an = sqrtf(an2) * 1.0001f;
        const float Bmax = ldexpf(an * Mn, -13) * 1.25f +
                           ldexpf(Am + fabsf(K0) + fmaxf(fabsf(tq[0]), fabsf(T)), -16) + 1e-30f;
        const float T2 = T + 2.0f * Bmax;

        float* stash = reinterpret_cast<float*>(rowbuf);
        uint2* lst = reinterpret_cast<uint2*>(rowbuf + 128);
        const int sw = row & 7;
        float tv[CAPT];
        int tj[CAPT];
#pragma unroll
        for (int i = 0; i < CAPT; ++i) { tv[i] = INFINITY; tj[i] = 0x7FFFFFFF; }
        int cnt = 0;
#pragma unroll 1
        for (int cp = 0; cp < npair; ++cp) {
          float va[32], vb[32];
          __syncwarp();
          tmem_ld32x2(tD + lrow + cp * 64, tD + lrow + cp * 64 + 32, va, vb);
          dt32(2 * cp, va);
          dt32(2 * cp + 1, vb);
#pragma unroll
          for (int hb = 0; hb < 2; ++hb) {
            const float (&v)[32] = hb ? vb : va;
            const int cb = 2 * cp + hb;
            uint32_t m8[4] = {0u, 0u, 0u, 0u};  // four independent partial masks
#pragma unroll
            for (int e = 0; e < 32; ++e) m8[e & 3] |= (v[e] <= T2 ? 1u : 0u) << e;
            uint32_t mk = (m8[0] | m8[1]) | (m8[2] | m8[3]);
            if (mk) {
#pragma unroll
              for (int k4 = 0; k4 < 8; ++k4)
                reinterpret_cast<float4*>(stash)[k4 ^ sw] = make_float4(v[4 * k4], v[4 * k4 + 1], v[4 * k4 + 2], v[4 * k4 + 3]);
              do {
                const int e = __ffs(mk) - 1;
                mk &= mk - 1;
                const float x = stash[(((e >> 2) ^ sw) << 2) | (e & 3)];
                const int j = cb * 32 + e;
                if (cnt < kList) lst[cnt] = make_uint2(__float_as_uint(x), (uint32_t)j);
                ++cnt;
                insert_top(tv, tj, Mc + 1, x, j);
              } while (mk);
            }
          }
        }
        const int mc = cnt < kList ? cnt : kList;

        const float kth = sel_at(tv, Mc - 1), nxt = sel_at(tv, Mc);
        // |our dt_j - the oracle's d_j + common term| <= Bb for every
        // candidate.  The tensor cores' fp32 accumulation is taken to move the
        // sum by at most two ulps of its running absolute value per product
        // added (at most 256 exact products: 2^-14 sum_c |a_c mu_jc| <=
        // 2^-14 |a| |mu_j| by Cauchy-Schwarz, twice that in dt = A - 2 D); the
        // fp32 product a = w o k and its bf16 split add 2^-17 |a| |mu_j| (the
        // factor 1.25 holds both); the fp32 A_j and the oracle's sequential
        // sums 2^-17 of their magnitudes each (the 2^-16 term).
        const float Bb = ldexpf(an * Mn, -13) * 1.25f + ldexpf(Am + fabsf(K0) + fabsf(kth), -16) + 1e-30f;
        const float lim = kth + 2.0f * Bb;
        // a list overflow (more than kList columns at or below T2) or a row or
        // table that is not finite is left to the exact rescoring of every
        // centroid
        const bool over = cnt > kList || !(an2 < INFINITY) || !(lim < INFINITY);
        const bool decided = !over && nxt > lim;
        int n = over ? kRecAll : Mc;
        if (decided) {
#pragma unroll
          for (int s = 0; s < kMaxFilterM; ++s)
            if (s < Mc) myl[1 + s] = (uint8_t)tj[s < CAPT ? s : 0];
        }
        // The band (every j with dt_j <= kth + 2B, ascending j) of the rows
        // that are not decided, from the list (lim <= T2)
        if (!over && !decided) {
          int c2 = 0;
          for (int i = 0; i < mc; ++i) {
            const uint2 en = lst[i];
            const bool take = __uint_as_float(en.x) <= lim;
            const int sl = c2 < kBand ? c2 : kBand - 1;
            if (take) myl[1 + sl] = (uint8_t)en.y;
            c2 += take ? 1 : 0;
          }
          n = c2 <= kBand ? c2 : kRecAll;
        }
        myl[0] = (uint8_t)n;
        const uint4 r0 = lds16(myl), r1 = lds16(myl + 16);
        rec[0] = r0.x; rec[1] = r0.y; rec[2] = r0.z; rec[3] = r0.w;
        rec[4] = r1.x; rec[5] = r1.y; rec[6] = r1.z; rec[7] = r1.w;
      }

      // ---- 4. candidates: the decided top-M, or an exact rescoring of the
      // band members (every centroid when the band was not listed).  The
      // rescoring is shared by the group: a row that needs it reserves a slice
      // of the (row, centroid) list, every thread evaluates list entries from
      // the parked rows, and the owner keeps the M smallest (dQ, j) of its
      // slice.  A row that finds no room in the list rescores itself.
      int cand[kMaxFilterM];
#pragma unroll
      for (int s = 0; s < kMaxFilterM; ++s) cand[s] = 0;
      bool rescore = false, band = false, listed = false;
      int rs_base = 0, rs_n = 0;
      auto rb = [&](int i) -> int { return (int)((rec[i >> 2] >> (8 * (i & 3))) & 0xFFu); };
      if (valid && !all_cand) {
        const int n = rb(0);
        bool idsok = true;
#pragma unroll
        for (int i = 1; i <= kBand; ++i)
          if (i <= n && rb(i) >= C) idsok = false;
        if (n == Mc && idsok) {
#pragma unroll
          for (int s = 0; s < kMaxFilterM; ++s) cand[s] = rb(1 + s);
        } else {
          rescore = true;
          band = n >= Mc && n <= kBand && idsok;  // a band holds at least M members
          rs_n = band ? n : C;
          rs_base = atomicAdd(&sCnt[0], rs_n);
          if (rs_base + rs_n <= kXRsCap) {
            listed = true;
            for (int m = 0; m < rs_n; ++m) {
              int j = m;
              if (band) {
#pragma unroll
                for (int i = 0; i < kBand; ++i)
                  if (i == m) j = rb(1 + i);
              }
              sRsPair[rs_base + m] = (uint16_t)((row << 8) | j);
            }
            atomicMax(&sCnt[2], rs_base + rs_n);
          }
        }
      }
      // every row is done with the selection scratch: the group's next tile
      fence_proxy_async_smem();
      const bool any_rescore = named_bar_or(1 + g, 128, rescore);
      if (row == 0 && u + 2 < u1) {
        issue_tile(u + 2);
        tma_pending = true;
      }
      if (any_rescore) {
        const int total = sCnt[2];  // the listed slices form the prefix [0, total)
        for (int q = row; q < total; q += 128) {
          const int pr = sRsPair[q];
          sRsDq[q] = dq_smem(sLo, pr >> 8, sMU, Npad, pr & 0xFF, sW);
        }
        named_bar_sync(1 + g, 128);
        if (rescore) {
          float ev[kMaxFilterM];
          int ej[kMaxFilterM];
#pragma unroll
          for (int s = 0; s < kMaxFilterM; ++s) { ev[s] = INFINITY; ej[s] = 0x7FFFFFFF; }
          float ek = INFINITY;
          for (int m = 0; m < rs_n; ++m) {  // ascending j in both cases
            float dq;
            int j;
            if (listed) {
              j = sRsPair[rs_base + m] & 0xFF;
              dq = sRsDq[rs_base + m];
            } else {
              j = m;
              if (band) {
#pragma unroll
                for (int i = 0; i < kBand; ++i)
                  if (i == m) j = rb(1 + i);
              }
              dq = dq_smem(sLo, row, sMU, Npad, j, sW);
            }
            if (dq < ek) {
              insert_top(ev, ej, Mc, dq, j);
              ek = sel_at(ev, Mc - 1);
            }
          }
#pragma unroll
          for (int s = 0; s < kMaxFilterM; ++s) cand[s] = ej[s];
        }
      }

      int id = 0;
      float sc[4], inv[4], zf[4];
      __half sh[4];
      uint32_t scode[4] = {0u, 0u, 0u, 0u};   // scale format 1: group codes and secondary scale
      __half s2h = __ushort_as_half(0);
      uint32_t zbyte = 0;
      uint64_t cj[RP], vj[RP];
#pragma unroll
      for (int i = 0; i < RP; ++i) { cj[i] = 0; vj[i] = 0; }
      float err0 = 0.0f;
      uint32_t cw[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) cw[i] = 0;
#pragma unroll
      for (int gi = 0; gi < 4; ++gi) { sc[gi] = 0.0f; inv[gi] = 0.0f; zf[gi] = 0.0f; sh[gi] = __ushort_as_half(0); }

      if (valid) {
        // ---- 5. QSAC score (Eq. 10, 12) of each candidate, lowest (S, j);
        // the group minima / maxima of the chosen residual feed the INT2
        // step.  Candidates are scored QB at a time, channel blocks of 16
        // outermost, so each block of the row is unpacked once per batch.
        constexpr int QB = 4;
        float bestS = INFINITY;
        int bestj = 0x7FFFFFFF;
        float bmn[4], bmx[4];
#pragma unroll
        for (int gi = 0; gi < 4; ++gi) { bmn[gi] = 0.0f; bmx[gi] = 0.0f; }
        const int ncand = all_cand ? C : Mc;
        for (int m0 = 0; m0 < ncand; m0 += QB) {
          const int nbq = ncand - m0 < QB ? ncand - m0 : QB;
          int jb[QB];
#pragma unroll
          for (int b = 0; b < QB; ++b) {
            const int m = m0 + b < ncand ? m0 + b : m0;
            int j = m;
            if (!all_cand) {
#pragma unroll
              for (int s = 0; s < kMaxFilterM; ++s)
                if (s == m) j = cand[s];
            }
            jb[b] = j;
          }
          // minima / maxima per quarter (32 channels); a group of 64 merges two
          float mx[QB][4], mn[QB][4];
#pragma unroll
          for (int b = 0; b < QB; ++b)
#pragma unroll
            for (int qq = 0; qq < 4; ++qq) { mx[b][qq] = -INFINITY; mn[b][qq] = INFINITY; }
#pragma unroll
          for (int cc = 0; cc < 8; ++cc) {
            const int qq = cc >> 1;
            uint64_t k2[8];
#pragma unroll
            {
              const uint4 ka = row_chunk(myrow, rkey, 2 * cc), kb = row_chunk(myrow, rkey, 2 * cc + 1);
              const uint32_t kw[8] = {ka.x, ka.y, ka.z, ka.w, kb.x, kb.y, kb.z, kb.w};
#pragma unroll
              for (int p = 0; p < 8; ++p) k2[p] = bf2_to_f2(kw[p]);
            }
#pragma unroll
            for (int b = 0; b < QB; ++b) {
              if (b < nbq) {
                const uint4 ma = lds16(sMU + sw_off(Npad, jb[b], 2 * cc));
                const uint4 mb = lds16(sMU + sw_off(Npad, jb[b], 2 * cc + 1));
                const uint32_t mw[8] = {ma.x, ma.y, ma.z, ma.w, mb.x, mb.y, mb.z, mb.w};
                float x[16];
#pragma unroll
                for (int p = 0; p < 8; ++p) f2unpack(sub2(k2[p], bf2_to_f2(mw[p])), x[2 * p], x[2 * p + 1]);
#pragma unroll
                for (int e = 0; e < 16; e += 2) {
                  mx[b][qq] = fmax3f(mx[b][qq], x[e], x[e + 1]);
                  mn[b][qq] = fmin3(mn[b][qq], x[e], x[e + 1]);
                }
              }
            }
          }
#pragma unroll
          for (int b = 0; b < QB; ++b) {
            if (b < nbq) {
              if (!gs32) {
                mx[b][0] = fmaxf(mx[b][0], mx[b][1]);
                mn[b][0] = fminf(mn[b][0], mn[b][1]);
                mx[b][1] = fmaxf(mx[b][2], mx[b][3]);
                mn[b][1] = fminf(mn[b][2], mn[b][3]);
              }
              float Sc = 0.0f;
#pragma unroll
              for (int gi = 0; gi < 4; ++gi) {
                if (gi < ng) {
                  const float Rg = __fsub_rn(mx[b][gi], mn[b][gi]);
                  Sc = __fadd_rn(Sc, __fmul_rn(Wg[gi], __fmul_rn(Rg, Rg)));
                }
              }
              const int j = jb[b];
              if (Sc < bestS || (Sc == bestS && j < bestj)) {
                bestS = Sc;
                bestj = j;
#pragma unroll
                for (int gi = 0; gi < 4; ++gi) { bmn[gi] = mn[b][gi]; bmx[gi] = mx[b][gi]; }
              }
            }
          }
        }
        id = bestj < C ? bestj : C - 1;

        // ---- 6. INT2 parameters (Eq. 1-2): range of the residual with 0
        // included; scale format 1 (App. D.1): s = code * s2 with s2 the
        // binary16 round-up of max_g range_g / 3 / 255 and code the smallest
        // byte covering range_g / 3
        float s32g[4];
        float smax = 0.0f;
#pragma unroll
        for (int gi = 0; gi < 4; ++gi) {
          s32g[gi] = 0.0f;
          if (gi < ng) {
            s32g[gi] = __fdiv_rn(__fsub_rn(fmaxf(0.0f, bmx[gi]), fminf(0.0f, bmn[gi])), 3.0f);
            smax = fmaxf(smax, s32g[gi]);
          }
        }
        float s2f = 0.0f;
        if (L.sf) {
          s2h = __float2half_ru(__fdiv_rn(smax, 255.0f));
          s2f = __half2float(s2h);
          if (smax > 0.0f && __fmul_rn(255.0f, s2f) < smax) {
            s2h = __ushort_as_half((unsigned short)(__half_as_ushort(s2h) + 1));
            s2f = __half2float(s2h);
          }
        }
#pragma unroll
        for (int gi = 0; gi < 4; ++gi) {
          sc[gi] = 0.0f; inv[gi] = 0.0f; zf[gi] = 0.0f; sh[gi] = __ushort_as_half(0);
          if (gi < ng) {
            const float lo = fminf(0.0f, bmn[gi]);
            if (L.sf) {
              int c = 0;
              if (s2f > 0.0f) {
                c = (int)ceilf(__fdiv_rn(s32g[gi], s2f));
                if (c > 0 && __fmul_rn((float)(c - 1), s2f) >= s32g[gi]) c -= 1;
                if (__fmul_rn((float)c, s2f) < s32g[gi]) c += 1;
                c = c > 255 ? 255 : c;
              }
              scode[gi] = (uint32_t)c;
              sc[gi] = __fmul_rn((float)c, s2f);
            } else {
              sh[gi] = __float2half_ru(s32g[gi]);
              sc[gi] = __half2float(sh[gi]);
            }
            int zq = 0;
            if (sc[gi] != 0.0f) {
              inv[gi] = __frcp_rn(sc[gi]);
              const int z = (int)rintf(__fmul_rn(-lo, inv[gi]));
              zq = z < 0 ? 0 : (z > 3 ? 3 : z);
            }
            zf[gi] = (float)zq;
            zbyte |= (uint32_t)zq << (2 * gi);
          }
        }

        // ---- 7. one channel pass: INT2 codes; Keys with PSAC also E (Eq. 4,
        // 13), c = U^T E, v = U^T (w o E) and err0 = sum_c w_c E_c^2, in
        // channel order
        const uint64_t MAG2 = f2pack(kMagic, kMagic);
        uint32_t kmag = 0u;  // the largest |k| bits of each half-word lane
#pragma unroll 1
        for (int wd = 0; wd < 8; ++wd) {
          const int gi = gs32 ? (wd >> 1) : (wd >> 2);
          const float s = sel4(sc, gi), iv = sel4(inv, gi), z = sel4(zf, gi);
          const uint64_t S2 = f2pack(s, s), Z2 = f2pack(z, z);
          uint32_t word = 0;
          const uint4 ma = lds16(sMU + sw_off(Npad, id, 2 * wd)), mb = lds16(sMU + sw_off(Npad, id, 2 * wd + 1));
          const uint32_t mw8[8] = {ma.x, ma.y, ma.z, ma.w, mb.x, mb.y, mb.z, mb.w};
#pragma unroll
          for (int hc = 0; hc < 2; ++hc) {
            const int ch = 2 * wd + hc;
            const uint4 kv = row_chunk(myrow, rkey, ch);
            const uint32_t kw[4] = {kv.x, kv.y, kv.z, kv.w};
            kmag = vmax_u16x2(vmax_u16x2(kmag, kw[0] & 0x7FFF7FFFu), vmax_u16x2(kw[1] & 0x7FFF7FFFu, kw[2] & 0x7FFF7FFFu));
            kmag = vmax_u16x2(kmag, kw[3] & 0x7FFF7FFFu);
#pragma unroll
            for (int p = 0; p < 4; ++p) {
              const uint64_t k2 = bf2_to_f2(kw[p]), m2 = bf2_to_f2(mw8[4 * hc + p]);
              float x0, x1;
              f2unpack(sub2(k2, m2), x0, x1);
              // y = x * (1/s) rounded on its own (the scalar intrinsic is never
              // fused into the following add), then rint(y) in both lanes
              const uint64_t y2 = f2pack(__fmul_rn(x0, iv), __fmul_rn(x1, iv));
              const uint64_t r2 = sub2(add2(y2, MAG2), MAG2);
              float q0, q1;
              f2unpack(add2(r2, Z2), q0, q1);
              q0 = fminf(fmaxf(q0, 0.0f), 3.0f);
              q1 = fminf(fmaxf(q1, 0.0f), 3.0f);
              const uint32_t b0 = __float_as_uint(q0 + kTwo23) & 3u, b1 = __float_as_uint(q1 + kTwo23) & 3u;
              word |= (b0 | (b1 << 16)) << (8 * hc + 2 * p);
              if constexpr (R > 0) {
                if (psac) {
                  // E = k - (mu + (q - z) s), then the channel pair's PSAC terms
                  const uint64_t dq2 = sub2(f2pack(q0, q1), Z2);
                  const uint64_t E2 = sub2(k2, add2(m2, mul2(dq2, S2)));
                  const int c0 = ch * 8 + 2 * p;
                  const uint64_t w2 = *reinterpret_cast<const uint64_t*>(sW + c0);
                  const uint64_t wE2 = mul2(w2, E2);
                  float E0, E1, wE0, wE1;
                  f2unpack(E2, E0, E1);
                  f2unpack(wE2, wE0, wE1);
                  const uint64_t e0 = f2pack(E0, E0), e1 = f2pack(E1, E1);
                  const uint64_t we0 = f2pack(wE0, wE0), we1 = f2pack(wE1, wE1);
                  const uint4* u0p = reinterpret_cast<const uint4*>(sU + c0 * R);
                  const uint4* u1p = reinterpret_cast<const uint4*>(sU + (c0 + 1) * R);
#pragma unroll
                  for (int i = 0; i < RP / 2; ++i) {
                    const uint4 q = u0p[i];
                    const uint64_t ua = f2pack(__uint_as_float(q.x), __uint_as_float(q.y));
                    const uint64_t ub = f2pack(__uint_as_float(q.z), __uint_as_float(q.w));
                    cj[2 * i] = fma2(e0, ua, cj[2 * i]);
                    vj[2 * i] = fma2(ua, we0, vj[2 * i]);
                    cj[2 * i + 1] = fma2(e0, ub, cj[2 * i + 1]);
                    vj[2 * i + 1] = fma2(ub, we0, vj[2 * i + 1]);
                  }
#pragma unroll
                  for (int i = 0; i < RP / 2; ++i) {
                    const uint4 q = u1p[i];
                    const uint64_t ua = f2pack(__uint_as_float(q.x), __uint_as_float(q.y));
                    const uint64_t ub = f2pack(__uint_as_float(q.z), __uint_as_float(q.w));
                    cj[2 * i] = fma2(e1, ua, cj[2 * i]);
                    vj[2 * i] = fma2(ua, we1, vj[2 * i]);
                    cj[2 * i + 1] = fma2(e1, ub, cj[2 * i + 1]);
                    vj[2 * i + 1] = fma2(ub, we1, vj[2 * i + 1]);
                  }
                  float t0, t1, w0, w1;
                  f2unpack(mul2(E2, E2), t0, t1);
                  f2unpack(w2, w0, w1);
                  err0 = __fmaf_rn(w0, t0, err0);
                  err0 = __fmaf_rn(w1, t1, err0);
                }
              }
            }
          }
#pragma unroll
          for (int i = 0; i < 8; ++i)
            if (i == wd) cw[i] = word;
        }
        // |k0_c - k_c| <= s/2 (the INT2 round trip), so the rebuilt values
        // stay inside the binary16 operands of attention when max|k| + s/2
        // does
        {
          const float km = fmaxf(__uint_as_float(kmag << 16), __uint_as_float(kmag & 0xFFFF0000u));
          const float smx = fmaxf(fmaxf(sc[0], sc[1]), fmaxf(sc[2], sc[3]));
          nbad |= bf16x2_out_of_f16(kmag) || !(km + 0.5f * smx < 65504.0f);
        }
      }

      // ---- 8. stores, PSAC
      uint32_t pcw[R > 0 ? R / 4 : 1];  // this token's PSAC codes and row scale when kept (Keys)
#pragma unroll
      for (int i = 0; i < (R > 0 ? R / 4 : 1); ++i) pcw[i] = 0;
      __half psg = __ushort_as_half(0);
      bool pkept = false;
      if (valid) {
        uint32_t* dcodes = reinterpret_cast<uint32_t*>(tb + (is_key ? L.k_codes : L.v_codes) + row * 32);
        reinterpret_cast<uint4*>(dcodes)[0] = make_uint4(cw[0], cw[1], cw[2], cw[3]);
        reinterpret_cast<uint4*>(dcodes)[1] = make_uint4(cw[4], cw[5], cw[6], cw[7]);
        if (L.sf) {
          uint8_t* dsc = tb + (is_key ? L.k_scales : L.v_scales) + (int64_t)row * ng;
#pragma unroll
          for (int gi = 0; gi < ng; ++gi) dsc[gi] = (uint8_t)scode[gi];
          reinterpret_cast<__half*>(tb + (is_key ? L.k_s2 : L.v_s2))[row] = s2h;
        } else if (ng == 4) {
          uint2 sv;
          sv.x = (uint32_t)__half_as_ushort(sh[0]) | ((uint32_t)__half_as_ushort(sh[1]) << 16);
          sv.y = (uint32_t)__half_as_ushort(sh[2]) | ((uint32_t)__half_as_ushort(sh[3]) << 16);
          *reinterpret_cast<uint2*>(tb + (is_key ? L.k_scales : L.v_scales) + row * 8) = sv;
        } else {
          *reinterpret_cast<uint32_t*>(tb + (is_key ? L.k_scales : L.v_scales) + row * 4) =
              (uint32_t)__half_as_ushort(sh[0]) | ((uint32_t)__half_as_ushort(sh[1]) << 16);
        }
        tb[(is_key ? L.k_ids : L.v_ids) + row] = (uint8_t)id;
        {
          uint8_t* dz = tb + (is_key ? L.k_zeros : L.v_zeros) + (int64_t)row * L.zb;
          dz[0] = (uint8_t)zbyte;
          for (int b = 1; b < L.zb; ++b) dz[b] = 0;
        }

        // ---- PSAC coefficients (Eq. 13, INT8 with a binary16 row scale) and
        // the keep rule (Eq. 16), Keys only
        if constexpr (R > 0) {
          if (psac) {
            float c[R], v[R];
#pragma unroll
            for (int i = 0; i < RP; ++i) {
              f2unpack(cj[i], c[2 * i], c[2 * i + 1]);
              f2unpack(vj[i], v[2 * i], v[2 * i + 1]);
            }
            float amax = 0.0f;
#pragma unroll
            for (int j = 0; j < R; ++j) amax = fmaxf(amax, fabsf(c[j]));
            const __half sgh = __float2half_ru(__fdiv_rn(amax, 127.0f));
            const float sg = __half2float(sgh);
            nbad |= !(127.0f * sg <= 65504.0f);  // C_hat = t sigma must stay a finite binary16
            const float sinv = sg != 0.0f ? __frcp_rn(sg) : 0.0f;
            float chat[R];
            uint32_t tq[R / 4];
#pragma unroll
            for (int i = 0; i < R / 4; ++i) tq[i] = 0;
#pragma unroll
            for (int j = 0; j < R; ++j) {
              const float qq = sg != 0.0f ? fminf(fmaxf(rintf(__fmul_rn(c[j], sinv)), -127.0f), 127.0f) : 0.0f;
              tq[j >> 2] |= ((uint32_t)(int)qq & 0xFFu) << (8 * (j & 3));
              chat[j] = __fmul_rn(qq, sg);
            }
            bool keep = false;  // sigma == 0: chat = 0, so errq == err0 and the rule says no
            if (sg != 0.0f) {
              // errq - err0 = chat^T G chat - 2 chat.v with G = U^T W U
              float quad = 0.0f, cv = 0.0f, cn2 = 0.0f, vn2 = 0.0f;
#pragma unroll
              for (int j = 0; j < R; ++j) {
                float gj = 0.0f;
#pragma unroll
                for (int k = 0; k < R; ++k) gj = fmaf(sG[j * R + k], chat[k], gj);
                quad = fmaf(chat[j], gj, quad);
                cv = fmaf(chat[j], v[j], cv);
                cn2 = fmaf(chat[j], chat[j], cn2);
                vn2 = fmaf(v[j], v[j], vn2);
              }
              float UF2 = 0.0f, wmax = 0.0f;
#pragma unroll
              for (int i = 0; i < 4; ++i) {
                UF2 += sMisc[8 + i];
                wmax = fmaxf(wmax, sMisc[12 + i]);
              }
              const float delta = fmaf(-2.0f, cv, quad);
              const float eq = fabsf(err0 + delta);
              const float Q = wmax * UF2 * cn2 * 1.0001f;
              const float bound =
                  ldexpf(eq + err0 + Q + sqrtf(err0 * Q) + sqrtf(eq * Q) + sqrtf(cn2 * vn2), -14) + 1e-35f;
              if (delta < -bound) {
                keep = true;
              } else if (!(delta > bound)) {
                // too close to call: the sequential evaluation of both sums
                float errq = 0.0f, e0s = 0.0f;
#pragma unroll 1
                for (int wd = 0; wd < 8; ++wd) {
                  const int gi = gs32 ? (wd >> 1) : (wd >> 2);
                  const float s = sel4(sc, gi), z = sel4(zf, gi);
                  uint32_t word = cw[0];
#pragma unroll
                  for (int i = 1; i < 8; ++i)
                    if (i == wd) word = cw[i];
#pragma unroll
                  for (int hc = 0; hc < 2; ++hc) {
                    const int ch = 2 * wd + hc;
                    const uint4 kv = row_chunk(myrow, rkey, ch);
                    const uint4 mv = lds16(sMU + sw_off(Npad, id, ch));
                    const uint32_t kw[4] = {kv.x, kv.y, kv.z, kv.w}, mw[4] = {mv.x, mv.y, mv.z, mv.w};
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                      const int cI = ch * 8 + e;
                      const float kf = __uint_as_float((e & 1) ? (kw[e >> 1] & 0xFFFF0000u) : (kw[e >> 1] << 16));
                      const float mf = __uint_as_float((e & 1) ? (mw[e >> 1] & 0xFFFF0000u) : (mw[e >> 1] << 16));
                      const int j16 = 8 * hc + e;
                      const float qv = (float)((word >> (16 * (j16 & 1) + 2 * (j16 >> 1))) & 3u);
                      const float E = __fsub_rn(kf, __fadd_rn(mf, __fmul_rn(__fsub_rn(qv, z), s)));
                      float uu = 0.0f;
#pragma unroll
                      for (int j = 0; j < R; ++j) uu = __fmaf_rn(sU[cI * R + j], chat[j], uu);
                      const float ep = __fsub_rn(E, uu);
                      errq = __fmaf_rn(sW[cI], __fmul_rn(ep, ep), errq);
                      e0s = __fmaf_rn(sW[cI], __fmul_rn(E, E), e0s);
                    }
                  }
                }
                keep = errq < e0s;
              }
            }
            if (keep) {
#pragma unroll
              for (int i = 0; i < R / 4; ++i) pcw[i] = tq[i];
              psg = sgh;
              pkept = true;
            }
          }
        }
      }

      // ---- 9. the tile's PSAC rows in the smaller of the two layouts (App.
      // D.1): dense (every token's row, dropped corrections as zeros) or
      // sparse (only the kept rows, compacted in token order), with the
      // tile's 128-bit keep mask naming the rows stored (row i is entry
      // popcount(mask below i)).
      if constexpr (R > 0) {
        if (is_key) {
          const uint32_t wmk = __ballot_sync(0xFFFFFFFFu, pkept);
          if (lane == 0) sCnt[4 + gw] = (int)wmk;
          named_bar_sync(1 + g, 128);
          uint32_t m4[4] = {(uint32_t)sCnt[4], (uint32_t)sCnt[5], (uint32_t)sCnt[6], (uint32_t)sCnt[7]};
          const int nt = (int)((a.N - (int64_t)tile * 128) < 128 ? (a.N - (int64_t)tile * 128) : 128);
          const int Kt = __popc(m4[0]) + __popc(m4[1]) + __popc(m4[2]) + __popc(m4[3]);
          const bool sparse = 16 + Kt * (R + 2) < nt * (R + 2);
          int e = row;
          if (sparse) {
            e = __popc(m4[gw] & ((1u << lane) - 1u));
#pragma unroll
            for (int w4 = 0; w4 < 3; ++w4) e += w4 < gw ? __popc(m4[w4]) : 0;
          } else {
#pragma unroll
            for (int w4 = 0; w4 < 4; ++w4) {
              const int nbits = nt - 32 * w4;
              m4[w4] = nbits >= 32 ? 0xFFFFFFFFu : (nbits > 0 ? (1u << nbits) - 1u : 0u);
            }
          }
          if (valid && (!sparse || pkept)) {
            int8_t* coef = reinterpret_cast<int8_t*>(tb + L.k_coef + (int64_t)e * R);
            if constexpr (R == 8) {
              *reinterpret_cast<uint2*>(coef) = make_uint2(pcw[0], pcw[1]);
            } else {
#pragma unroll
              for (int i = 0; i < R / 16; ++i)
                reinterpret_cast<uint4*>(coef)[i] = make_uint4(pcw[4 * i], pcw[4 * i + 1], pcw[4 * i + 2], pcw[4 * i + 3]);
            }
            reinterpret_cast<__half*>(tb + L.k_sigma)[e] = psg;
          }
          if (row == 0)
            *reinterpret_cast<uint4*>(head + L.pmask + (int64_t)tile * 16) = make_uint4(m4[0], m4[1], m4[2], m4[3]);
        }
      }
      // the group's next tile writes its operand into the rows' buffer: every
      // read of the parked rows comes first (for Key tiles with PSAC the
      // layout step's barrier above already orders them)
      if (!(R > 0 && is_key)) named_bar_sync(1 + g, 128);
    }
    s0 = s1;
  }

  // ---- exit: copies or MMAs still in flight (a unit not reached after a
  // wait ran out) are waited for before the CTA's memory goes away
  __syncthreads();
  const bool tout = stop || sFlag[0] || sFlag[1];
  if (row == 0 && tma_pending) mbar_wait(bar_tma, ph_tma);
  if (row == 0 && mma_pending) mbar_wait(bar_mma, ph_mma);
  if (tid == 0 && tout) atomicCAS(reinterpret_cast<int*>(a.base), 0, (int)QWM_ERR_TIMEOUT);
  if (nbad) atomicCAS(reinterpret_cast<int*>(a.base), 0, (int)QWM_ERR_NONFINITE);
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tbase, 512);
  }
}

// Launch of the M = 4 instance (the paper's default candidate count has its
// own ranked-list length) or the shared one (the other counts up to
// kMaxFilterM, and M >= C where no selection runs), PSAC rank R.
template <int R>
cudaError_t launch_fused_rank(const AppendArgs& a, const CUtensorMap* maps, cudaStream_t st) {
  constexpr int smem = XSmem<R>::BYTES;
  auto kern = a.M == 4 ? append_fused<5, R> : append_fused<kMaxFilterM + 1, R>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  int dev = 0, nsm = 0;
  e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return e;
  const int tiles = (int)((a.N + 127) / 128);
  const int units = 2 * a.L.H * tiles;
  const int grid = units < nsm ? units : nsm;
  kern<<<grid, XNT, smem, st>>>(a, maps[0], maps[1], maps[2], maps[3], tiles, units);
  return cudaGetLastError();
}

}  // namespace

// One translation unit per PSAC rank (append_fused.cu: r = 0 and the
// dispatch; append_fused_r8.cu, _r16.cu, _r32.cu), compiled in parallel.
// maps: the Key and Value token maps, then the Key and Value table maps.
cudaError_t append_fused_r0(const AppendArgs& a, const CUtensorMap* maps, cudaStream_t st);
cudaError_t append_fused_r8(const AppendArgs& a, const CUtensorMap* maps, cudaStream_t st);
cudaError_t append_fused_r16(const AppendArgs& a, const CUtensorMap* maps, cudaStream_t st);
cudaError_t append_fused_r32(const AppendArgs& a, const CUtensorMap* maps, cudaStream_t st);

}  // namespace qwm
