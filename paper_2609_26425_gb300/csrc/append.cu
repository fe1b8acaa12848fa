// append.cu -- quantize-on-append: a tensor-core candidate filter followed by
// the exact per-token quantisation.
//
// Kernel 1, append_filter (persistent, one CTA per SM, two groups of 128
// token rows).  For a run of 128-token tiles of one (head, K/V side):
//   * once per run, B = w o mu for all C centroids (Sec. 4.1, Eq. 9 expanded
//     as dQ_j = sum_c w_c k_c^2 - 2 D_j + A_j with D = K (w o mu)^T and
//     A_j = sum_c w_c mu_jc^2) is split into two binary16 operands
//     B_hi = f16(w o mu), B_lo = f16(w o mu - B_hi), so that B_hi + B_lo
//     carries w o mu to 2^-22 relative;
//   * per tile, the bf16 token rows arrive by TMA (128-byte swizzled), are
//     converted in place to binary16, and two tcgen05 MMAs accumulate
//     D = K B_hi^T + K B_lo^T (fp32, 128 x C) in TMEM;
//   * each thread reads its row of D and keeps the M+1 smallest
//     dt_j = A_j - 2 D_j.  With the error bound B of dt (the split operand,
//     the fp32 accumulation, and the fp32 rounding of the sequential
//     Query-aware distance the selection is defined on), every centroid of
//     the exact top-M lies within 2B of the M-th smallest dt; when the
//     (M+1)-th lies beyond that band the top-M is decided, otherwise the band
//     members (at most 16) are listed for exact rescoring.
//   The decision record of a token (count byte + up to 16 centroid ids) is
//   parked in the token's own 32 code bytes of the destination slot.
//
// Kernel 2, append_quant (one CTA per 128-token tile, thread = token; the
// tile arrives by TMA).  It reads the record, rescores band members exactly
// when needed, evaluates the QSAC score (Eq. 10, 12) of each candidate, and
// quantises the residual to INT2 (Eq. 1-2) with packing.  For Keys, the same
// channel pass accumulates the PSAC projection c = U_r^T E (Eq. 13) in
// channel order (one fused multiply-add per term) together with
// v = U_r^T (w o E) and err0 = sum_c w_c E_c^2;
// the keep rule (Eq. 16, diagonal-w form) compares
// errq - err0 = chat^T (U^T W U) chat - 2 chat.v against a rigorous bound of
// its difference to the sequential evaluation, and evaluates the two sums
// sequentially only when they are too close to call.  All arithmetic that
// decides an output is fp32 in channel order with every rounding explicit:
// a separately rounded multiply or add, or one fused multiply-add per term
// of a sum of products (packed two lanes at a time where the lanes are
// independent), identical to the sequential evaluation of the formulas.
//
// M >= C skips the filter (every centroid is a candidate); 8 < M < C goes to
// the generic kernel (append_generic.cu).
#include "ptx_sm103.cuh"
#include "qwm_internal.cuh"
#include "append_common.cuh"

namespace qwm {
namespace {

using namespace ptx;


// ============================================================================
// Kernel 1: candidate filter
// ============================================================================
constexpr int FG = 2;                       // token groups per CTA
constexpr int FNT = FG * 128;
constexpr int F_BHI = 0;                    // [2][256 rows][128 B] f16
constexpr int F_BLO = 65536;
constexpr int F_A = 131072;                 // FG x [2][128 rows][128 B]
constexpr int F_AJ = F_A + FG * 32768;      // A_j [256] fp32
constexpr int F_W = F_AJ + 1024;            // w [128]
constexpr int F_RED = F_W + 512;            // [8 warps][4]
constexpr int F_LIST = F_RED + 128;         // FNT x 32-byte records
constexpr int F_BAR = F_LIST + FNT * 32;    // 4 mbarriers, flags, TMEM slot
constexpr int F_SMEM = F_BAR + 64 + 1024;

// CAPT = M + 1 (the ranked list of a row), or kMaxFilterM + 1 for the
// candidate counts without their own instance; FULL: the Keys' distance is
// the full quadratic form (qwm_quantize_append_full).
template <int CAPT, bool FULL>
__global__ void __launch_bounds__(FNT, 1)
    append_filter(const AppendArgs a, const __grid_constant__ CUtensorMap tm_k,
                  const __grid_constant__ CUtensorMap tm_v, int tiles, int units) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  const Layout& L = a.L;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = tid >> 7, row = tid & 127;
  const int C = L.C, H = L.H, Mc = a.M;
  const int Npad = (C + 15) & ~15;

  float* sAj = reinterpret_cast<float*>(sm + F_AJ);
  float* sW = reinterpret_cast<float*>(sm + F_W);
  float* sRed = reinterpret_cast<float*>(sm + F_RED);
  uint8_t* myl = sm + F_LIST + tid * 32;
  const uint32_t bar_tma = smem_u32(sm + F_BAR + 8 * g);
  const uint32_t bar_mma = smem_u32(sm + F_BAR + 16 + 8 * g);
  volatile int* flagA = reinterpret_cast<volatile int*>(sm + F_BAR + 32);  // [FG] copy timed out
  volatile int* flagB = reinterpret_cast<volatile int*>(sm + F_BAR + 40);  // [FG] MMA timed out
  uint32_t* tslot = reinterpret_cast<uint32_t*>(sm + F_BAR + 48);
  uint8_t* sA = sm + F_A + g * 32768;

  if (warp == 0) {
    tmem_alloc(smem_u32(tslot), 512);
    tmem_relinquish();
  }
  if (tid == 0) {
    for (int i = 0; i < 4; ++i) mbar_init(smem_u32(sm + F_BAR + 8 * i), 1);
    fence_mbar_init();
    flagA[0] = flagA[1] = 0;
    flagB[0] = flagB[1] = 0;
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tbase = *tslot;
  const uint32_t tD = tbase + (uint32_t)(g * 256);
  const uint32_t lrow = (uint32_t)((warp & 3) * 32) << 16;

  const int nb = gridDim.x;
  const int u0 = (int)((int64_t)blockIdx.x * units / nb);
  const int u1 = (int)((int64_t)(blockIdx.x + 1) * units / nb);
  uint32_t ph_tma = 0, ph_mma = 0;

  for (int s0 = u0; s0 < u1;) {
    const int pair = s0 / tiles;                 // side * H + h
    const int s1 = min(u1, (pair + 1) * tiles);
    const bool is_key = pair < H;
    const int h = pair % H;
    const bool use_w = is_key && a.w != nullptr;
    const __nv_bfloat16* tab = (is_key ? a.kc : a.vc) + (size_t)h * C * 128;
    const CUtensorMap* tm = is_key ? &tm_k : &tm_v;
    uint8_t* head = a.base + head_offset(L, a.slot, h);
    const int64_t o_rec = is_key ? L.k_codes : L.v_codes;

    // ---- B_hi, B_lo and A_j of this (head, side)
    if (tid < 128) sW[tid] = use_w ? a.w[(size_t)h * 128 + tid] : 1.0f;
    __syncthreads();
    // With the full quadratic form (App. C.4, Keys only), B = M mu_j and
    // A_j = mu_j^T M mu_j; the bound then needs max |mu_j| and the largest
    // row sum of |M| (mun2, mabs).
    const bool full = FULL && is_key;
    const float* Mh = full ? a.Mq + (size_t)h * 128 * 128 : nullptr;
    float n2 = 0.0f, amax = 0.0f, mun2 = 0.0f, mabs = 0.0f;
    if (full && tid < 128) {
      const float4* Mr = reinterpret_cast<const float4*>(Mh + (size_t)tid * 128);
      for (int c4 = 0; c4 < 32; ++c4) {
        const float4 m4 = __ldg(Mr + c4);
        mabs += fabsf(m4.x) + fabsf(m4.y) + fabsf(m4.z) + fabsf(m4.w);
      }
      mabs *= 1.0001f;  // the fp32 sum of the absolute values, rounded up
    }
    if (full) {
      const int j = tid;
      if (j < C) {
        const __nv_bfloat16* mr = tab + (size_t)j * 128;
        uint32_t muw[64];
#pragma unroll
        for (int ch = 0; ch < 16; ++ch) {
          const uint4 m = ldg16(mr + ch * 8);
          muw[4 * ch] = m.x; muw[4 * ch + 1] = m.y; muw[4 * ch + 2] = m.z; muw[4 * ch + 3] = m.w;
        }
        float A = 0.0f;
#pragma unroll 1
        for (int ch = 0; ch < 16; ++ch) {
          float b8[8];
#pragma unroll
          for (int o = 0; o < 8; ++o) {
            const float4* Mr = reinterpret_cast<const float4*>(Mh + (size_t)(ch * 8 + o) * 128);
            float acc = 0.0f;
#pragma unroll
            for (int c4 = 0; c4 < 32; ++c4) {
              const float4 m4 = __ldg(Mr + c4);
              const uint32_t w0 = muw[2 * c4], w1 = muw[2 * c4 + 1];
              acc = fmaf(m4.x, __uint_as_float(w0 << 16), acc);
              acc = fmaf(m4.y, __uint_as_float(w0 & 0xFFFF0000u), acc);
              acc = fmaf(m4.z, __uint_as_float(w1 << 16), acc);
              acc = fmaf(m4.w, __uint_as_float(w1 & 0xFFFF0000u), acc);
            }
            b8[o] = acc;
          }
          uint32_t hw[4], lw[4];
#pragma unroll
          for (int p2 = 0; p2 < 4; ++p2) {
            const float b0 = b8[2 * p2], b1 = b8[2 * p2 + 1];
            const uint32_t mw = muw[4 * ch + p2];
            const float m0 = __uint_as_float(mw << 16), m1 = __uint_as_float(mw & 0xFFFF0000u);
            A = fmaf(m0, b0, fmaf(m1, b1, A));
            n2 = fmaf(b0, b0, fmaf(b1, b1, n2));
            mun2 = fmaf(m0, m0, fmaf(m1, m1, mun2));
            const __half2 hh = __floats2half2_rn(b0, b1);
            const float2 hf = __half22float2(hh);
            hw[p2] = *reinterpret_cast<const uint32_t*>(&hh);
            lw[p2] = pack_f16(b0 - hf.x, b1 - hf.y);
          }
          const int off = sw_off(Npad, j, ch);
          *reinterpret_cast<uint4*>(sm + F_BHI + off) = make_uint4(hw[0], hw[1], hw[2], hw[3]);
          *reinterpret_cast<uint4*>(sm + F_BLO + off) = make_uint4(lw[0], lw[1], lw[2], lw[3]);
        }
        sAj[j] = A;
        amax = fabsf(A);
      } else {
        if (j < Npad) {
#pragma unroll
          for (int ch = 0; ch < 16; ++ch) {
            const int off = sw_off(Npad, j, ch);
            *reinterpret_cast<uint4*>(sm + F_BHI + off) = make_uint4(0, 0, 0, 0);
            *reinterpret_cast<uint4*>(sm + F_BLO + off) = make_uint4(0, 0, 0, 0);
          }
        }
        sAj[j] = INFINITY;  // j in [C, 256): never selected
      }
    } else {
      const int j = tid;
      if (j < C) {
        const __nv_bfloat16* mr = tab + (size_t)j * 128;
        float A = 0.0f;
#pragma unroll 4
        for (int ch = 0; ch < 16; ++ch) {
          const uint4 m = ldg16(mr + ch * 8);
          const uint32_t mw[4] = {m.x, m.y, m.z, m.w};
          uint32_t hw[4], lw[4];
#pragma unroll
          for (int p = 0; p < 4; ++p) {
            const float m0 = __uint_as_float(mw[p] << 16), m1 = __uint_as_float(mw[p] & 0xFFFF0000u);
            const float w0 = __fmul_rn(sW[ch * 8 + 2 * p], m0), w1 = __fmul_rn(sW[ch * 8 + 2 * p + 1], m1);
            A = fmaf(w0, m0, fmaf(w1, m1, A));
            n2 = fmaf(w0, w0, fmaf(w1, w1, n2));
            const __half2 hh = __floats2half2_rn(w0, w1);
            const float2 hf = __half22float2(hh);
            hw[p] = *reinterpret_cast<const uint32_t*>(&hh);
            lw[p] = pack_f16(w0 - hf.x, w1 - hf.y);
          }
          const int off = sw_off(Npad, j, ch);
          *reinterpret_cast<uint4*>(sm + F_BHI + off) = make_uint4(hw[0], hw[1], hw[2], hw[3]);
          *reinterpret_cast<uint4*>(sm + F_BLO + off) = make_uint4(lw[0], lw[1], lw[2], lw[3]);
        }
        sAj[j] = A;
        amax = fabsf(A);
      } else {
        if (j < Npad) {
#pragma unroll
          for (int ch = 0; ch < 16; ++ch) {
            const int off = sw_off(Npad, j, ch);
            *reinterpret_cast<uint4*>(sm + F_BHI + off) = make_uint4(0, 0, 0, 0);
            *reinterpret_cast<uint4*>(sm + F_BLO + off) = make_uint4(0, 0, 0, 0);
          }
        }
        sAj[j] = INFINITY;  // j in [C, 256): never selected
      }
    }
#pragma unroll
    for (int off = 16; off; off >>= 1) {
      n2 = fmaxf(n2, __shfl_xor_sync(0xFFFFFFFFu, n2, off));
      amax = fmaxf(amax, __shfl_xor_sync(0xFFFFFFFFu, amax, off));
      mun2 = fmaxf(mun2, __shfl_xor_sync(0xFFFFFFFFu, mun2, off));
      mabs = fmaxf(mabs, __shfl_xor_sync(0xFFFFFFFFu, mabs, off));
    }
    if (lane == 0) {
      sRed[4 * warp] = n2;
      sRed[4 * warp + 1] = amax;
      sRed[4 * warp + 2] = mun2;
      sRed[4 * warp + 3] = mabs;
    }
    fence_proxy_async_smem();
    __syncthreads();
    float W2 = 0.0f, Am = 0.0f, Mu2 = 0.0f, Mab = 0.0f;
#pragma unroll
    for (int i = 0; i < FNT / 32; ++i) {
      W2 = fmaxf(W2, sRed[4 * i]);
      Am = fmaxf(Am, sRed[4 * i + 1]);
      Mu2 = fmaxf(Mu2, sRed[4 * i + 2]);
      Mab = fmaxf(Mab, sRed[4 * i + 3]);
    }
    const float Wn = sqrtf(W2);
    const float Mun = sqrtf(Mu2) * 1.0001f;

    // ---- the tiles of this run, alternating between the two groups
    for (int u = s0 + g; u < s1; u += FG) {
      const int tile = u - pair * tiles;
      if (row == 0) {
        mbar_arrive_expect_tx(bar_tma, 32768);
        tma_load_3d(smem_u32(sA), tm, 0, h, tile * 128, bar_tma);
        tma_load_3d(smem_u32(sA + 16384), tm, 64, h, tile * 128, bar_tma);
      }
      if (!mbar_wait(bar_tma, ph_tma)) flagA[g] = 1;
      ph_tma ^= 1;

      // bf16 row -> binary16 in place; |k|^2, sum_c w_c k_c^2, max |k_c|
      float kn2 = 0.0f, K0 = 0.0f, kmx = 0.0f;
#pragma unroll 4
      for (int ch = 0; ch < 16; ++ch) {
        uint4* p = reinterpret_cast<uint4*>(sA + sw_off(128, row, ch));
        const uint4 v = *p;
        const uint32_t vw[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const float k0 = __uint_as_float(vw[q] << 16), k1 = __uint_as_float(vw[q] & 0xFFFF0000u);
          kn2 = fmaf(k0, k0, fmaf(k1, k1, kn2));
          K0 = fmaf(sW[ch * 8 + 2 * q] * k0, k0, fmaf(sW[ch * 8 + 2 * q + 1] * k1, k1, K0));
          kmx = fmax3f(kmx, fabsf(k0), fabsf(k1));
        }
        *p = bf16x8_to_f16x8(v);
      }
      fence_proxy_async_smem();
      tc_fence_before();
      named_bar_sync(1 + g, 128);
      tc_fence_after();
      if (flagA[g]) break;
      if (row == 0) {
        const uint32_t aA = smem_u32(sA);
        const uint32_t id = idesc_f16(128, Npad, false);
#pragma unroll
        for (int hl = 0; hl < 2; ++hl) {
          const uint32_t aB = smem_u32(sm + (hl ? F_BLO : F_BHI));
#pragma unroll
          for (int kb = 0; kb < 2; ++kb)
#pragma unroll
            for (int ks = 0; ks < 4; ++ks)
              umma_ss(tD, desc_sw128(aA + kb * 16384 + ks * 32), desc_sw128(aB + kb * Npad * 128 + ks * 32), id,
                      (hl | kb | ks) != 0);
        }
        umma_commit(bar_mma);
      }
      if (!mbar_wait(bar_mma, ph_mma)) flagB[g] = 1;
      ph_mma ^= 1;
      tc_fence_after();

      // ---- selection over dt_j = A_j - 2 D_j (the TMEM reads are
      // warp-collective, every other step is per row).
      //   1. the minima of 16 interleaved column groups (column j in group
      //      j % 16); their (M+1)-th smallest, T, bounds the (M+1)-th
      //      smallest dt from above;
      //   2. a second pass marks the columns with dt <= T in a bit mask per
      //      32 columns (usually a handful per row); only those are ranked
      //      (the M+1 smallest, ties to the lower j) and listed, in
      //      ascending j, in this group's A tile (free once the MMA has
      //      completed), with the values of a 32-column block stashed there
      //      when the block has one.
      constexpr int kList = 16;
      const int nchunk = ((Npad + 63) >> 6) << 1;  // pairs of 32-column blocks (at most 256 columns)
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
      for (int cb = 0; cb < nchunk; cb += 2) {
        float va[32], vb[32];
        __syncwarp();
        tmem_ld32x2(tD + lrow + cb * 32, tD + lrow + cb * 32 + 32, va, vb);
        dt32(cb, va);
        dt32(cb + 1, vb);
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

      // [kList] entries of (dt, column) per row after a 32-float stash, slot-swizzled
      uint8_t* rowbuf = sA + row * 256;
      float* stash = reinterpret_cast<float*>(rowbuf);
      uint2* lst = reinterpret_cast<uint2*>(rowbuf + 128);
      const int sw = row & 7;
      float tv[CAPT];
      int tj[CAPT];
#pragma unroll
      for (int i = 0; i < CAPT; ++i) { tv[i] = INFINITY; tj[i] = 0x7FFFFFFF; }
      int cnt = 0;
#pragma unroll 1
      for (int cb = 0; cb < nchunk; cb += 2) {
        float va[32], vb[32];
        __syncwarp();
        tmem_ld32x2(tD + lrow + cb * 32, tD + lrow + cb * 32 + 32, va, vb);
        dt32(cb, va);
        dt32(cb + 1, vb);
#pragma unroll
        for (int hb = 0; hb < 2; ++hb) {
          const float (&v)[32] = hb ? vb : va;
          uint32_t mk = 0;
#pragma unroll
          for (int e = 0; e < 32; ++e) mk |= (v[e] <= T ? 1u : 0u) << e;
          if (mk) {
#pragma unroll
            for (int k4 = 0; k4 < 8; ++k4)
              reinterpret_cast<float4*>(stash)[k4 ^ sw] = make_float4(v[4 * k4], v[4 * k4 + 1], v[4 * k4 + 2], v[4 * k4 + 3]);
            do {
              const int e = __ffs(mk) - 1;
              mk &= mk - 1;
              const float x = stash[(((e >> 2) ^ sw) << 2) | (e & 3)];
              const int j = (cb + hb) * 32 + e;
              if (cnt < kList) lst[cnt] = make_uint2(__float_as_uint(x), (uint32_t)j);
              ++cnt;
              insert_top(tv, tj, Mc + 1, x, j);
            } while (mk);
          }
        }
      }
      const int mc = cnt < kList ? cnt : kList;

      const float kth = sel_at(tv, Mc - 1), nxt = sel_at(tv, Mc);
      const float kn = sqrtf(kn2);
      // |our dt_j - the oracle's d_j + common term| <= Bb for every candidate.
      // The tensor cores' fp32 accumulation is taken to move the sum by at most
      // two ulps of its running absolute value per product added (256 products:
      // 2^-14 |k| |B_j| by Cauchy-Schwarz, twice that in dt = A - 2 D); the
      // operand split adds 2^-22 |k| |B_j|, the fp32 A_j and the oracle's
      // sequential sums 2^-17 of their magnitudes each, and binary16 subnormal
      // operands an absolute 2^-25 per element (the 2^-19 term).  For the full
      // form (App. C.4) every one of these is below 2^-13 (|k| + max|mu|)^2
      // max_c sum_c' |M_cc'| (the norm of M for a symmetric M).
      const float Bb = full ? ldexpf((kn + Mun) * (kn + Mun) * Mab, -13) + ldexpf(kn + Wn, -19) + 1e-30f
                            : ldexpf(kn * Wn, -13) + ldexpf(Am + K0 + fabsf(kth), -16) + ldexpf(kn + Wn, -19) +
                                  1e-30f;
      const float lim = kth + 2.0f * Bb;
      // a list overflow (more than kList columns at or below T), a row out of
      // the binary16 range, or a table whose w o mu rows reach beyond it (the
      // f16 operand would not hold them) is left to the exact rescoring of
      // every centroid
      const bool over = cnt > kList || !(kmx <= 65504.0f) || !(kn2 < INFINITY) || !(lim < INFINITY) ||
                        !(Wn < 65504.0f);
      const bool decided = !over && nxt > lim;
      int n = over ? kRecAll : Mc;
      if (decided) {
#pragma unroll
        for (int s = 0; s < kMaxFilterM; ++s)
          if (s < Mc) myl[1 + s] = (uint8_t)tj[s < CAPT ? s : 0];
      }
      // The band (every j with dt_j <= kth + 2B, ascending j) of the rows
      // that are not decided: from the list when it covers the band
      // (lim <= T), otherwise from all columns.
      const bool need_band = !over && !decided;
      if (need_band && lim <= T) {
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
      const bool need_scan = need_band && !(lim <= T);
      if (__any_sync(0xFFFFFFFFu, need_scan)) {
        int c2 = 0;
#pragma unroll 1
        for (int cb = 0; cb < nchunk; cb += 2) {
          float va[32], vb[32];
          __syncwarp();
          tmem_ld32x2(tD + lrow + cb * 32, tD + lrow + cb * 32 + 32, va, vb);
          dt32(cb, va);
          dt32(cb + 1, vb);
#pragma unroll
          for (int e = 0; e < 64; ++e) {
            const float x = e < 32 ? va[e] : vb[e - 32];
            const bool take = need_scan && x <= lim;
            const int sl = c2 < kBand ? c2 : kBand - 1;
            if (take) myl[1 + sl] = (uint8_t)(cb * 32 + e);
            c2 += take ? 1 : 0;
          }
        }
        if (need_scan) n = c2 <= kBand ? c2 : kRecAll;
      }
      myl[0] = (uint8_t)n;
      const int64_t t = (int64_t)tile * 128 + row;
      if (t < a.N) {
        uint8_t* dst = head + L.tiles_off + (int64_t)tile * L.tile_bytes + o_rec + row * 32;
        reinterpret_cast<uint4*>(dst)[0] = reinterpret_cast<const uint4*>(myl)[0];
        reinterpret_cast<uint4*>(dst)[1] = reinterpret_cast<const uint4*>(myl)[1];
      }
      fence_proxy_async_smem();  // the list lived in the A tile, which the next copy overwrites
      tc_fence_before();
      named_bar_sync(1 + g, 128);
      if (flagB[g]) break;
    }
    __syncthreads();
    if (flagA[0] | flagA[1] | flagB[0] | flagB[1]) break;
    s0 = s1;
  }
  if (tid == 0 && (flagA[0] | flagA[1] | flagB[0] | flagB[1]))
    atomicCAS(reinterpret_cast<int*>(a.base), 0, (int)QWM_ERR_TIMEOUT);
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tbase, 512);
  }
}

// ============================================================================
// Kernel 2: exact quantisation, thread = token
// ============================================================================
constexpr int QNT = 128;
template <int R>
struct QSmem {
  static constexpr int K = 0;                                 // token tile, bf16, swizzled
  static constexpr int U = 32768;                             // U [128][R] fp32
  static constexpr int G = U + (R > 0 ? 128 * R * 4 : 0);     // U^T W U [R][R] fp32
  static constexpr int W = G + (R > 0 ? R * R * 4 : 0);       // w [128] fp32
  static constexpr int MISC = W + 512;                        // W_g[4], |U|_F^2 and max w per warp, list count
  static constexpr int RS = MISC + 128;                       // rescoring list: [kRsCap] (row, j) u16
  static constexpr int RSD = RS + 2 * 512;                    //   and their distances, fp32
  static constexpr int BAR = RSD + 4 * 512;
  static constexpr int BYTES = BAR + 64 + 1024;
};

constexpr int kRsCap = 512;             // (token, centroid) pairs rescored together per tile

// Exact Query-aware distance (Eq. 9) in channel order, one fused
// multiply-add per term on the rounded square.
__device__ __forceinline__ float exact_dq(const uint8_t* sK, int row, const __nv_bfloat16* mu, const float* sW) {
  float acc = 0.0f;
#pragma unroll 4
  for (int cc = 0; cc < 8; ++cc) {
    uint32_t mw[8];
    ldg32(mu + cc * 16, mw);
    const uint4 ka = lds16(sK + sw_off(128, row, 2 * cc)), kb = lds16(sK + sw_off(128, row, 2 * cc + 1));
    const uint32_t kw[8] = {ka.x, ka.y, ka.z, ka.w, kb.x, kb.y, kb.z, kb.w};
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


template <int R, int GS>
__global__ void __launch_bounds__(QNT, (R > 16 ? 3 : 4))
    append_quant(const AppendArgs a, const __grid_constant__ CUtensorMap tm_k,
                 const __grid_constant__ CUtensorMap tm_v, int tiles, int units, int nsm, int cps) {
  using S = QSmem<R>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  const Layout& L = a.L;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int H = L.H, C = L.C;
  constexpr int ng = 128 / GS;
  constexpr int RP = R > 0 ? R / 2 : 1;
  const int Mc = a.M;
  const bool all_cand = Mc >= C;

  const uint8_t* sK = sm + S::K;
  float* sU = reinterpret_cast<float*>(sm + S::U);
  float* sG = reinterpret_cast<float*>(sm + S::G);
  float* sW = reinterpret_cast<float*>(sm + S::W);
  float* sMisc = reinterpret_cast<float*>(sm + S::MISC);
  int* sRsCount = reinterpret_cast<int*>(sm + S::MISC + 64);
  uint32_t* sPMask = reinterpret_cast<uint32_t*>(sm + S::MISC + 16);  // the tile's PSAC keep bits, per warp
  uint16_t* sRsPair = reinterpret_cast<uint16_t*>(sm + S::RS);
  float* sRsDq = reinterpret_cast<float*>(sm + S::RSD);
  const uint32_t bar = smem_u32(sm + S::BAR);

  // Work unit u = (side * H + h) * tiles + tile; this CTA takes the
  // contiguous run [u0, u1), so its per-(head, side) setup is redone only
  // where the run crosses into the next head or side, and the head's
  // centroid table stays hot in L1.
  // With one full wave (nsm * cps CTAs), CTA b is taken to run on SM
  // b % nsm, and the cps CTAs of one SM get adjacent runs (one head's table).
  int li = blockIdx.x;
  if ((int)gridDim.x == nsm * cps) li = (li % nsm) * cps + li / nsm;
  const int u0 = (int)((int64_t)li * units / gridDim.x);
  const int u1 = (int)((int64_t)(li + 1) * units / gridDim.x);
  auto issue_tile = [&](int u) {
    const int pr = u / tiles, tl = u - pr * tiles;
    const CUtensorMap* tm = pr < H ? &tm_k : &tm_v;
    mbar_arrive_expect_tx(bar, 32768);
    tma_load_3d(smem_u32(sm + S::K), tm, 0, pr % H, tl * 128, bar);
    tma_load_3d(smem_u32(sm + S::K + 16384), tm, 64, pr % H, tl * 128, bar);
  };
  if (tid == 0) {
    mbar_init(bar, 1);
    fence_mbar_init();
    if (u0 < u1) issue_tile(u0);
  }
  uint32_t ph = 0;
  int cur_pair = -1;
  // A Key or Value or a table value beyond the binary16 range (or not a
  // number) cannot be held by the cache's binary16 operands: reported in the
  // cache's status word as QWM_ERR_NONFINITE once this CTA is done.
  bool nbad = false;

  for (int u = u0; u < u1; ++u) {
    const int pair = u / tiles;
    const int tile = u - pair * tiles, h = pair % H;
    const bool is_key = pair < H;
    const int64_t t = (int64_t)tile * 128 + tid;
    const bool valid = t < a.N;
    const __nv_bfloat16* tab = (is_key ? a.kc : a.vc) + (size_t)h * C * 128;
    const bool use_w = is_key && a.w != nullptr;
    const bool psac = R > 0 && is_key && a.U != nullptr;
    uint8_t* head = a.base + head_offset(L, a.slot, h);
    uint8_t* tb = head + L.tiles_off + (int64_t)tile * L.tile_bytes;
    const __nv_bfloat16* xr = (is_key ? a.k : a.v) + ((size_t)(valid ? t : 0) * H + h) * 128;

    // The chunk's own tables travel with the slot, stored as binary16 (exact
    // for bf16 values in the binary16 range), the operand type of the
    // attention kernel's tensor-core path.
    if (tile == 0) {
      const uint32_t* src = reinterpret_cast<const uint32_t*>(tab);
      __half2* dst = reinterpret_cast<__half2*>(head + (is_key ? L.ktab : L.vtab));
      for (int i = tid; i < C * 64; i += QNT) {
        const uint32_t pr = src[i];
        nbad |= bf16x2_out_of_f16(pr);
        dst[i] = __floats2half2_rn(__uint_as_float(pr << 16), __uint_as_float(pr & 0xFFFF0000u));
      }
      if (psac) {
        __nv_bfloat16* ut = reinterpret_cast<__nv_bfloat16*>(head + L.ut);
        const __nv_bfloat16* Uh = a.U + (size_t)h * 128 * R;
        for (int i = tid; i < R * 128; i += QNT) ut[i] = Uh[(size_t)(i % 128) * R + i / 128];  // U_r^T [r][d]
      }
    }

    // ---- per-(head, side) setup: w, W_g, U (fp32), U^T W U, |U|_F^2, max w
    if (pair != cur_pair) {
      __syncthreads();  // the previous unit's last readers of these arrays are done
      sW[tid] = use_w ? a.w[(size_t)h * 128 + tid] : 1.0f;
      if constexpr (R > 0) {
        if (psac) {
          const __nv_bfloat16* Uh = a.U + (size_t)h * 128 * R;
          for (int i = tid; i < 128 * R; i += QNT) sU[i] = __bfloat162float(Uh[i]);  // [d][r]
        }
      }
      __syncthreads();
      if (tid < ng) {
        float Wg = 0.0f;
        for (int c = tid * GS; c < (tid + 1) * GS; ++c) Wg = __fadd_rn(Wg, sW[c]);
        sMisc[tid] = Wg;
      }
      if constexpr (R > 0) {
        if (psac) {
          // U^T W U (any order; it enters only with its error bound): thread
          // (j, k pair) accumulates two entries over the channels
          for (int e = tid; e < R * RP; e += QNT) {
            const int j = e / RP, kp = e % RP;
            uint64_t acc = 0;
            for (int c = 0; c < 128; ++c) {
              const float uw = sU[c * R + j] * sW[c];
              acc = fma2(f2pack(uw, uw), *reinterpret_cast<const uint64_t*>(sU + c * R + 2 * kp), acc);
            }
            *reinterpret_cast<uint64_t*>(sG + j * R + 2 * kp) = acc;
          }
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
      __syncthreads();
      cur_pair = pair;
    }
    float Wg[4];
#pragma unroll
    for (int gi = 0; gi < 4; ++gi) Wg[gi] = gi < ng ? sMisc[gi] : 0.0f;

    // ---- the filter's record for this token, then the tile
    uint32_t rec[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) rec[i] = 0;
    uint32_t* dcodes = reinterpret_cast<uint32_t*>(tb + (is_key ? L.k_codes : L.v_codes) + tid * 32);
    if (!all_cand && valid) {
      const uint4 r0 = ldg16(dcodes), r1 = ldg16(dcodes + 4);
      rec[0] = r0.x; rec[1] = r0.y; rec[2] = r0.z; rec[3] = r0.w;
      rec[4] = r1.x; rec[5] = r1.y; rec[6] = r1.z; rec[7] = r1.w;
    }
    if (tid == 0) *sRsCount = 0;  // the previous unit's list was last read before a barrier
    const bool ok = mbar_wait(bar, ph);
    ph ^= 1;
    if (__syncthreads_or(!ok)) {
      if (tid == 0) atomicCAS(reinterpret_cast<int*>(a.base), 0, (int)QWM_ERR_TIMEOUT);
      break;
    }

    // ---- part A (reads the tile): candidates, QSAC, INT2 parameters, the
    // channel pass
    int id = 0;
    const __nv_bfloat16* mr = tab;
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

    // ---- 1. candidates: the filter's decided top-M, or an exact rescoring
    // of the band members (every centroid when the band was not listed).
    // Rescoring is done by the whole CTA: each such token reserves a slice
    // of the (token, centroid) list, every thread evaluates list entries,
    // and the owner keeps the M smallest (dQ, j) of its slice.
    int cand[kMaxFilterM];
#pragma unroll
    for (int s = 0; s < kMaxFilterM; ++s) cand[s] = 0;
    bool rescore = false;
    int rs_base = 0, rs_n = 0;
    bool band = false;
    if (valid && !all_cand) {
      auto rb = [&](int i) -> int { return (int)((rec[i >> 2] >> (8 * (i & 3))) & 0xFFu); };
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
        rs_base = atomicAdd(sRsCount, rs_n);
        if (rs_base + rs_n <= kRsCap) {
          for (int m = 0; m < rs_n; ++m) {
            int j = m;
            if (band) {
#pragma unroll
              for (int i = 0; i < kBand; ++i)
                if (i == m) j = rb(1 + i);
            }
            sRsPair[rs_base + m] = (uint16_t)((tid << 8) | j);
          }
        }
      }
    }
    if (__syncthreads_or(rescore)) {
      const int total = min(*sRsCount, kRsCap);
      for (int q = tid; q < total; q += QNT) {
        const int pr = sRsPair[q];
        sRsDq[q] = exact_dq(sK, pr >> 8, tab + (size_t)(pr & 0xFF) * 128, sW);
      }
      __syncthreads();
      if (rescore) {
        float ev[kMaxFilterM];
        int ej[kMaxFilterM];
#pragma unroll
        for (int s = 0; s < kMaxFilterM; ++s) { ev[s] = INFINITY; ej[s] = 0x7FFFFFFF; }
        float ek = INFINITY;
        const bool listed = rs_base + rs_n <= kRsCap;
        for (int m = 0; m < rs_n; ++m) {  // ascending j in both cases
          float dq;
          int j;
          if (listed) {
            j = sRsPair[rs_base + m] & 0xFF;
            dq = sRsDq[rs_base + m];
          } else {
            j = m;
            if (band) {
              auto rb = [&](int i) -> int { return (int)((rec[i >> 2] >> (8 * (i & 3))) & 0xFFu); };
#pragma unroll
              for (int i = 0; i < kBand; ++i)
                if (i == m) j = rb(1 + i);
            }
            dq = exact_dq(sK, tid, tab + (size_t)j * 128, sW);
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

    if (valid) {
      // ---- 2. QSAC score (Eq. 10, 12) of each candidate, lowest (S, j); the
      // group minima / maxima of the chosen residual feed the INT2 step.
      // Candidates are scored QB at a time, channel blocks of 16 outermost, so
      // that each block of the token row is read once per batch and the batch's
      // centroid rows are in flight together (32-byte loads, whole sectors).
      constexpr int QB = 4;
      float bestS = INFINITY;
      int bestj = 0x7FFFFFFF;
      float bmn[4], bmx[4];
    #pragma unroll
      for (int gi = 0; gi < 4; ++gi) { bmn[gi] = 0.0f; bmx[gi] = 0.0f; }
      const int ncand = all_cand ? C : Mc;
      for (int m0 = 0; m0 < ncand; m0 += QB) {
        const int nb = ncand - m0 < QB ? ncand - m0 : QB;
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
        float mx[QB][4], mn[QB][4];
    #pragma unroll
        for (int b = 0; b < QB; ++b)
    #pragma unroll
          for (int gi = 0; gi < 4; ++gi) { mx[b][gi] = -INFINITY; mn[b][gi] = INFINITY; }
    #pragma unroll
        for (int cc = 0; cc < 8; ++cc) {
          const int gi = (cc * 16) / GS;
          const uint4 ka = lds16(sK + sw_off(128, tid, 2 * cc)), kb = lds16(sK + sw_off(128, tid, 2 * cc + 1));
          const uint32_t kw[8] = {ka.x, ka.y, ka.z, ka.w, kb.x, kb.y, kb.z, kb.w};
          uint64_t k2[8];
    #pragma unroll
          for (int p = 0; p < 8; ++p) k2[p] = bf2_to_f2(kw[p]);
    #pragma unroll
          for (int b = 0; b < QB; ++b) {
            if (b < nb) {
              uint32_t mw[8];
              ldg32(tab + (size_t)jb[b] * 128 + cc * 16, mw);
              float x[16];
    #pragma unroll
              for (int p = 0; p < 8; ++p) f2unpack(sub2(k2[p], bf2_to_f2(mw[p])), x[2 * p], x[2 * p + 1]);
    #pragma unroll
              for (int e = 0; e < 16; e += 2) {
                mx[b][gi] = fmax3f(mx[b][gi], x[e], x[e + 1]);
                mn[b][gi] = fmin3(mn[b][gi], x[e], x[e + 1]);
              }
            }
          }
        }
    #pragma unroll
        for (int b = 0; b < QB; ++b) {
          if (b < nb) {
            float Sc = 0.0f;
    #pragma unroll
            for (int gi = 0; gi < ng; ++gi) {
              const float Rg = __fsub_rn(mx[b][gi], mn[b][gi]);
              Sc = __fadd_rn(Sc, __fmul_rn(Wg[gi], __fmul_rn(Rg, Rg)));
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
      mr = tab + (size_t)id * 128;

      // ---- 3. INT2 parameters (Eq. 1-2): range of the residual with 0 included;
      // scale format 1 (App. D.1): s = code * s2 with s2 the binary16 round-up of
      // max_g range_g / 3 / 255 and code the smallest byte covering range_g / 3
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

      // ---- 4. one channel pass: INT2 codes; Keys with PSAC also E (Eq. 4, 13),
      // c = U^T E, v = U^T (w o E) and err0 = sum_c w_c E_c^2, in channel order
      const uint64_t MAG2 = f2pack(kMagic, kMagic);
      uint32_t kmag = 0u;  // the largest |k| bits of each half-word lane
      uint32_t mwn[8];
      ldg32(mr, mwn);
    #pragma unroll 1
      for (int wd = 0; wd < 8; ++wd) {
        const int gi = (wd * 16) / GS;
        const float s = sel4(sc, gi), iv = sel4(inv, gi), z = sel4(zf, gi);
        const uint64_t S2 = f2pack(s, s), Z2 = f2pack(z, z);
        uint32_t word = 0;
        uint32_t mw8[8];
    #pragma unroll
        for (int i = 0; i < 8; ++i) mw8[i] = mwn[i];
        if (wd < 7) ldg32(mr + (wd + 1) * 16, mwn);  // the next word's centroid chunk, one step ahead
    #pragma unroll
        for (int hc = 0; hc < 2; ++hc) {
          const int ch = 2 * wd + hc;
          const uint4 kv = lds16(sK + sw_off(128, tid, ch));
          const uint32_t kw[4] = {kv.x, kv.y, kv.z, kv.w};
          kmag = vmax_u16x2(vmax_u16x2(kmag, kv.x & 0x7FFF7FFFu), vmax_u16x2(kv.y & 0x7FFF7FFFu, kv.z & 0x7FFF7FFFu));
          kmag = vmax_u16x2(kmag, kv.w & 0x7FFF7FFFu);
    #pragma unroll
          for (int p = 0; p < 4; ++p) {
            const uint64_t k2 = bf2_to_f2(kw[p]), m2 = bf2_to_f2(mw8[4 * hc + p]);
            float x0, x1;
            f2unpack(sub2(k2, m2), x0, x1);
            // y = x * (1/s) rounded on its own (the scalar intrinsic is never fused
            // into the following add), then rint(y) in both lanes
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
                const uint4* u0 = reinterpret_cast<const uint4*>(sU + c0 * R);
                const uint4* u1 = reinterpret_cast<const uint4*>(sU + (c0 + 1) * R);
    #pragma unroll
                for (int i = 0; i < RP / 2; ++i) {
                  const uint4 q = u0[i];
                  const uint64_t ua = f2pack(__uint_as_float(q.x), __uint_as_float(q.y));
                  const uint64_t ub = f2pack(__uint_as_float(q.z), __uint_as_float(q.w));
                  cj[2 * i] = fma2(e0, ua, cj[2 * i]);
                  vj[2 * i] = fma2(ua, we0, vj[2 * i]);
                  cj[2 * i + 1] = fma2(e0, ub, cj[2 * i + 1]);
                  vj[2 * i + 1] = fma2(ub, we0, vj[2 * i + 1]);
                }
    #pragma unroll
                for (int i = 0; i < RP / 2; ++i) {
                  const uint4 q = u1[i];
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
      // |k0_c - k_c| <= s/2 (the INT2 round trip), so the rebuilt values stay
      // inside the binary16 operands of attention when max|k| + s/2 does
      {
        const float km = fmaxf(__uint_as_float(kmag << 16), __uint_as_float(kmag & 0xFFFF0000u));
        const float sm = fmaxf(fmaxf(sc[0], sc[1]), fmaxf(sc[2], sc[3]));
        nbad |= bf16x2_out_of_f16(kmag) || !(km + 0.5f * sm < 65504.0f);
      }
    }
    // every read of the tile is done: refill it with the next unit's tokens
    fence_proxy_async_smem();
    __syncthreads();
    if (tid == 0 && u + 1 < u1) issue_tile(u + 1);

    // ---- part B: stores, PSAC
    uint32_t pcw[R > 0 ? R / 4 : 1];  // this token's PSAC codes and row scale when kept (Keys)
#pragma unroll
    for (int i = 0; i < (R > 0 ? R / 4 : 1); ++i) pcw[i] = 0;
    __half psg = __ushort_as_half(0);
    bool pkept = false;
    if (valid) {
      reinterpret_cast<uint4*>(dcodes)[0] = make_uint4(cw[0], cw[1], cw[2], cw[3]);
      reinterpret_cast<uint4*>(dcodes)[1] = make_uint4(cw[4], cw[5], cw[6], cw[7]);
      if (L.sf) {
        uint8_t* dsc = tb + (is_key ? L.k_scales : L.v_scales) + (int64_t)tid * ng;
    #pragma unroll
        for (int gi = 0; gi < ng; ++gi) dsc[gi] = (uint8_t)scode[gi];
        reinterpret_cast<__half*>(tb + (is_key ? L.k_s2 : L.v_s2))[tid] = s2h;
      } else if constexpr (ng == 4) {
        uint2 sv;
        sv.x = (uint32_t)__half_as_ushort(sh[0]) | ((uint32_t)__half_as_ushort(sh[1]) << 16);
        sv.y = (uint32_t)__half_as_ushort(sh[2]) | ((uint32_t)__half_as_ushort(sh[3]) << 16);
        *reinterpret_cast<uint2*>(tb + (is_key ? L.k_scales : L.v_scales) + tid * 8) = sv;
      } else {
        *reinterpret_cast<uint32_t*>(tb + (is_key ? L.k_scales : L.v_scales) + tid * 4) =
            (uint32_t)__half_as_ushort(sh[0]) | ((uint32_t)__half_as_ushort(sh[1]) << 16);
      }
      tb[(is_key ? L.k_ids : L.v_ids) + tid] = (uint8_t)id;
      {
        uint8_t* dz = tb + (is_key ? L.k_zeros : L.v_zeros) + (int64_t)tid * L.zb;
        dz[0] = (uint8_t)zbyte;
        for (int b = 1; b < L.zb; ++b) dz[b] = 0;
      }

      // ---- 5. PSAC coefficients (Eq. 13, INT8 with a binary16 row scale) and
      // the keep rule (Eq. 16), Keys only
      if constexpr (R > 0) {
        if (is_key) {
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
              for (int i = 0; i < QNT / 32; ++i) {
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
                float errq = 0.0f, e0 = 0.0f;
    #pragma unroll 1
                for (int wd = 0; wd < 8; ++wd) {
                  const int gi = (wd * 16) / GS;
                  const float s = sel4(sc, gi), z = sel4(zf, gi);
                  uint32_t word = cw[0];
    #pragma unroll
                  for (int i = 1; i < 8; ++i)
                    if (i == wd) word = cw[i];
    #pragma unroll
                  for (int hc = 0; hc < 2; ++hc) {
                    const int ch = 2 * wd + hc;
                    const uint4 kv = ldg16(xr + ch * 8);
                    const uint4 mv = ldg16(mr + ch * 8);
                    const uint32_t kw[4] = {kv.x, kv.y, kv.z, kv.w}, mw[4] = {mv.x, mv.y, mv.z, mv.w};
    #pragma unroll
                    for (int e = 0; e < 8; ++e) {
                      const int c = ch * 8 + e;
                      const float kf = __uint_as_float((e & 1) ? (kw[e >> 1] & 0xFFFF0000u) : (kw[e >> 1] << 16));
                      const float mf = __uint_as_float((e & 1) ? (mw[e >> 1] & 0xFFFF0000u) : (mw[e >> 1] << 16));
                      const int j16 = 8 * hc + e;
                      const float q = (float)((word >> (16 * (j16 & 1) + 2 * (j16 >> 1))) & 3u);
                      const float E = __fsub_rn(kf, __fadd_rn(mf, __fmul_rn(__fsub_rn(q, z), s)));
                      float u = 0.0f;
    #pragma unroll
                      for (int j = 0; j < R; ++j) u = __fmaf_rn(sU[c * R + j], chat[j], u);
                      const float ep = __fsub_rn(E, u);
                      errq = __fmaf_rn(sW[c], __fmul_rn(ep, ep), errq);
                      e0 = __fmaf_rn(sW[c], __fmul_rn(E, E), e0);
                    }
                  }
                }
                keep = errq < e0;
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
    }

    // ---- 6. the tile's PSAC rows in the smaller of the two layouts (App.
    // D.1): dense (every token's row, dropped corrections as zeros) or
    // sparse (only the kept rows, compacted in token order), with the tile's
    // 128-bit keep mask naming the rows stored (row i is entry
    // popcount(mask below i)).
    if constexpr (R > 0) {
      if (is_key) {
        const uint32_t wm = __ballot_sync(0xFFFFFFFFu, pkept);
        if (lane == 0) sPMask[warp] = wm;
        __syncthreads();
        uint32_t m4[4] = {sPMask[0], sPMask[1], sPMask[2], sPMask[3]};
        const int nt = (int)((a.N - (int64_t)tile * 128) < 128 ? (a.N - (int64_t)tile * 128) : 128);
        const int Kt = __popc(m4[0]) + __popc(m4[1]) + __popc(m4[2]) + __popc(m4[3]);
        const bool sparse = 16 + Kt * (R + 2) < nt * (R + 2);
        int e = tid;
        if (sparse) {
          e = __popc(m4[warp] & ((1u << lane) - 1u));
#pragma unroll
          for (int w4 = 0; w4 < 3; ++w4) e += w4 < warp ? __popc(m4[w4]) : 0;
        } else {
#pragma unroll
          for (int w4 = 0; w4 < 4; ++w4) {
            const int nb = nt - 32 * w4;
            m4[w4] = nb >= 32 ? 0xFFFFFFFFu : (nb > 0 ? (1u << nb) - 1u : 0u);
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
        if (tid == 0)
          *reinterpret_cast<uint4*>(head + L.pmask + (int64_t)tile * 16) = make_uint4(m4[0], m4[1], m4[2], m4[3]);
      }
    }
  }
  if (nbad) atomicCAS(reinterpret_cast<int*>(a.base), 0, (int)QWM_ERR_NONFINITE);
}

// ============================================================================
// Host side
// ============================================================================
template <int R, int GS>
cudaError_t launch_quant(const AppendArgs& a, const CUtensorMap& tk, const CUtensorMap& tv, cudaStream_t st) {
  constexpr int smem = QSmem<R>::BYTES;
  cudaError_t e = cudaFuncSetAttribute(append_quant<R, GS>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  int dev = 0, nsm = 0, cps = 0;
  e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
  if (e == cudaSuccess) e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&cps, append_quant<R, GS>, QNT, smem);
  if (e != cudaSuccess) return e;
  const int tiles = (int)((a.N + 127) / 128);
  const int units = tiles * a.L.H * 2;
  const int slots = nsm * (cps > 0 ? cps : 1);
  const unsigned grid = (unsigned)(units < slots ? units : slots);  // persistent: one wave
  append_quant<R, GS><<<grid, QNT, smem, st>>>(a, tk, tv, tiles, units, nsm, cps > 0 ? cps : 1);
  return cudaGetLastError();
}
template <int R>
cudaError_t launch_quant_r(const AppendArgs& a, const CUtensorMap& tk, const CUtensorMap& tv, cudaStream_t st) {
  return a.L.G == 32 ? launch_quant<R, 32>(a, tk, tv, st) : launch_quant<R, 64>(a, tk, tv, st);
}

}  // namespace

cudaError_t launch_append(const AppendArgs& a, cudaStream_t st) {
  if (a.M > kMaxFilterM && a.M < a.L.C) return launch_append_generic(a, st);
  if (!a.Mq || a.M >= a.L.C) return launch_append_fused(a, st);
  // The Keys' candidates by the full quadratic form (App. C.4): the filter,
  // the rescoring of its undecided rows, then the quantize kernel.
  alignas(64) CUtensorMap tk, tv;
  if (!make_token_map(&tk, a.k, a.N, a.L.H, 128) || !make_token_map(&tv, a.v, a.N, a.L.H, 128))
    return cudaErrorInvalidValue;
  int dev = 0, nsm = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return e;
  auto kern = a.M == 4 ? append_filter<5, true> : (a.M == 1 ? append_filter<2, true>
                  : (a.M == 2 ? append_filter<3, true> : append_filter<kMaxFilterM + 1, true>));
  e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, F_SMEM);
  if (e != cudaSuccess) return e;
  const int tiles = (int)((a.N + 127) / 128);
  const int units = 2 * a.L.H * tiles;
  const int grid = units < nsm ? units : nsm;
  kern<<<grid, FNT, F_SMEM, st>>>(a, tk, tv, tiles, units);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  e = launch_full_rescore(a, st);
  if (e != cudaSuccess) return e;
  switch (a.L.r) {
    case 0: return launch_quant_r<0>(a, tk, tv, st);
    case 8: return launch_quant_r<8>(a, tk, tv, st);
    case 16: return launch_quant_r<16>(a, tk, tv, st);
    case 32: return launch_quant_r<32>(a, tk, tv, st);
  }
  return cudaErrorInvalidValue;
}

}  // namespace qwm
