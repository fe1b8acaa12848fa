// append.cu -- quantize-on-append with a tensor-core distance filter.
//
// Per CTA: 128 new tokens of one head, Keys (blockIdx.z = 0) or Values (1);
// thread = token.  Steps (Sec. 4.1 QSAC, Sec. 2 Eq. 1-4 INT2, Sec. 4.2 PSAC):
//   1. Candidate filter on tcgen05: D = K (w o mu)^T for all C centroids in
//      one f16 MMA into TMEM, so that dQ_j - sum_c w_c k_c^2 = A_j - 2 D_j
//      with A_j = sum_c w_c mu_jc^2 (Eq. 9 expanded).  The f16 rounding of
//      w o mu and the fp32 accumulation give an error below
//      B = 2^-9 |k| max_j |w o mu_j| + 2^-15 max_j A_j + 2^-18 (|k| + ...)
//      (a bound with a 4x margin over the f16 rounding term), so every
//      centroid among the true top-M lies within 2B of the M-th smallest
//      filtered distance.  When exactly M centroids fall inside that band
//      they are the top-M; otherwise the band members are rescored with the
//      exact Query-aware distance (fp32, channel order) and the M smallest
//      (ties to the lower index) kept.
//   2. QSAC score (Eq. 10, 12) of each candidate, INT2 residual quantisation
//      and packing, and for Keys the PSAC coefficients with the keep rule, all
//      with explicitly rounded fp32 operations in channel order, identical to
//      a sequential evaluation of the formulas.
// M >= C skips the filter (every centroid is a candidate); 8 < M < C goes to
// the generic kernel (append_generic.cu).
#include "ptx_sm103.cuh"
#include "qwm_internal.cuh"

namespace qwm {
namespace {

using namespace ptx;

constexpr int NT = 128;        // threads = tokens per CTA
constexpr int kMaxFilterM = 8;
constexpr int kBand = 16;      // band members rescored exactly before falling back to all C

constexpr int OFF_A = 0;                          // K tile, f16, 2 blocks of 128 x 128 B
constexpr int OFF_B = 32768;                      // w o mu, f16, 2 blocks of Npad x 128 B
constexpr int OFF_AJ = OFF_B + 65536;             // A_j [256] fp32
constexpr int OFF_W = OFF_AJ + 1024;              // w [128]
constexpr int OFF_WG = OFF_W + 512;               // W_g [4]
constexpr int OFF_RED = OFF_WG + 16;              // [4 warps][2] maxima
constexpr int OFF_U = OFF_RED + 48;               // U [128][r] bf16 (<= 8 KB)
constexpr int OFF_LIST = OFF_U + 8192;            // band lists [128][16] u8
constexpr int OFF_BAR = OFF_LIST + NT * kBand;    // mbarrier + TMEM slot
constexpr int SMEM_BYTES = OFF_BAR + 64 + 1024;   // + alignment slack

__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }
__device__ __forceinline__ uint4 ldg16(const void* p) { return __ldg(reinterpret_cast<const uint4*>(p)); }

// Swizzled 16-byte store into K-major operand blocks of `rows` rows.
__device__ __forceinline__ void st_chunk_rows(uint8_t* base, int rows, int row, int ch, uint4 v) {
  const int kb = ch >> 3, pos = (ch & 7) ^ (row & 7);
  *reinterpret_cast<uint4*>(base + (size_t)kb * rows * 128 + row * 128 + pos * 16) = v;
}

__device__ __forceinline__ void unpack8(const uint4 v, float (&f)[8]) {
  f[0] = bf_lo(v.x); f[1] = bf_hi(v.x); f[2] = bf_lo(v.y); f[3] = bf_hi(v.y);
  f[4] = bf_lo(v.z); f[5] = bf_hi(v.z); f[6] = bf_lo(v.w); f[7] = bf_hi(v.w);
}
__device__ __forceinline__ float sel4(const float (&a)[4], int g) {
  return g == 0 ? a[0] : (g == 1 ? a[1] : (g == 2 ? a[2] : a[3]));
}
__device__ __forceinline__ int sel4i(const int (&a)[4], int g) {
  return g == 0 ? a[0] : (g == 1 ? a[1] : (g == 2 ? a[2] : a[3]));
}

// Exact Query-aware distance (Eq. 9) in channel order: xr is the token row,
// mu the centroid row (bf16), sW the weights.
__device__ __forceinline__ float exact_dq(const __nv_bfloat16* xr, const __nv_bfloat16* mu, const float* sW) {
  float acc = 0.0f;
#pragma unroll 1
  for (int ch = 0; ch < 16; ++ch) {
    float kf[8], mf[8];
    unpack8(ldg16(xr + ch * 8), kf);
    unpack8(ldg16(mu + ch * 8), mf);
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      const float t = __fsub_rn(kf[e], mf[e]);
      acc = __fadd_rn(acc, __fmul_rn(sW[ch * 8 + e], __fmul_rn(t, t)));
    }
  }
  return acc;
}

// Insert (v, j) into the ascending list of the Mc smallest (value, index)
// pairs; indices arrive in ascending order, so an equal value stays behind.
__device__ __forceinline__ void insert_top(float (&tv)[kMaxFilterM], int (&tj)[kMaxFilterM], int Mc, float v, int j) {
#pragma unroll
  for (int s = 0; s < kMaxFilterM; ++s) {
    if (s < Mc && v < tv[s]) {
      const float ov = tv[s];
      const int oj = tj[s];
      tv[s] = v;
      tj[s] = j;
      v = ov;
      j = oj;
    }
  }
}
__device__ __forceinline__ float kth_of(const float (&tv)[kMaxFilterM], int Mc) {
  float k = tv[0];
#pragma unroll
  for (int s = 1; s < kMaxFilterM; ++s)
    if (s == Mc - 1) k = tv[s];
  return k;
}

template <int R, int GS>
__global__ void __launch_bounds__(NT, 2) append_kernel(const AppendArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  const Layout& L = a.L;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int h = blockIdx.y;
  const bool is_key = blockIdx.z == 0;
  const int64_t t = (int64_t)blockIdx.x * NT + tid;
  const bool valid = t < a.N;
  const int C = L.C, H = L.H;
  constexpr int r = R, G = GS, ng = 128 / GS;
  const int Mc = a.M;
  const bool all_cand = Mc >= C;
  const int Npad = (C + 15) & ~15;
  const __nv_bfloat16* x = is_key ? a.k : a.v;
  const __nv_bfloat16* tab = (is_key ? a.kc : a.vc) + (size_t)h * C * 128;
  const bool use_w = is_key && a.w != nullptr;
  const bool psac = is_key && a.U != nullptr && r > 0;
  uint8_t* head = a.base + head_offset(L, a.slot, h);

  float* sAj = reinterpret_cast<float*>(sm + OFF_AJ);
  float* sW = reinterpret_cast<float*>(sm + OFF_W);
  float* sWg = reinterpret_cast<float*>(sm + OFF_WG);
  float* sRed = reinterpret_cast<float*>(sm + OFF_RED);
  __nv_bfloat16* sU = reinterpret_cast<__nv_bfloat16*>(sm + OFF_U);
  uint8_t* myl = sm + OFF_LIST + tid * kBand;
  const uint32_t bar = smem_u32(sm + OFF_BAR);
  uint32_t* tslot = reinterpret_cast<uint32_t*>(sm + OFF_BAR + 16);

  // The chunk's own tables travel with the slot (one CTA per head and K/V),
  // stored as binary16 (exact for bf16 values in the binary16 range), the
  // operand type of the attention kernel's tensor-core path.
  if (blockIdx.x == 0) {
    const uint32_t* src = reinterpret_cast<const uint32_t*>(tab);
    __half2* dst = reinterpret_cast<__half2*>(head + (is_key ? L.ktab : L.vtab));
    for (int i = tid; i < C * 64; i += NT) {
      const uint32_t pr = src[i];
      dst[i] = __floats2half2_rn(bf_lo(pr), bf_hi(pr));
    }
    if (psac) {
      __nv_bfloat16* ut = reinterpret_cast<__nv_bfloat16*>(head + L.ut);
      const __nv_bfloat16* Uh = a.U + (size_t)h * 128 * r;
      for (int i = tid; i < r * 128; i += NT) ut[i] = Uh[(size_t)(i % 128) * r + i / 128];  // U_r^T [r][d]
    }
  }

  if (!all_cand && warp == 0) {
    tmem_alloc(smem_u32(tslot), 256);
    tmem_relinquish();
  }
  if (tid == 0) {
    mbar_init(bar, 1);
    fence_mbar_init();
  }
  sW[tid] = use_w ? a.w[(size_t)h * 128 + tid] : 1.0f;
  if (psac)
    for (int i = tid; i < 128 * r; i += NT) sU[i] = a.U[(size_t)h * 128 * r + i];  // [d][r]
  __syncthreads();
  if (tid < ng) {
    float Wg = 0.0f;
    for (int c = tid * G; c < (tid + 1) * G; ++c) Wg = __fadd_rn(Wg, sW[c]);
    sWg[tid] = Wg;
  }

  // ---- this thread's f16 operand row and |k|^2
  const __nv_bfloat16* xr = x + ((size_t)(valid ? t : 0) * H + h) * 128;
  float knorm2 = 0.0f;
  if (!all_cand) {
#pragma unroll 4
    for (int ch = 0; ch < 16; ++ch) {
      const uint4 v = valid ? ldg16(xr + ch * 8) : make_uint4(0, 0, 0, 0);
      st_chunk_rows(sm + OFF_A, 128, tid, ch, bf16x8_to_f16x8(v));
      float kf[8];
      unpack8(v, kf);
#pragma unroll
      for (int e = 0; e < 8; ++e) knorm2 = fmaf(kf[e], kf[e], knorm2);
    }
  }

  uint32_t tD = 0;
  float bandB = 0.0f;
  if (!all_cand) {
    // ---- w o mu rows (f16 operand B), A_j and the norms for the bound
    float wmax2 = 0.0f, amax = 0.0f;
    for (int j = tid; j < Npad; j += NT) {
      float A = 0.0f, n2 = 0.0f;
      if (j < C) {
        const __nv_bfloat16* mr = tab + (size_t)j * 128;
#pragma unroll 4
        for (int ch = 0; ch < 16; ++ch) {
          const uint4 m = ldg16(mr + ch * 8);
          const uint32_t mw[4] = {m.x, m.y, m.z, m.w};
          uint32_t ow[4];
#pragma unroll
          for (int p = 0; p < 4; ++p) {
            const float m0 = bf_lo(mw[p]), m1 = bf_hi(mw[p]);
            const float w0 = __fmul_rn(sW[ch * 8 + 2 * p], m0), w1 = __fmul_rn(sW[ch * 8 + 2 * p + 1], m1);
            A = fmaf(w0, m0, fmaf(w1, m1, A));
            n2 = fmaf(w0, w0, fmaf(w1, w1, n2));
            ow[p] = pack_f16(w0, w1);
          }
          st_chunk_rows(sm + OFF_B, Npad, j, ch, make_uint4(ow[0], ow[1], ow[2], ow[3]));
        }
        sAj[j] = A;
      } else {
#pragma unroll
        for (int ch = 0; ch < 16; ++ch) st_chunk_rows(sm + OFF_B, Npad, j, ch, make_uint4(0, 0, 0, 0));
        sAj[j] = INFINITY;
      }
      wmax2 = fmaxf(wmax2, n2);
      amax = fmaxf(amax, fabsf(A));
    }
#pragma unroll
    for (int off = 16; off; off >>= 1) {
      wmax2 = fmaxf(wmax2, __shfl_xor_sync(0xFFFFFFFFu, wmax2, off));
      amax = fmaxf(amax, __shfl_xor_sync(0xFFFFFFFFu, amax, off));
    }
    if (lane == 0) {
      sRed[2 * warp] = wmax2;
      sRed[2 * warp + 1] = amax;
    }
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    tD = *tslot;
    if (tid == 0) {
      const uint32_t aA = smem_u32(sm + OFF_A), aB = smem_u32(sm + OFF_B);
      const uint32_t id = idesc_f16(128, Npad, false);
#pragma unroll
      for (int kb = 0; kb < 2; ++kb)
#pragma unroll
        for (int ks = 0; ks < 4; ++ks)
          umma_ss(tD, desc_sw128(aA + kb * 16384 + ks * 32), desc_sw128(aB + kb * Npad * 128 + ks * 32), id,
                  (kb | ks) != 0);
      umma_commit(bar);
    }
    float W2 = 0.0f, Am = 0.0f;
#pragma unroll
    for (int i = 0; i < NT / 32; ++i) {
      W2 = fmaxf(W2, sRed[2 * i]);
      Am = fmaxf(Am, sRed[2 * i + 1]);
    }
    const float kn = sqrtf(knorm2), Wn = sqrtf(W2);
    bandB = ldexpf(kn * Wn, -9) + ldexpf(Am, -15) + ldexpf(kn + Wn + 1.0f, -18);
  }

  // ---- 1. candidates
  int ncand = 0;  // candidates in myl (all_cand: every centroid)
  bool timeout = false;
  if (!all_cand) {
    const bool ok = __all_sync(0xFFFFFFFFu, mbar_wait(bar, 0));
    if (!ok) {
      timeout = true;
    } else {
      tc_fence_after();
      const uint32_t lrow = (uint32_t)(warp * 32) << 16;
      float tv[kMaxFilterM];
      int tj[kMaxFilterM];
#pragma unroll
      for (int s = 0; s < kMaxFilterM; ++s) { tv[s] = INFINITY; tj[s] = 0x7FFFFFFF; }
      float kth = INFINITY;
      float v[32];
      for (int cb = 0; cb * 32 < Npad; ++cb) {
        tmem_ld32(tD + lrow + cb * 32, v);
#pragma unroll
        for (int e = 0; e < 32; ++e) {
          const int j = cb * 32 + e;
          if (j < C) {
            const float dt = fmaf(-2.0f, v[e], sAj[j]);
            if (dt < kth) {
              insert_top(tv, tj, Mc, dt, j);
              kth = kth_of(tv, Mc);
            }
          }
        }
      }
      const float thr = kth + 2.0f * bandB;
      int nb = 0;
      for (int cb = 0; cb * 32 < Npad; ++cb) {
        tmem_ld32(tD + lrow + cb * 32, v);
#pragma unroll
        for (int e = 0; e < 32; ++e) {
          const int j = cb * 32 + e;
          if (j < C && fmaf(-2.0f, v[e], sAj[j]) <= thr) {
            if (nb < kBand) myl[nb] = (uint8_t)j;
            ++nb;
          }
        }
      }
      if (valid) {
        if (nb == Mc) {
          ncand = Mc;
        } else {
          // rescore exactly: the band members, or every centroid if the band overflowed
          float ev[kMaxFilterM];
          int ej[kMaxFilterM];
#pragma unroll
          for (int s = 0; s < kMaxFilterM; ++s) { ev[s] = INFINITY; ej[s] = 0x7FFFFFFF; }
          float ek = INFINITY;
          const int n_eval = nb <= kBand ? nb : C;
          for (int m = 0; m < n_eval; ++m) {
            const int j = nb <= kBand ? myl[m] : m;
            const float dq = exact_dq(xr, tab + (size_t)j * 128, sW);
            if (dq < ek) {
              insert_top(ev, ej, Mc, dq, j);
              ek = kth_of(ev, Mc);
            }
          }
#pragma unroll
          for (int s = 0; s < kMaxFilterM; ++s)
            if (s < Mc) myl[s] = (uint8_t)ej[s];
          ncand = Mc;
        }
      }
    }
  } else {
    ncand = C;
  }

  // ---- 2. QSAC score over the candidates (Eq. 10, 12), lowest (S, j)
  if (valid && !timeout) {
    float bestS = INFINITY;
    int bestj = 0x7FFFFFFF;
    for (int m = 0; m < ncand; ++m) {
      const int j = all_cand ? m : myl[m];
      const __nv_bfloat16* mr = tab + (size_t)j * 128;
      float mx[4], mn[4];
#pragma unroll
      for (int g = 0; g < 4; ++g) { mx[g] = -INFINITY; mn[g] = INFINITY; }
#pragma unroll
      for (int ch = 0; ch < 16; ++ch) {
        float kf[8], mf[8];
        unpack8(ldg16(xr + ch * 8), kf);
        unpack8(ldg16(mr + ch * 8), mf);
        const int g = (ch * 8) / G;
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const float rc = __fsub_rn(kf[e], mf[e]);
          mx[g] = fmaxf(mx[g], rc);
          mn[g] = fminf(mn[g], rc);
        }
      }
      float S = 0.0f;
#pragma unroll
      for (int g = 0; g < 4; ++g) {
        if (g < ng) {
          const float Rg = __fsub_rn(mx[g], mn[g]);
          S = __fadd_rn(S, __fmul_rn(sWg[g], __fmul_rn(Rg, Rg)));
        }
      }
      if (S < bestS || (S == bestS && j < bestj)) { bestS = S; bestj = j; }
    }
    const int id = bestj < C ? bestj : C - 1;
    const __nv_bfloat16* mr = tab + (size_t)id * 128;

    // ---- 3. INT2 residual quantisation (Eq. 1-2) of x = k - mu_id
    float lo[4], hi[4];
#pragma unroll
    for (int g = 0; g < 4; ++g) { lo[g] = 0.0f; hi[g] = 0.0f; }
#pragma unroll
    for (int ch = 0; ch < 16; ++ch) {
      float kf[8], mf[8];
      unpack8(ldg16(xr + ch * 8), kf);
      unpack8(ldg16(mr + ch * 8), mf);
      const int g = (ch * 8) / G;
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        const float xc = __fsub_rn(kf[e], mf[e]);
        lo[g] = fminf(lo[g], xc);
        hi[g] = fmaxf(hi[g], xc);
      }
    }
    float sc[4], inv[4];
    int zq[4];
    __half sh[4];
    uint32_t zbyte = 0;
#pragma unroll
    for (int g = 0; g < 4; ++g) {
      sc[g] = 0.0f; inv[g] = 0.0f; zq[g] = 0; sh[g] = __ushort_as_half(0);
      if (g < ng) {
        sh[g] = __float2half_ru(__fdiv_rn(__fsub_rn(hi[g], lo[g]), 3.0f));
        sc[g] = __half2float(sh[g]);
        if (sc[g] != 0.0f) {
          inv[g] = __frcp_rn(sc[g]);
          const int z = (int)rintf(__fmul_rn(-lo[g], inv[g]));
          zq[g] = z < 0 ? 0 : (z > 3 ? 3 : z);
        }
        zbyte |= (uint32_t)zq[g] << (2 * g);
      }
    }
    const int64_t tile = t / kTile;
    const int rowi = (int)(t % kTile);
    uint8_t* tb = head + L.tiles_off + tile * L.tile_bytes;
    uint32_t* dcodes = reinterpret_cast<uint32_t*>(tb + (is_key ? L.k_codes : L.v_codes) + rowi * 32);
    // 16 channels per word: even channel 2k at bits 2k, odd channel 2k+1 at 16 + 2k
#pragma unroll 1
    for (int wd = 0; wd < 8; ++wd) {
      uint32_t word = 0;
#pragma unroll
      for (int hc = 0; hc < 2; ++hc) {
        const int ch = 2 * wd + hc;
        float kf[8], mf[8];
        unpack8(ldg16(xr + ch * 8), kf);
        unpack8(ldg16(mr + ch * 8), mf);
        const int g = (ch * 8) / G;
        const float s = sel4(sc, g), iv = sel4(inv, g);
        const int z = sel4i(zq, g);
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const float xc = __fsub_rn(kf[e], mf[e]);
          int q = 0;
          if (s != 0.0f) {
            q = (int)rintf(__fmul_rn(xc, iv)) + z;
            q = q < 0 ? 0 : (q > 3 ? 3 : q);
          }
          const int j16 = 8 * hc + e;
          word |= (uint32_t)q << (16 * (j16 & 1) + 2 * (j16 >> 1));
        }
      }
      dcodes[wd] = word;
    }
    __half* dsc = reinterpret_cast<__half*>(tb + (is_key ? L.k_scales : L.v_scales) + (int64_t)rowi * ng * 2);
#pragma unroll
    for (int g = 0; g < 4; ++g)
      if (g < ng) dsc[g] = sh[g];
    tb[(is_key ? L.k_ids : L.v_ids) + rowi] = (uint8_t)id;
    uint8_t* dz = tb + (is_key ? L.k_zeros : L.v_zeros) + (int64_t)rowi * L.zb;
    dz[0] = (uint8_t)zbyte;
    for (int b = 1; b < L.zb; ++b) dz[b] = 0;

    // ---- 4. PSAC (Eq. 13, 16) with the keep rule, Keys only
    if constexpr (R > 0) {
      if (is_key) {
        int8_t* coef = reinterpret_cast<int8_t*>(tb + L.k_coef + (int64_t)rowi * R);
        __half* sig = reinterpret_cast<__half*>(tb + L.k_sigma) + rowi;
        if (!psac) {
#pragma unroll
          for (int j = 0; j < R; ++j) coef[j] = 0;
          *sig = __ushort_as_half(0);
        } else {
          // E_c = k_c - k0_c, k0_c = mu_c + s (q_c - z); q_c re-read from the packed word
          float cj[R];
#pragma unroll
          for (int j = 0; j < R; ++j) cj[j] = 0.0f;
#pragma unroll 1
          for (int ch = 0; ch < 16; ++ch) {
            float kf[8], mf[8];
            unpack8(ldg16(xr + ch * 8), kf);
            unpack8(ldg16(mr + ch * 8), mf);
            const int g = (ch * 8) / G;
            const float s = sel4(sc, g);
            const int z = sel4i(zq, g);
            const uint32_t word = dcodes[ch >> 1];
#pragma unroll
            for (int e = 0; e < 8; ++e) {
              const int j16 = 8 * (ch & 1) + e;
              const int q = (word >> (16 * (j16 & 1) + 2 * (j16 >> 1))) & 3;
              const float E = __fsub_rn(kf[e], __fadd_rn(mf[e], __fmul_rn((float)(q - z), s)));
              const __nv_bfloat16* ur = sU + (ch * 8 + e) * R;
#pragma unroll
              for (int j = 0; j < R; ++j) cj[j] = __fadd_rn(cj[j], __fmul_rn(E, __bfloat162float(ur[j])));
            }
          }
          float amax = 0.0f;
#pragma unroll
          for (int j = 0; j < R; ++j) amax = fmaxf(amax, fabsf(cj[j]));
          const __half sgh = __float2half_ru(__fdiv_rn(amax, 127.0f));
          const float sg = __half2float(sgh);
          const float sinv = sg != 0.0f ? __frcp_rn(sg) : 0.0f;
#pragma unroll
          for (int j = 0; j < R; ++j) {  // cj becomes chat = t * sigma
            const float qq = sg != 0.0f ? fminf(fmaxf(rintf(__fmul_rn(cj[j], sinv)), -127.0f), 127.0f) : 0.0f;
            cj[j] = __fmul_rn(qq, sg);
          }
          // keep only if sum_c w_c (E_c - (U chat)_c)^2 < sum_c w_c E_c^2, both in channel order
          float errq = 0.0f, err0 = 0.0f;
#pragma unroll 1
          for (int ch = 0; ch < 16; ++ch) {
            float kf[8], mf[8];
            unpack8(ldg16(xr + ch * 8), kf);
            unpack8(ldg16(mr + ch * 8), mf);
            const int g = (ch * 8) / G;
            const float s = sel4(sc, g);
            const int z = sel4i(zq, g);
            const uint32_t word = dcodes[ch >> 1];
#pragma unroll
            for (int e = 0; e < 8; ++e) {
              const int c = ch * 8 + e;
              const int j16 = 8 * (ch & 1) + e;
              const int q = (word >> (16 * (j16 & 1) + 2 * (j16 >> 1))) & 3;
              const float E = __fsub_rn(kf[e], __fadd_rn(mf[e], __fmul_rn((float)(q - z), s)));
              const __nv_bfloat16* ur = sU + c * R;
              float u = 0.0f;
#pragma unroll
              for (int j = 0; j < R; ++j) u = __fadd_rn(u, __fmul_rn(__bfloat162float(ur[j]), cj[j]));
              const float ep = __fsub_rn(E, u);
              errq = __fadd_rn(errq, __fmul_rn(sW[c], __fmul_rn(ep, ep)));
              err0 = __fadd_rn(err0, __fmul_rn(sW[c], __fmul_rn(E, E)));
            }
          }
          const bool keep = errq < err0;
#pragma unroll
          for (int j = 0; j < R; ++j) coef[j] = keep ? (int8_t)(int)rintf(__fmul_rn(cj[j], sinv)) : (int8_t)0;
          *sig = keep ? sgh : __ushort_as_half(0);
        }
      }
    }
  }
  if (timeout && tid == 0) atomicCAS(reinterpret_cast<int*>(a.base), 0, (int)QWM_ERR_TIMEOUT);

  if (!all_cand) {
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
      tc_fence_after();
      tmem_dealloc(tD, 256);
    }
  }
}

template <int R, int GS>
cudaError_t launch_rg(const AppendArgs& a, cudaStream_t st) {
  cudaError_t e = cudaFuncSetAttribute(append_kernel<R, GS>, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES);
  if (e != cudaSuccess) return e;
  dim3 grid((unsigned)((a.N + NT - 1) / NT), (unsigned)a.L.H, 2);
  append_kernel<R, GS><<<grid, NT, SMEM_BYTES, st>>>(a);
  return cudaGetLastError();
}
template <int R>
cudaError_t launch_r(const AppendArgs& a, cudaStream_t st) {
  return a.L.G == 32 ? launch_rg<R, 32>(a, st) : launch_rg<R, 64>(a, st);
}

}  // namespace

cudaError_t launch_append(const AppendArgs& a, cudaStream_t st) {
  if (a.M > kMaxFilterM && a.M < a.L.C) return launch_append_generic(a, st);
  switch (a.L.r) {
    case 0: return launch_r<0>(a, st);
    case 8: return launch_r<8>(a, st);
    case 16: return launch_r<16>(a, st);
    case 32: return launch_r<32>(a, st);
  }
  return cudaErrorInvalidValue;
}

}  // namespace qwm
