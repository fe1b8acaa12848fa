// attend.cu -- attention of new queries over the packed 2-bit cache and the
// active bf16 chunk, on the sm_103a tensor cores (tcgen05 + TMEM).
//
// Per CTA: 128 queries of one head.  For every 128-key tile of every cached
// chunk the CTA
//   1. rebuilds K_hat0 = mu_id + s (q - z) (Sec. 2 Eq. 4) in shared memory as an
//      f16 MMA operand (128-byte swizzled, K-major), plus r extra columns
//      C_hat = t * sigma of the PSAC coefficients (Sec. 4.2 Eq. 16),
//   2. issues S = [Q | Q U_r] [K_hat0 | C_hat]^T on tcgen05 into TMEM: the
//      PSAC logit correction Q U_r C^T (Eq. 17) rides along as r extra
//      reduction columns, with Q U_r of the chunk's own U_r computed once per
//      chunk into the extra columns of the Q operand,
//   3. rebuilds V_hat (same reconstruction, no PSAC) while the MMA runs,
//   4. runs the online softmax on its TMEM row (thread = query row; the O
//      accumulator is rescaled only when the running maximum grows by more
//      than 2^8, which keeps every P <= 2^8), writes P as bf16 operand,
//   5. issues O += P V_hat on tcgen05 into TMEM.
// The active chunk's dense bf16 K/V tiles run through the same loop without
// the PSAC columns.  MMA operands are binary16 (11 significant bits; the
// bf16 inputs convert exactly) with fp32 accumulation: same tensor rate as
// bf16, but 8x finer rounding of the rebuilt keys, which keeps the logits of
// outlier channels accurate.  Inputs must stay inside the binary16 range.  All mbarrier waits are bounded; a wait that runs out
// records QWM_ERR_TIMEOUT in the cache's status word and the CTA leaves.
#include "ptx_sm103.cuh"
#include "qwm_internal.cuh"

namespace qwm {
namespace {

using namespace ptx;

constexpr int NT = 128;
constexpr float kTauLog2 = 8.0f;
constexpr int BLK = 16384;  // one 128-row x 128-byte swizzled operand block
constexpr int OFF_Q = 0;                 // 3 blocks: Q[:, 0:64], Q[:, 64:128], Q U_r
constexpr int OFF_K = OFF_Q + 3 * BLK;   // 3 blocks: K_hat[:, 0:64], [:, 64:128], C_hat
constexpr int OFF_V = OFF_K + 3 * BLK;   // 2 blocks: V_hat[:, 0:64], [:, 64:128]
constexpr int OFF_P = OFF_V + 2 * BLK;   // 2 blocks: P[:, 0:64], [:, 64:128]
constexpr int OFF_UT = OFF_P + 2 * BLK;  // U_r^T [r][128] bf16 (8 KB)
constexpr int OFF_BAR = OFF_UT + 8192;
constexpr int SMEM_BYTES = OFF_BAR + 64 + 1024;  // + alignment slack

// Store 8 bf16 (16 bytes) of row `row`, chunk `ch` (columns 8ch..8ch+7) into
// a sequence of 128-byte-swizzled blocks of 128 rows x 64 columns.
__device__ __forceinline__ void st_chunk(uint8_t* base, int row, int ch, uint4 v) {
  const int kb = ch >> 3, pos = (ch & 7) ^ (row & 7);
  *reinterpret_cast<uint4*>(base + kb * BLK + row * 128 + pos * 16) = v;
}

__device__ __forceinline__ uint4 ldg16(const void* p) { return __ldg(reinterpret_cast<const uint4*>(p)); }

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// K_hat0 or V_hat row `row` of a packed tile into swizzled shared memory.
__device__ __forceinline__ void dequant_row(uint8_t* dst, int row, const uint8_t* tb, int64_t o_codes,
                                            int64_t o_scales, int64_t o_ids, int64_t o_zeros, int zb, int ng,
                                            int gshift, const uint8_t* tab) {
  const uint4 c0 = ldg16(tb + o_codes + row * 32);
  const uint4 c1 = ldg16(tb + o_codes + row * 32 + 16);
  const uint32_t cw[8] = {c0.x, c0.y, c0.z, c0.w, c1.x, c1.y, c1.z, c1.w};
  const int id = tb[o_ids + row];
  const uint32_t zbyte = tb[o_zeros + (int64_t)row * zb];
  const __half* sp = reinterpret_cast<const __half*>(tb + o_scales + (int64_t)row * ng * 2);
  float sc[4];
#pragma unroll
  for (int g = 0; g < 4; ++g) sc[g] = g < ng ? __half2float(sp[g]) : 0.0f;
  const uint8_t* mu = tab + (int64_t)id * 256;
#pragma unroll
  for (int ch = 0; ch < 16; ++ch) {
    const int g = (ch * 8) >> gshift;
    const float s = sc[g];
    const float zf = (float)((zbyte >> (2 * g)) & 3u);
    const uint32_t bits = (cw[ch >> 1] >> ((ch & 1) * 16)) & 0xFFFFu;
    const uint4 m = ldg16(mu + ch * 16);
    const uint32_t mw[4] = {m.x, m.y, m.z, m.w};
    uint32_t ow[4];
#pragma unroll
    for (int p = 0; p < 4; ++p) {
      const float q0 = (float)((bits >> (4 * p)) & 3u), q1 = (float)((bits >> (4 * p + 2)) & 3u);
      const float v0 = __uint_as_float(mw[p] << 16) + (q0 - zf) * s;
      const float v1 = __uint_as_float(mw[p] & 0xFFFF0000u) + (q1 - zf) * s;
      ow[p] = pack_f16(v0, v1);
    }
    st_chunk(dst, row, ch, make_uint4(ow[0], ow[1], ow[2], ow[3]));
  }
}

__device__ __forceinline__ void zero_row(uint8_t* dst, int row, int nch) {
  for (int ch = 0; ch < nch; ++ch) st_chunk(dst, row, ch, make_uint4(0, 0, 0, 0));
}

__device__ __forceinline__ void copy_row(uint8_t* dst, int row, const __nv_bfloat16* src) {
#pragma unroll
  for (int ch = 0; ch < 16; ++ch) st_chunk(dst, row, ch, bf16x8_to_f16x8(ldg16(src + ch * 8)));
}

__global__ void __launch_bounds__(NT, 1) attend_kernel(const AttendArgs a, const AttendSlots S) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  const Layout& L = a.L;
  const int tid = threadIdx.x, warp = tid >> 5;
  const int h = blockIdx.y;
  const int H = L.H, r = L.r;
  const int rpad = r == 8 ? 16 : r;
  const int gshift = L.G == 32 ? 5 : 6;
  const int64_t qi = (int64_t)blockIdx.x * 128 + tid;
  const bool qvalid = qi < a.Nq;

  uint8_t* sQ = sm + OFF_Q;
  uint8_t* sK = sm + OFF_K;
  uint8_t* sV = sm + OFF_V;
  uint8_t* sP = sm + OFF_P;
  __nv_bfloat16* sUt = reinterpret_cast<__nv_bfloat16*>(sm + OFF_UT);
  const uint32_t barS = smem_u32(sm + OFF_BAR), barO = barS + 8;
  uint32_t* tslot = reinterpret_cast<uint32_t*>(sm + OFF_BAR + 16);

  if (warp == 0) {
    tmem_alloc(smem_u32(tslot), 256);
    tmem_relinquish();
  }
  if (tid == 0) {
    mbar_init(barS, 1);
    mbar_init(barO, 1);
    fence_mbar_init();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tbase = *tslot;
  const uint32_t tS = tbase, tO = tbase + 128;
  const uint32_t lrow = (uint32_t)(warp * 32) << 16;  // this warp's TMEM lanes

  // Q tile, row = thread
  const __nv_bfloat16* qrow = a.q + ((size_t)(qvalid ? qi : 0) * H + h) * 128;
  if (qvalid) copy_row(sQ, tid, qrow);
  else zero_row(sQ, tid, 16);
  if (r > 0) zero_row(sQ + 2 * BLK, tid, rpad / 8);

  const uint32_t aQ = smem_u32(sQ), aK = smem_u32(sK), aV = smem_u32(sV), aP = smem_u32(sP);
  constexpr uint32_t idS = idesc_f16(128, 128, false);
  constexpr uint32_t idPV = idesc_f16(128, 64, true);
  const float sl2 = a.sm_scale * 1.4426950408889634f;

  float m_run = -INFINITY, l_run = 0.0f;
  uint32_t phS = 0, phO = 0;
  bool o_init = false, aborted = false;
  bool pv_pending = false;  // a committed P V_hat MMA not yet waited for

  const int n_units = S.n + (a.Ncur > 0 ? 1 : 0);
  for (int u = 0; u < n_units && !aborted; ++u) {
    const bool dense = (u == S.n);
    const int ntok = dense ? (int)a.Ncur : S.tokens[u];
    const uint8_t* hb = dense ? nullptr : a.base + head_offset(L, S.slot[u], h);
    const bool psac = !dense && S.psac[u] && r > 0;
    if (psac) {
      // Q U_r of this chunk's basis into the extra operand columns (Eq. 17).
      __syncthreads();  // previous readers of sUt are done
      for (int i = tid; i < r * 16; i += NT)
        reinterpret_cast<uint4*>(sUt)[i] = ldg16(hb + L.ut + (int64_t)i * 16);
      __syncthreads();
      float acc[32];
#pragma unroll
      for (int j = 0; j < 32; ++j) acc[j] = 0.0f;
      if (qvalid) {
        for (int ch = 0; ch < 16; ++ch) {
          const uint4 qv = ldg16(qrow + ch * 8);
          const uint32_t qw[4] = {qv.x, qv.y, qv.z, qv.w};
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            const float qf = __uint_as_float(e & 1 ? (qw[e >> 1] & 0xFFFF0000u) : (qw[e >> 1] << 16));
            const int c = ch * 8 + e;
#pragma unroll
            for (int j = 0; j < 32; ++j)
              if (j < r) acc[j] = fmaf(qf, __bfloat162float(sUt[j * 128 + c]), acc[j]);
          }
        }
      }
#pragma unroll
      for (int c2 = 0; c2 < 4; ++c2) {
        if (c2 * 8 >= rpad) break;
        uint32_t w4[4];
#pragma unroll
        for (int p = 0; p < 4; ++p) {
          const int j = c2 * 8 + 2 * p;
          w4[p] = pack_f16(j < r ? acc[j] : 0.0f, j + 1 < r ? acc[j + 1] : 0.0f);
        }
        st_chunk(sQ + 2 * BLK, tid, c2, make_uint4(w4[0], w4[1], w4[2], w4[3]));
      }
    }

    const int ntiles = (ntok + 127) / 128;
    for (int tl = 0; tl < ntiles; ++tl) {
      const int nvalid = min(128, ntok - tl * 128);
      const bool rvalid = tid < nvalid;
      const uint8_t* tb = dense ? nullptr : hb + L.tiles_off + (int64_t)tl * L.tile_bytes;
      // ---- K_hat tile (row = key)
      if (dense) {
        if (rvalid) copy_row(sK, tid, a.kcur + ((size_t)(tl * 128 + tid) * H + h) * 128);
        else zero_row(sK, tid, 16);
      } else {
        if (rvalid) dequant_row(sK, tid, tb, L.k_codes, L.k_scales, L.k_ids, L.k_zeros, L.zb, L.ng, gshift, hb + L.ktab);
        else zero_row(sK, tid, 16);
        if (psac) {
          if (rvalid) {
            const int8_t* cp = reinterpret_cast<const int8_t*>(tb + L.k_coef + (int64_t)tid * r);
            const float sg = __half2float(*reinterpret_cast<const __half*>(tb + L.k_sigma + tid * 2));
            for (int c2 = 0; c2 * 8 < rpad; ++c2) {
              uint32_t w4[4];
#pragma unroll
              for (int p = 0; p < 4; ++p) {
                const int j = c2 * 8 + 2 * p;
                const float t0 = j < r ? (float)cp[j] * sg : 0.0f;
                const float t1 = j + 1 < r ? (float)cp[j + 1] * sg : 0.0f;
                w4[p] = pack_f16(t0, t1);
              }
              st_chunk(sK + 2 * BLK, tid, c2, make_uint4(w4[0], w4[1], w4[2], w4[3]));
            }
          } else {
            zero_row(sK + 2 * BLK, tid, rpad / 8);
          }
        }
      }
      fence_proxy_async_smem();
      tc_fence_before();
      __syncthreads();
      if (tid == 0) {
        tc_fence_after();
#pragma unroll
        for (int kb = 0; kb < 2; ++kb)
#pragma unroll
          for (int ks = 0; ks < 4; ++ks)
            umma_bf16(tS, desc_sw128(aQ + kb * BLK + ks * 32), desc_sw128(aK + kb * BLK + ks * 32), idS,
                      (kb | ks) != 0);
        if (psac)
          for (int ks = 0; ks < rpad / 16; ++ks)
            umma_bf16(tS, desc_sw128(aQ + 2 * BLK + ks * 32), desc_sw128(aK + 2 * BLK + ks * 32), idS, 1u);
        umma_commit(barS);
      }
      bool fail = false;
      // ---- the previous P V_hat MMA must finish before V_hat, P and O are reused
      if (pv_pending) {
        fail |= !mbar_wait(barO, phO);
        phO ^= 1u;
        pv_pending = false;
        tc_fence_after();
      }
      // ---- V_hat tile
      if (dense) {
        if (rvalid) copy_row(sV, tid, a.vcur + ((size_t)(tl * 128 + tid) * H + h) * 128);
        else zero_row(sV, tid, 16);
      } else {
        if (rvalid) dequant_row(sV, tid, tb, L.v_codes, L.v_scales, L.v_ids, L.v_zeros, L.zb, L.ng, gshift, hb + L.vtab);
        else zero_row(sV, tid, 16);
      }
      // ---- logits ready
      fail |= !mbar_wait(barS, phS);
      phS ^= 1u;
      tc_fence_after();
      fail = __any_sync(0xFFFFFFFFu, fail);  // tcgen05.ld below is warp-collective
      if (!fail) {
        // online softmax on this thread's row (Eq. 5 logits times sm_scale)
        float mt = -INFINITY;
        float v[32];
#pragma unroll
        for (int cb = 0; cb < 4; ++cb) {
          tmem_ld32(tS + lrow + cb * 32, v);
#pragma unroll
          for (int e = 0; e < 32; ++e)
            if (cb * 32 + e < nvalid) mt = fmaxf(mt, v[e]);
        }
        const float m_new = fmaxf(m_run, mt);
        const bool need = (m_new - m_run) * sl2 > kTauLog2;
        float alpha = 1.0f;
        if (need) {
          alpha = ex2((m_run - m_new) * sl2);
          m_run = m_new;
          l_run *= alpha;
        }
        if (__any_sync(0xFFFFFFFFu, need) && o_init) {
#pragma unroll
          for (int cb = 0; cb < 4; ++cb) {
            tmem_ld32(tO + lrow + cb * 32, v);
#pragma unroll
            for (int e = 0; e < 32; ++e) v[e] *= alpha;
            tmem_st32(tO + lrow + cb * 32, v);
          }
        }
        const float mb = m_run * sl2;
        float lsum = 0.0f;
#pragma unroll
        for (int cb = 0; cb < 4; ++cb) {
          tmem_ld32(tS + lrow + cb * 32, v);
          uint32_t pk[16];
#pragma unroll
          for (int e = 0; e < 32; e += 2) {
            const float p0 = (cb * 32 + e < nvalid) ? ex2(v[e] * sl2 - mb) : 0.0f;
            const float p1 = (cb * 32 + e + 1 < nvalid) ? ex2(v[e + 1] * sl2 - mb) : 0.0f;
            lsum += p0 + p1;
            pk[e >> 1] = pack_f16(p0, p1);
          }
#pragma unroll
          for (int k = 0; k < 4; ++k)
            st_chunk(sP, tid, cb * 4 + k, make_uint4(pk[4 * k], pk[4 * k + 1], pk[4 * k + 2], pk[4 * k + 3]));
        }
        l_run += lsum;
      }
      fence_proxy_async_smem();
      tc_fence_before();
      if (__syncthreads_or(fail)) {
        aborted = true;
        break;
      }
      if (tid == 0) {
        tc_fence_after();
#pragma unroll
        for (int ks = 0; ks < 8; ++ks) {
          const uint64_t ad = desc_sw128(aP + (ks >> 2) * BLK + (ks & 3) * 32);
#pragma unroll
          for (int nh = 0; nh < 2; ++nh)
            umma_bf16(tO + nh * 64, ad, desc_sw128(aV + nh * BLK + ks * 2048), idPV,
                      (o_init || ks > 0) ? 1u : 0u);
        }
        umma_commit(barO);
      }
      o_init = true;
      pv_pending = true;
    }
  }

  bool ok = !aborted;
  if (pv_pending) {
    ok = mbar_wait(barO, phO) && ok;
    tc_fence_after();
  }
  ok = __syncthreads_and(ok);
  if (ok) {
    const float inv_l = 1.0f / l_run;
    float v[32];
#pragma unroll
    for (int cb = 0; cb < 4; ++cb) {
      tmem_ld32(tO + lrow + cb * 32, v);
      if (qvalid) {
        uint4* dst = reinterpret_cast<uint4*>(a.out + ((size_t)qi * H + h) * 128 + cb * 32);
#pragma unroll
        for (int k = 0; k < 4; ++k)
          dst[k] = make_uint4(pack_bf16(v[8 * k] * inv_l, v[8 * k + 1] * inv_l),
                              pack_bf16(v[8 * k + 2] * inv_l, v[8 * k + 3] * inv_l),
                              pack_bf16(v[8 * k + 4] * inv_l, v[8 * k + 5] * inv_l),
                              pack_bf16(v[8 * k + 6] * inv_l, v[8 * k + 7] * inv_l));
      }
    }
    if (a.lse && qvalid) a.lse[(size_t)h * a.Nq + qi] = m_run * a.sm_scale + logf(l_run);
  } else if (tid == 0) {
    atomicCAS(a.status, 0, (int)QWM_ERR_TIMEOUT);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tbase, 256);
  }
}

}  // namespace

cudaError_t launch_attend(const AttendArgs& a, const AttendSlots& slots, cudaStream_t st) {
  cudaError_t e = cudaFuncSetAttribute(attend_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES);
  if (e != cudaSuccess) return e;
  dim3 grid((unsigned)((a.Nq + 127) / 128), (unsigned)a.L.H);
  attend_kernel<<<grid, NT, SMEM_BYTES, st>>>(a, slots);
  return cudaGetLastError();
}

}  // namespace qwm
