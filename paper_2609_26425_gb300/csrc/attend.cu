// attend.cu -- attention of new queries over the packed 2-bit cache and the
// active bf16 chunk, on the sm_103a tensor cores (tcgen05 + TMEM).
//
// Per CTA: 256 queries (two 128-row Q tiles) of one head, 17 warps with fixed
// roles that hand work to each other through mbarriers:
//   warps 0-3, 4-7   softmax of Q tile 0 / 1: thread = query row; reads its
//                    logit row S_i from TMEM, keeps the running max and sum,
//                    writes P_i as f16 back into the same TMEM columns, and
//                    at chunk boundaries computes Q U_r of the next chunk
//                    (Sec. 4.2 Eq. 17) into the extra Q operand columns;
//   warps 8-11       rebuild K_hat0 = mu_id + s (q - z) (Sec. 2 Eq. 4) of each
//                    128-key tile into a 2-stage shared-memory ring, plus the
//                    r PSAC columns C_hat = t * sigma (Eq. 16);
//   warps 12-15      rebuild V_hat (same reconstruction, no PSAC) into a
//                    second 2-stage ring;
//   warp 16          allocates TMEM and issues every MMA from one thread:
//                    S_i = [Q_i | Q_i U_r] [K_hat0 | C_hat]^T (the PSAC logit
//                    term rides along as extra reduction columns) and
//                    O_i += P_i V_hat with P_i read straight from TMEM.
// TMEM (512 columns): S0 | S1 | O0 | O1, 128 fp32 columns each; P_i aliases
// the first 64 columns of S_i.  MMAs of one thread execute in issue order, so
// S_i of the next tile never overtakes the P_i V_hat MMA that reads P_i.
// The O accumulator is rescaled only when the running maximum grows by more
// than 2^8 (every P stays <= 2^8).  Operands are binary16 with fp32
// accumulation: the bf16 rate with 8x finer rounding of the rebuilt keys.
// Every mbarrier wait is bounded; a wait that runs out records
// QWM_ERR_TIMEOUT in the cache's status word and that role leaves its loop.
#include "ptx_sm103.cuh"
#include "qwm_internal.cuh"

namespace qwm {
namespace {

using namespace ptx;

constexpr int kWarps = 17;
constexpr int NT = kWarps * 32;
constexpr int W_DQV = 12, W_MMA = 16;
constexpr float kTauLog2 = 8.0f;
constexpr int BLK = 16384;               // 128 rows x 128 bytes, 128-byte swizzled
constexpr int OFF_Q = 0;                 // Q0 (2 blocks), Q1 (2 blocks)
constexpr int OFF_QU = 4 * BLK;          // Q_i U_r at columns [i*rpad, (i+1)*rpad)
constexpr int OFF_K = 5 * BLK;           // K_hat0 stage 0, 1 (2 blocks each)
constexpr int OFF_C = 9 * BLK;           // C_hat of stage s at columns [s*rpad, (s+1)*rpad)
constexpr int OFF_V = 10 * BLK;          // V_hat stage 0, 1 (2 blocks each)
constexpr int OFF_BAR = 14 * BLK;
enum { B_KFULL = 0, B_KEMPTY = 2, B_VFULL = 4, B_VEMPTY = 6, B_SFULL = 8, B_PFULL = 10, B_QU = 12, B_OFINAL = 14,
       NBAR = 15 };
constexpr int SMEM_BYTES = OFF_BAR + 256 + 1024;  // + alignment slack

// 8 f16 (16 bytes) of row `row`, chunk `ch` (columns 8ch..8ch+7) into a run of
// 128-byte-swizzled blocks of 128 rows x 64 columns.
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

__device__ __forceinline__ uint32_t ex2_f16x2(uint32_t x) {
  uint32_t y;
  asm("ex2.approx.f16x2 %0, %1;" : "=r"(y) : "r"(x));
  return y;
}
// (a, b) = (a, b) * (s, s) + (c, c) as one packed f32x2 fma.
__device__ __forceinline__ void fma2(float& a, float& b, uint64_t ss, uint64_t cc) {
  uint64_t x;
  asm("mov.b64 %0, {%1, %2};" : "=l"(x) : "f"(a), "f"(b));
  asm("fma.rn.f32x2 %0, %0, %1, %2;" : "+l"(x) : "l"(ss), "l"(cc));
  asm("mov.b64 {%0, %1}, %2;" : "=f"(a), "=f"(b) : "l"(x));
}
__device__ __forceinline__ uint64_t splat2(float a) {
  uint64_t x;
  asm("mov.b64 %0, {%1, %1};" : "=l"(x) : "f"(a));
  return x;
}
// acc + (low half of h2 as f16), acc + (high half), in one mixed-precision add each.
__device__ __forceinline__ float add_f16lo(float acc, uint32_t h2) {
  float r;
  asm("{\n\t.reg .f16 lo, hi;\n\tmov.b32 {lo, hi}, %1;\n\tadd.rn.f32.f16 %0, lo, %2;\n\t}" : "=f"(r) : "r"(h2), "f"(acc));
  return r;
}
__device__ __forceinline__ float add_f16hi(float acc, uint32_t h2) {
  float r;
  asm("{\n\t.reg .f16 lo, hi;\n\tmov.b32 {lo, hi}, %1;\n\tadd.rn.f32.f16 %0, hi, %2;\n\t}" : "=f"(r) : "r"(h2), "f"(acc));
  return r;
}
__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float m;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(m) : "f"(a), "f"(b), "f"(c));
  return m;
}

// 32-byte read-only global load (address 32-byte aligned).
__device__ __forceinline__ void ldg32B(const void* p, uint32_t (&r)[8]) {
  asm volatile("ld.global.nc.v8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7])
               : "l"(p));
}

__device__ __forceinline__ uint32_t h2u(__half2 h) { return *reinterpret_cast<uint32_t*>(&h); }
__device__ __forceinline__ __half2 u2h(uint32_t u) { return *reinterpret_cast<__half2*>(&u); }

// The packed fields of one cache row, loaded one tile ahead of their use so
// that their latency overlaps the rebuild of the current tile.
struct RowPack {
  uint4 c0, c1;   // 128 INT2 codes
  uint32_t idz;   // centroid id | zero-point byte << 8
  uint2 sc;       // group scales (binary16), d/G <= 4 of them
  uint4 cf0, cf1; // PSAC INT8 codes (Keys, r <= 32)
  uint32_t sg;    // PSAC row scale (binary16 bits)
};

__device__ __forceinline__ RowPack load_pack(const uint8_t* tb, int row, int64_t o_codes, int64_t o_scales,
                                             int64_t o_ids, int64_t o_zeros, int zb, int ng, bool with_psac,
                                             int64_t o_coef, int64_t o_sigma, int r) {
  RowPack p;
  p.c0 = ldg16(tb + o_codes + row * 32);
  p.c1 = ldg16(tb + o_codes + row * 32 + 16);
  p.idz = (uint32_t)tb[o_ids + row] | ((uint32_t)tb[o_zeros + (int64_t)row * zb] << 8);
  const uint8_t* sp = tb + o_scales + (int64_t)row * ng * 2;
  p.sc = ng == 4 ? __ldg(reinterpret_cast<const uint2*>(sp)) : make_uint2(__ldg(reinterpret_cast<const uint32_t*>(sp)), 0u);
  p.cf0 = make_uint4(0, 0, 0, 0);
  p.cf1 = make_uint4(0, 0, 0, 0);
  p.sg = 0;
  if (with_psac) {
    const uint8_t* cp = tb + o_coef + (int64_t)row * r;
    if (r == 8) {
      const uint2 v = __ldg(reinterpret_cast<const uint2*>(cp));
      p.cf0 = make_uint4(v.x, v.y, 0, 0);
    } else {
      p.cf0 = ldg16(cp);
      if (r == 32) p.cf1 = ldg16(cp + 16);
    }
    p.sg = __ldg(reinterpret_cast<const unsigned short*>(tb + o_sigma + row * 2));
  }
  return p;
}

// One row of K_hat0 or V_hat: mu_id + s_g (q - z_g), computed as packed f16
// pairs: the two codes of channels (2k, 2k+1) sit at bits 2k and 16 + 2k of
// their 16-channel word, so (word >> 2k) & 0x00030003 | 0x64006400 is the f16
// pair (1024 + q, 1024 + q'), (1024 + q) - (1024 + z) = q - z exactly, and one
// f16 fma adds the centroid with a single rounding.  The table is binary16.
__device__ __forceinline__ void dequant_row(uint8_t* dst, int row, const RowPack& p, int ng, int gshift,
                                            const uint8_t* tab) {
  const uint32_t cw[8] = {p.c0.x, p.c0.y, p.c0.z, p.c0.w, p.c1.x, p.c1.y, p.c1.z, p.c1.w};
  const uint32_t zbyte = (p.idz >> 8) & 0xFFu;
  const uint32_t sw[2] = {p.sc.x, p.sc.y};
  __half2 s2[4], z2[4];
#pragma unroll
  for (int g = 0; g < 4; ++g) {
    const uint32_t sbits = g < ng ? ((sw[g >> 1] >> (16 * (g & 1))) & 0xFFFFu) : 0u;
    s2[g] = u2h(sbits | (sbits << 16));
    const uint32_t zz = 0x6400u | ((zbyte >> (2 * g)) & 3u);
    z2[g] = u2h(zz | (zz << 16));
  }
  const uint8_t* mu = tab + (int64_t)(p.idz & 0xFFu) * 256;
#pragma unroll
  for (int half = 0; half < 2; ++half) {
    uint4 mrow[8];  // half a centroid row in flight at once
#pragma unroll
    for (int i = 0; i < 8; ++i) mrow[i] = ldg16(mu + (half * 8 + i) * 16);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int ch = half * 8 + i;
      const int g = (ch * 8) >> gshift;
      const uint32_t word = cw[ch >> 1];
      const uint32_t mw[4] = {mrow[i].x, mrow[i].y, mrow[i].z, mrow[i].w};
      uint32_t ow[4];
#pragma unroll
      for (int q2 = 0; q2 < 4; ++q2) {
        const int k = 4 * (ch & 1) + q2;
        const uint32_t qq = ((word >> (2 * k)) & 0x00030003u) | 0x64006400u;
        ow[q2] = h2u(__hfma2(__hsub2(u2h(qq), z2[g]), s2[g], u2h(mw[q2])));
      }
      st_chunk(dst, row, ch, make_uint4(ow[0], ow[1], ow[2], ow[3]));
    }
  }
}

__device__ __forceinline__ void zero_row(uint8_t* dst, int row, int ch0, int nch) {
  for (int ch = ch0; ch < ch0 + nch; ++ch) st_chunk(dst, row, ch, make_uint4(0, 0, 0, 0));
}

__device__ __forceinline__ void copy_row(uint8_t* dst, int row, const __nv_bfloat16* src) {
#pragma unroll
  for (int ch = 0; ch < 16; ++ch) st_chunk(dst, row, ch, bf16x8_to_f16x8(ldg16(src + ch * 8)));
}

struct Unit {
  int ntok;
  const uint8_t* hb;  // head block of the slot (cached chunk) or null (active chunk)
  bool psac;
};

__device__ __forceinline__ Unit unit_at(const AttendArgs& a, const AttendSlots& S, int u, int h) {
  Unit x;
  if (u < S.n) {
    x.ntok = S.tokens[u];
    x.hb = a.base + head_offset(a.L, S.slot[u], h);
    x.psac = S.psac[u] && a.L.r > 0;
  } else {
    x.ntok = (int)a.Ncur;
    x.hb = nullptr;
    x.psac = false;
  }
  return x;
}

// Walks the KV tiles of every unit (cached chunks in order, then the active
// chunk) in the order all roles process them.
struct TileCursor {
  int u, tl, n_units, ntiles;
  Unit U;
  __device__ __forceinline__ void init(const AttendArgs& a, const AttendSlots& S, int h, int nu) {
    u = 0; tl = 0; n_units = nu; ntiles = 0;
    if (nu > 0) { U = unit_at(a, S, 0, h); ntiles = (U.ntok + 127) / 128; }
  }
  __device__ __forceinline__ bool valid() const { return u < n_units; }
  __device__ __forceinline__ void next(const AttendArgs& a, const AttendSlots& S, int h) {
    if (++tl >= ntiles) {
      tl = 0;
      if (++u < n_units) { U = unit_at(a, S, u, h); ntiles = (U.ntok + 127) / 128; }
    }
  }
  __device__ __forceinline__ int nvalid() const { return min(128, U.ntok - tl * 128); }
};

// Q_i U_r of one query row (fp32 sums of bf16 products), as f16 into the
// shared Q U_r block at columns [i*rpad, i*rpad + rpad).
__device__ __forceinline__ void write_qu(uint8_t* sQU, int i, int row, bool qvalid, const __nv_bfloat16* qrow,
                                         const uint8_t* ut, int r, int rpad) {
  float acc[32];
#pragma unroll
  for (int j = 0; j < 32; ++j) acc[j] = 0.0f;
  if (qvalid) {
    for (int ch = 0; ch < 16; ++ch) {
      const uint4 qv = ldg16(qrow + ch * 8);
      const uint32_t qw[4] = {qv.x, qv.y, qv.z, qv.w};
      float qf[8];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        qf[2 * e] = __uint_as_float(qw[e] << 16);
        qf[2 * e + 1] = __uint_as_float(qw[e] & 0xFFFF0000u);
      }
#pragma unroll
      for (int j = 0; j < 32; ++j) {
        if (j < r) {
          const uint4 uv = ldg16(ut + ((int64_t)j * 128 + ch * 8) * 2);
          const uint32_t uw[4] = {uv.x, uv.y, uv.z, uv.w};
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            acc[j] = fmaf(qf[2 * e], __uint_as_float(uw[e] << 16), acc[j]);
            acc[j] = fmaf(qf[2 * e + 1], __uint_as_float(uw[e] & 0xFFFF0000u), acc[j]);
          }
        }
      }
    }
  }
#pragma unroll
  for (int c2 = 0; c2 < 4; ++c2) {
    if (c2 * 8 < rpad) {
      uint32_t w4[4];
#pragma unroll
      for (int p = 0; p < 4; ++p) {
        const int j = c2 * 8 + 2 * p;
        w4[p] = pack_f16(j < r ? acc[j] : 0.0f, j + 1 < r ? acc[j + 1] : 0.0f);
      }
      st_chunk(sQU, row, (i * rpad) / 8 + c2, make_uint4(w4[0], w4[1], w4[2], w4[3]));
    }
  }
}

__global__ void __launch_bounds__(NT, 1) attend_kernel(const AttendArgs a, const AttendSlots S) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  const Layout& L = a.L;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int h = blockIdx.y;
  const int H = L.H, r = L.r;
  const int rpad = r == 8 ? 16 : r;
  const int gshift = L.G == 32 ? 5 : 6;
  const int64_t q0 = (int64_t)blockIdx.x * 256;
  const int n_units = S.n + (a.Ncur > 0 ? 1 : 0);

  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + OFF_BAR);
  uint32_t* tslot = reinterpret_cast<uint32_t*>(sm + OFF_BAR + NBAR * 8);
  int* s_err = reinterpret_cast<int*>(sm + OFF_BAR + NBAR * 8 + 8);
  auto bar = [&](int i) { return smem_u32(bars + i); };

  if (warp == W_MMA) {
    tmem_alloc(smem_u32(tslot), 512);
    tmem_relinquish();
  }
  if (tid == 0) {
    for (int s = 0; s < 2; ++s) {
      mbar_init(bar(B_KFULL + s), 128);
      mbar_init(bar(B_KEMPTY + s), 1);
      mbar_init(bar(B_VFULL + s), 128);
      mbar_init(bar(B_VEMPTY + s), 1);
      mbar_init(bar(B_SFULL + s), 1);
      mbar_init(bar(B_PFULL + s), 128);
      mbar_init(bar(B_QU + s), 128);
    }
    mbar_init(bar(B_OFINAL), 1);
    *s_err = 0;
    fence_mbar_init();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tbase = *tslot;

  if (warp < 8) {
    // ------------------------------------------------------------ softmax
    const int i = warp >> 2;
    const int row = tid & 127;
    const int64_t qi = q0 + 128 * i + row;
    const bool qvalid = qi < a.Nq;
    const uint32_t lrow = (uint32_t)((warp & 3) * 32) << 16;
    const uint32_t tS = tbase + 128 * i + lrow, tO = tbase + 256 + 128 * i + lrow;
    const __nv_bfloat16* qrow = a.q + ((size_t)(qvalid ? qi : 0) * H + h) * 128;
    uint8_t* sQi = sm + OFF_Q + i * 2 * BLK;
    if (qvalid) copy_row(sQi, row, qrow);
    else zero_row(sQi, row, 0, 16);
    if (n_units > 0) {
      const Unit u0 = unit_at(a, S, 0, h);
      if (u0.psac) write_qu(sm + OFF_QU, i, row, qvalid, qrow, u0.hb + L.ut, r, rpad);
    }
    fence_proxy_async_smem();
    mbar_arrive(bar(B_QU + i));

    const float sl2 = a.sm_scale * 1.4426950408889634f;
    float m_run = -INFINITY, l_run = 0.0f;
    uint32_t jt = 0;
    bool ok = true;
    for (int u = 0; u < n_units && ok; ++u) {
      const Unit U = unit_at(a, S, u, h);
      const int ntiles = (U.ntok + 127) / 128;
      for (int tl = 0; tl < ntiles; ++tl, ++jt) {
        const int nvalid = min(128, U.ntok - tl * 128);
        ok = __all_sync(0xFFFFFFFFu, mbar_wait(bar(B_SFULL + i), jt & 1));
        if (!ok) break;
        tc_fence_after();
        // ---- row maximum: the four 32-column blocks of S_i, two loads per wait
        float va[32], vb[32];
        float mt = -INFINITY;
#pragma unroll
        for (int cp = 0; cp < 2; ++cp) {
          tmem_ld32x2(tS + 64 * cp, tS + 64 * cp + 32, va, vb);
          if (nvalid == 128) {
#pragma unroll
            for (int e = 0; e < 32; e += 2) {
              mt = fmax3(mt, va[e], va[e + 1]);
              mt = fmax3(mt, vb[e], vb[e + 1]);
            }
          } else {
#pragma unroll
            for (int e = 0; e < 32; ++e) {
              if (64 * cp + e < nvalid) mt = fmaxf(mt, va[e]);
              if (64 * cp + 32 + e < nvalid) mt = fmaxf(mt, vb[e]);
            }
          }
        }
        const float m_new = fmaxf(m_run, mt);
        const bool need = (m_new - m_run) * sl2 > kTauLog2;
        float alpha = 1.0f;
        if (need) {
          alpha = ex2((m_run - m_new) * sl2);
          m_run = m_new;
          l_run *= alpha;
        }
        // S_i of this tile completing implies the previous P_i V MMA is done,
        // so O_i can be rescaled here.
        if (__any_sync(0xFFFFFFFFu, need) && jt > 0) {
#pragma unroll
          for (int cb = 0; cb < 4; ++cb) {
            tmem_ld32(tO + cb * 32, va);
#pragma unroll
            for (int e = 0; e < 32; ++e) va[e] *= alpha;
            tmem_st32(tO + cb * 32, va);
          }
        }
        // ---- P = exp2(s * scale * log2(e) - m) as f16 pairs (one MUFU op per
        // pair), written over the S columns already read; the row sum adds
        // exactly those f16 values, 32 at a time in a packed f16 tree (each
        // partial <= 32 * 2^8, exact to 2^-11 relative), then in fp32.
        const float mb = m_run * sl2;
        const uint64_t SL = splat2(sl2), MB = splat2(-mb);
        float lsum = 0.0f;
        auto exp_block = [&](const float (&v)[32], uint32_t (&pk)[16], int col0, bool full) {
#pragma unroll
          for (int e = 0; e < 32; e += 2) {
            float x0 = v[e], x1 = v[e + 1];
            fma2(x0, x1, SL, MB);
            if (!full) {
              if (col0 + e >= nvalid) x0 = -INFINITY;
              if (col0 + e + 1 >= nvalid) x1 = -INFINITY;
            }
            pk[e >> 1] = ex2_f16x2(pack_f16(x0, x1));
          }
        };
        auto sum_block = [&](const uint32_t (&pk)[16]) -> float {
          __half2 t8[8];
#pragma unroll
          for (int k = 0; k < 8; ++k) t8[k] = __hadd2(u2h(pk[2 * k]), u2h(pk[2 * k + 1]));
#pragma unroll
          for (int k = 0; k < 4; ++k) t8[k] = __hadd2(t8[2 * k], t8[2 * k + 1]);
          t8[0] = __hadd2(t8[0], t8[1]);
          t8[2] = __hadd2(t8[2], t8[3]);
          const float2 f = __half22float2(__hadd2(t8[0], t8[2]));
          return f.x + f.y;
        };
#pragma unroll
        for (int cp = 0; cp < 2; ++cp) {
          tmem_ld32x2(tS + 64 * cp, tS + 64 * cp + 32, va, vb);
          uint32_t pk[16];
          exp_block(va, pk, 64 * cp, nvalid == 128);
          tmem_st16(tS + 32 * cp, pk);  // P of columns 64cp..64cp+31 over columns already read
          lsum += sum_block(pk);
          exp_block(vb, pk, 64 * cp + 32, nvalid == 128);
          tmem_st16(tS + 32 * cp + 16, pk);
          lsum += sum_block(pk);
        }
        tmem_wait_st();
        l_run += lsum;
        tc_fence_before();
        mbar_arrive(bar(B_PFULL + i));
      }
      if (ok && u + 1 < n_units) {
        const Unit Un = unit_at(a, S, u + 1, h);
        if (Un.psac) {
          // S_i of this chunk's last tile has completed: the Q U_r columns are free.
          write_qu(sm + OFF_QU, i, row, qvalid, qrow, Un.hb + L.ut, r, rpad);
          fence_proxy_async_smem();
          mbar_arrive(bar(B_QU + i));
        }
      }
    }
    if (ok) ok = __all_sync(0xFFFFFFFFu, mbar_wait(bar(B_OFINAL), 0));
    if (ok) {
      tc_fence_after();
      const float inv_l = 1.0f / l_run;
      float v[32];
#pragma unroll
      for (int cb = 0; cb < 4; ++cb) {
        tmem_ld32(tO + cb * 32, v);
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
    } else {
      *s_err = 1;
    }
  } else if (warp < W_MMA) {
    // ------------------------------------------------------------ dequant K (warps 8-11) / V (12-15)
    const bool isK = warp < W_DQV;
    const int64_t o_codes = isK ? L.k_codes : L.v_codes, o_scales = isK ? L.k_scales : L.v_scales;
    const int64_t o_ids = isK ? L.k_ids : L.v_ids, o_zeros = isK ? L.k_zeros : L.v_zeros;
    // Four lanes per row: lane q of a quad rebuilds channels 16q..16q+15 and
    // 64+16q..64+16q+15 of its row (chunks 2q, 2q+1, 8+2q, 9+2q), reading
    // 32-byte slices, so one warp-wide load touches 8 centroid rows (8 cache
    // lines) instead of 32.  Warp w of the group covers rows 32w..32w+31 in
    // four passes of 8 rows, two passes per round of loads.  The rows'
    // centroid ids and zero-points of the next tile are loaded one tile ahead.
    const int q = lane & 3, rr = lane >> 2;
    const int wrow = (warp & 3) * 32 + rr;  // row of pass p: wrow + 8p
    TileCursor cur;
    cur.init(a, S, h, n_units);
    auto load_ids = [&](const TileCursor& c) -> uint64_t {  // 4 ids | 4 zero bytes << 32
      uint64_t v = 0;
      if (c.valid() && c.U.hb) {
        const uint8_t* tb = c.U.hb + L.tiles_off + (int64_t)c.tl * L.tile_bytes;
        const int nv = c.nvalid();
#pragma unroll
        for (int p = 0; p < 4; ++p) {
          const int row = wrow + 8 * p;
          if (row < nv)
            v |= ((uint64_t)tb[o_ids + row] << (8 * p)) | ((uint64_t)tb[o_zeros + (int64_t)row * L.zb] << (32 + 8 * p));
        }
      }
      return v;
    };
    uint64_t idn = load_ids(cur);
    uint32_t jt = 0;
    bool ok = true;
    while (cur.valid()) {
      const uint64_t idc = idn;
      TileCursor nc = cur;
      nc.next(a, S, h);
      idn = load_ids(nc);
      const int st = jt & 1;
      const uint32_t ph = (jt >> 1) & 1;
      const int nv = cur.nvalid();
      if (!mbar_wait(bar((isK ? B_KEMPTY : B_VEMPTY) + st), ph ^ 1)) {
        ok = false;
        break;
      }
      uint8_t* dst = sm + (isK ? OFF_K : OFF_V) + st * 2 * BLK;
      const uint8_t* tb = cur.U.hb ? cur.U.hb + L.tiles_off + (int64_t)cur.tl * L.tile_bytes : nullptr;
      const uint8_t* tab = cur.U.hb ? cur.U.hb + (isK ? L.ktab : L.vtab) : nullptr;
      const bool psac_lane = isK && cur.U.psac && q * 8 < r;
#pragma unroll
      for (int rd = 0; rd < 2; ++rd) {
        uint32_t mv[2][2][8];  // [pass][slice][words]
        uint32_t cwv[2][2];
        uint32_t scv[2][2];
        uint2 cfv[2];          // PSAC INT8 codes 8q..8q+7 of the row (Keys)
        uint32_t sgv[2];       // PSAC row scale (binary16 bits)
#pragma unroll
        for (int pp = 0; pp < 2; ++pp) {
          const int p = 2 * rd + pp;
          const int row = wrow + 8 * p;
#pragma unroll
          for (int sl = 0; sl < 2; ++sl) {
#pragma unroll
            for (int e = 0; e < 8; ++e) mv[pp][sl][e] = 0u;
            cwv[pp][sl] = 0u;
            scv[pp][sl] = 0u;
          }
          cfv[pp] = make_uint2(0u, 0u);
          sgv[pp] = 0u;
          if (row < nv) {
            if (tb) {
              if (psac_lane) {  // the row's PSAC codes ride in the same round of loads
                cfv[pp] = __ldg(reinterpret_cast<const uint2*>(tb + L.k_coef + (int64_t)row * r + q * 8));
                sgv[pp] = __ldg(reinterpret_cast<const unsigned short*>(tb + L.k_sigma + row * 2));
              }
              const uint8_t* mu = tab + (int64_t)((idc >> (8 * p)) & 0xFFu) * 256;
              ldg32B(mu + 32 * q, mv[pp][0]);
              ldg32B(mu + 128 + 32 * q, mv[pp][1]);
              const uint8_t* cp = tb + o_codes + row * 32;
              cwv[pp][0] = __ldg(reinterpret_cast<const uint32_t*>(cp + 4 * q));
              cwv[pp][1] = __ldg(reinterpret_cast<const uint32_t*>(cp + 16 + 4 * q));
              const unsigned short* sp = reinterpret_cast<const unsigned short*>(tb + o_scales + (int64_t)row * L.ng * 2);
              scv[pp][0] = __ldg(sp + ((16 * q) >> gshift));
              scv[pp][1] = __ldg(sp + ((64 + 16 * q) >> gshift));
            } else {
              const __nv_bfloat16* src = (isK ? a.kcur : a.vcur) + ((size_t)(cur.tl * 128 + row) * H + h) * 128;
              const uint4 v0 = ldg16(src + 16 * q), v1 = ldg16(src + 16 * q + 8);
              const uint4 v2 = ldg16(src + 64 + 16 * q), v3 = ldg16(src + 64 + 16 * q + 8);
              const uint4 f0 = bf16x8_to_f16x8(v0), f1 = bf16x8_to_f16x8(v1);
              const uint4 f2 = bf16x8_to_f16x8(v2), f3 = bf16x8_to_f16x8(v3);
              mv[pp][0][0] = f0.x; mv[pp][0][1] = f0.y; mv[pp][0][2] = f0.z; mv[pp][0][3] = f0.w;
              mv[pp][0][4] = f1.x; mv[pp][0][5] = f1.y; mv[pp][0][6] = f1.z; mv[pp][0][7] = f1.w;
              mv[pp][1][0] = f2.x; mv[pp][1][1] = f2.y; mv[pp][1][2] = f2.z; mv[pp][1][3] = f2.w;
              mv[pp][1][4] = f3.x; mv[pp][1][5] = f3.y; mv[pp][1][6] = f3.z; mv[pp][1][7] = f3.w;
            }
          }
        }
#pragma unroll
        for (int pp = 0; pp < 2; ++pp) {
          const int p = 2 * rd + pp;
          const int row = wrow + 8 * p;
          const uint32_t zbyte = (uint32_t)((idc >> (32 + 8 * p)) & 0xFFu);
#pragma unroll
          for (int sl = 0; sl < 2; ++sl) {
            const int c0 = 8 * sl + 2 * q;  // first of the two chunks of this slice
            uint32_t ow[8];
            if (tb && row < nv) {
              const int g = (64 * sl + 16 * q) >> gshift;
              const uint32_t sb = scv[pp][sl];
              const __half2 s2 = u2h(sb | (sb << 16));
              const uint32_t zz = 0x6400u | ((zbyte >> (2 * g)) & 3u);
              const __half2 z2 = u2h(zz | (zz << 16));
              const uint32_t word = cwv[pp][sl];
#pragma unroll
              for (int k = 0; k < 8; ++k) {  // channel pairs (2k, 2k+1) of the 16-channel word
                const uint32_t qq = ((word >> (2 * k)) & 0x00030003u) | 0x64006400u;
                ow[k] = h2u(__hfma2(__hsub2(u2h(qq), z2), s2, u2h(mv[pp][sl][k])));
              }
            } else {
#pragma unroll
              for (int k = 0; k < 8; ++k) ow[k] = mv[pp][sl][k];
            }
            st_chunk(dst, row, c0, make_uint4(ow[0], ow[1], ow[2], ow[3]));
            st_chunk(dst, row, c0 + 1, make_uint4(ow[4], ow[5], ow[6], ow[7]));
          }
          if (isK && cur.U.psac && q * 8 < rpad) {
            // C_hat = t * sigma (Eq. 16), PSAC columns 8q..8q+7 of the row, in
            // f16: byte b of an INT8 code t becomes the f16 1024 + (t + 128)
            // (its byte XOR 0x80 under exponent bits 0x64), minus 1152 gives t
            // exactly, and one f16 multiply rounds t * sigma once.
            uint32_t w4[4] = {0u, 0u, 0u, 0u};
            if (tb && row < nv && q * 8 < r) {
              const __half2 sg2 = u2h(sgv[pp] | (sgv[pp] << 16));
              const __half2 off2 = u2h(0x64806480u);  // (1152, 1152)
              const uint32_t cwd[2] = {cfv[pp].x ^ 0x80808080u, cfv[pp].y ^ 0x80808080u};
#pragma unroll
              for (int q2 = 0; q2 < 4; ++q2) {
                const uint32_t b0 = 2 * (q2 & 1);
                const uint32_t t2 = __byte_perm(cwd[q2 >> 1], 0x64646464u, b0 | (4u << 4) | ((b0 + 1) << 8) | (4u << 12));
                w4[q2] = h2u(__hmul2(__hsub2(u2h(t2), off2), sg2));
              }
            }
            st_chunk(sm + OFF_C, row, (st * rpad) / 8 + q, make_uint4(w4[0], w4[1], w4[2], w4[3]));
          }
        }
      }
      fence_proxy_async_smem();
      mbar_arrive(bar((isK ? B_KFULL : B_VFULL) + st));
      cur = nc;
      ++jt;
    }
    if (!ok) *s_err = 1;
  } else {
    // ------------------------------------------------------------ MMA issue (one thread)
    // Order per KV tile j: P0 V(j), S0(j+1), P1 V(j), S1(j+1), so that the
    // softmax of Q tile 0 on tile j+1 overlaps the softmax of Q tile 1 on
    // tile j (S_i(j+1) reuses the TMEM columns of P_i(j) after P_i V(j) has
    // read them: MMAs of one thread run in issue order).
    if (lane == 0) {
      const uint32_t aQ = smem_u32(sm + OFF_Q), aQU = smem_u32(sm + OFF_QU);
      const uint32_t aK = smem_u32(sm + OFF_K), aC = smem_u32(sm + OFF_C), aV = smem_u32(sm + OFF_V);
      constexpr uint32_t idS = idesc_f16(128, 128, false);
      constexpr uint32_t idPV = idesc_f16(128, 64, true);
      int total = 0;
      for (int u = 0; u < n_units; ++u) total += (unit_at(a, S, u, h).ntok + 127) / 128;
      TileCursor sc;  // next tile to issue S for
      sc.init(a, S, h, n_units);
      uint32_t sjt = 0, qph[2] = {0, 0};
      bool ok = true;
      auto issue_S = [&](int i) -> bool {
        const int st = sjt & 1;
        const uint32_t ph = (sjt >> 1) & 1;
        if (sc.tl == 0 && (sc.u == 0 || sc.U.psac)) {
          if (!mbar_wait(bar(B_QU + i), qph[i])) return false;
          qph[i] ^= 1;
        }
        if (i == 0 && !mbar_wait(bar(B_KFULL + st), ph)) return false;
        tc_fence_after();
        const uint32_t tS = tbase + 128 * i;
#pragma unroll
        for (int kb = 0; kb < 2; ++kb)
#pragma unroll
          for (int ks = 0; ks < 4; ++ks)
            umma_ss(tS, desc_sw128(aQ + (2 * i + kb) * BLK + ks * 32), desc_sw128(aK + (2 * st + kb) * BLK + ks * 32),
                    idS, (kb | ks) != 0);
        if (sc.U.psac)
          for (int ks = 0; ks < rpad / 16; ++ks)
            umma_ss(tS, desc_sw128(aQU + i * rpad * 2 + ks * 32), desc_sw128(aC + st * rpad * 2 + ks * 32), idS, 1u);
        umma_commit(bar(B_SFULL + i));
        if (i == 1) {
          umma_commit(bar(B_KEMPTY + st));
          sc.next(a, S, h);
          ++sjt;
        }
        return true;
      };
      if (total > 0) ok = issue_S(0) && issue_S(1);
      for (int jt = 0; jt < total && ok; ++jt) {
        const int st = jt & 1;
        const uint32_t ph = (jt >> 1) & 1;
        if (!(ok = mbar_wait(bar(B_VFULL + st), ph))) break;
#pragma unroll
        for (int i = 0; i < 2; ++i) {
          if (!(ok = mbar_wait(bar(B_PFULL + i), jt & 1))) break;
          tc_fence_after();
          const uint32_t tP = tbase + 128 * i, tO = tbase + 256 + 128 * i;
#pragma unroll
          for (int ks = 0; ks < 8; ++ks)
#pragma unroll
            for (int nh = 0; nh < 2; ++nh)
              umma_ts(tO + 64 * nh, tP + 8 * ks, desc_sw128(aV + (2 * st + nh) * BLK + ks * 2048), idPV,
                      (jt > 0 || ks > 0) ? 1u : 0u);
          if (i == 1) umma_commit(bar(B_VEMPTY + st));
          if (jt + 1 < total && !(ok = issue_S(i))) break;
        }
      }
      umma_commit(bar(B_OFINAL));
      if (!ok) *s_err = 1;
    }
    __syncwarp();
  }

  tc_fence_before();
  __syncthreads();
  if (tid == 0 && *s_err) atomicCAS(a.status, 0, (int)QWM_ERR_TIMEOUT);
  if (warp == W_MMA) {
    tc_fence_after();
    tmem_dealloc(tbase, 512);
  }
}

}  // namespace

cudaError_t launch_attend(const AttendArgs& a, const AttendSlots& slots, cudaStream_t st) {
  cudaError_t e = cudaFuncSetAttribute(attend_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES);
  if (e != cudaSuccess) return e;
  dim3 grid((unsigned)((a.Nq + 255) / 256), (unsigned)a.L.H);
  attend_kernel<<<grid, NT, SMEM_BYTES, st>>>(a, slots);
  return cudaGetLastError();
}

}  // namespace qwm
