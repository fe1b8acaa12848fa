// append_generic.cu -- quantize-on-append for any candidate count M: QSAC
// centroid assignment (Sec. 4.1 Eq. 9, 10, 12), INT2 residual quantization
// with packing (Sec. 2 Eq. 1-4, App. D.1) and the PSAC coefficients of the Key
// error (Sec. 4.2 Eq. 13, 16).  Every Query-aware distance is evaluated
// exactly on CUDA cores; append.cu's tensor-core kernel handles M <= 8 and
// M >= C and hands the other candidate counts to this one.
//
// One CTA handles TT tokens of one head for Keys (blockIdx.z = 0) or Values
// (blockIdx.z = 1).  Every quantity that decides an integer (distances, QSAC
// scores, scales, codes, PSAC codes, keep test) is evaluated in fp32 with
// explicitly rounded operations (__fadd_rn / __fmul_rn / __fdiv_rn, never
// contracted, and one __fmaf_rn per term of the sums of products), summed in
// channel order, so the packed output is bit-exact against a sequential fp32
// evaluation of the same formulas.
#include "ptx_sm103.cuh"
#include "qwm_internal.cuh"

namespace qwm {
namespace {

using ptx::bf16x2_out_of_f16;

constexpr int TT = 32;         // tokens per CTA
constexpr int NT = 256;        // threads per CTA
constexpr int NW = NT / 32;
constexpr int MU_W = 65;       // padded SMEM row stride of a centroid (32-bit words)

__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }
__device__ __forceinline__ float bf2f(__nv_bfloat16 b) { return __bfloat162float(b); }

struct Smem {
  uint32_t* mu;      // [C][MU_W] centroid rows (bf16 pairs)
  float* x;          // [TT][128] tokens
  float* w;          // [128]
  float* wg;         // [4] group weight sums
  float* dq;         // [TT][C] Query-aware distances
  __nv_bfloat16* U;  // [128][r]
  float* e;          // [NW][128] PSAC error
  float* tq;         // [NW][128] weighted error terms after correction
  float* t0;         // [NW][128] weighted error terms before correction
  int* cand;         // [NW][256] candidates
};

__host__ __device__ inline size_t smem_bytes(int C, int r) {
  size_t b = 0;
  b += (size_t)C * MU_W * 4;
  b += (size_t)TT * 128 * 4;
  b += 128 * 4 + 16;
  b += (size_t)TT * C * 4;
  b += (size_t)128 * r * 2 + 16;
  b += (size_t)NW * 128 * 4 * 3;
  b += (size_t)NW * 256 * 4;
  return b;
}

__global__ void __launch_bounds__(NT, 1) append_generic_kernel(const AppendArgs a) {
  extern __shared__ __align__(16) uint8_t smem_raw[];
  const Layout& L = a.L;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int h = blockIdx.y;
  const bool is_key = blockIdx.z == 0;
  const int64_t t0 = (int64_t)blockIdx.x * TT;
  const int C = L.C, G = L.G, ng = L.ng, r = L.r, H = L.H;
  const int glanes = G / 4;  // lanes per group (4 channels per lane)
  const __nv_bfloat16* x = is_key ? a.k : a.v;
  const __nv_bfloat16* tab = (is_key ? a.kc : a.vc) + (size_t)h * C * 128;
  const bool use_w = is_key && a.w != nullptr;
  const bool psac = is_key && a.U != nullptr && r > 0;
  uint8_t* head = a.base + head_offset(L, a.slot, h);

  Smem s;
  uint8_t* p = smem_raw;
  s.mu = reinterpret_cast<uint32_t*>(p); p += (size_t)C * MU_W * 4;
  s.x = reinterpret_cast<float*>(p); p += (size_t)TT * 128 * 4;
  s.w = reinterpret_cast<float*>(p); p += 128 * 4;
  s.wg = reinterpret_cast<float*>(p); p += 16;
  s.dq = reinterpret_cast<float*>(p); p += (size_t)TT * C * 4;
  s.U = reinterpret_cast<__nv_bfloat16*>(p); p += round_up((int64_t)128 * r * 2 + 16, 16);
  s.e = reinterpret_cast<float*>(p); p += NW * 128 * 4;
  s.tq = reinterpret_cast<float*>(p); p += NW * 128 * 4;
  s.t0 = reinterpret_cast<float*>(p); p += NW * 128 * 4;
  s.cand = reinterpret_cast<int*>(p);

  // The chunk's own tables travel with the slot (one CTA per head and K/V),
  // stored as binary16 (exact for bf16 values in the binary16 range), the
  // operand type of the attention kernel's tensor-core path.
  // A Key or Value or a table value beyond the binary16 range (or not a
  // number) cannot be held by the cache's binary16 operands: reported in the
  // cache's status word as QWM_ERR_NONFINITE.
  bool nbad = false;
  if (blockIdx.x == 0) {
    const uint32_t* src = reinterpret_cast<const uint32_t*>(tab);
    __half2* dst = reinterpret_cast<__half2*>(head + (is_key ? L.ktab : L.vtab));
    for (int i = tid; i < C * 64; i += NT) {
      const uint32_t pr = src[i];
      nbad |= bf16x2_out_of_f16(pr);
      dst[i] = __floats2half2_rn(bf_lo(pr), bf_hi(pr));
    }
    if (psac) {
      __nv_bfloat16* ut = reinterpret_cast<__nv_bfloat16*>(head + L.ut);
      const __nv_bfloat16* Uh = a.U + (size_t)h * 128 * r;
      for (int i = tid; i < r * 128; i += NT) {
        const int j = i / 128, c = i % 128;
        ut[i] = Uh[(size_t)c * r + j];  // U_r^T [r][d]
      }
    }
  }

  for (int i = tid; i < C * 64; i += NT) {
    const int j = i >> 6, wd = i & 63;
    s.mu[j * MU_W + wd] = reinterpret_cast<const uint32_t*>(tab + (size_t)j * 128)[wd];
  }
  if (tid < 128) s.w[tid] = use_w ? a.w[(size_t)h * 128 + tid] : 1.0f;
  for (int i = tid; i < TT * 64; i += NT) {
    const int ti = i >> 6, wd = i & 63;
    const int64_t t = t0 + ti;
    uint32_t pr = 0;
    if (t < a.N) {
      pr = reinterpret_cast<const uint32_t*>(x + ((size_t)t * H + h) * 128)[wd];
      nbad |= bf16x2_out_of_f16(pr);
    }
    s.x[ti * 128 + 2 * wd] = bf_lo(pr);
    s.x[ti * 128 + 2 * wd + 1] = bf_hi(pr);
  }
  if (psac)
    for (int i = tid; i < 128 * r; i += NT) s.U[i] = a.U[(size_t)h * 128 * r + i];  // [d][r]
  if (nbad) atomicCAS(reinterpret_cast<int*>(a.base), 0, (int)QWM_ERR_NONFINITE);
  // PSAC rows are written at their token's index; each kept row sets its bit
  // in the tile's keep mask (zeroed before the launch), and psac_tile_finish
  // then stores each tile in the dense or the sparse layout.
  __syncthreads();
  if (tid < ng) {
    float Wg = 0.0f;
    for (int c = tid * G; c < (tid + 1) * G; ++c) Wg = __fadd_rn(Wg, s.w[c]);
    s.wg[tid] = Wg;
  }

  // ---- 1. Query-aware distance dQ_j = sum_c w_c (k_c - mu_jc)^2 (Eq. 9)
  for (int j = tid; j < C; j += NT) {
    float acc[TT];
#pragma unroll
    for (int i = 0; i < TT; ++i) acc[i] = 0.0f;
    const uint32_t* row = s.mu + j * MU_W;
    for (int cw = 0; cw < 64; ++cw) {
      const uint32_t pr = row[cw];
      const float m0 = bf_lo(pr), m1 = bf_hi(pr);
      const float w0 = s.w[2 * cw], w1 = s.w[2 * cw + 1];
#pragma unroll
      for (int i = 0; i < TT; ++i) {
        float t = __fsub_rn(s.x[i * 128 + 2 * cw], m0);
        acc[i] = __fmaf_rn(w0, __fmul_rn(t, t), acc[i]);
        t = __fsub_rn(s.x[i * 128 + 2 * cw + 1], m1);
        acc[i] = __fmaf_rn(w1, __fmul_rn(t, t), acc[i]);
      }
    }
#pragma unroll
    for (int i = 0; i < TT; ++i) s.dq[i * C + j] = acc[i];
  }
  __syncthreads();

  // ---- 2.-5. one warp per token
  const int Mc = a.M;
  int* cand = s.cand + warp * 256;
  for (int i = warp; i < TT; i += NW) {
    const int64_t t = t0 + i;
    if (t >= a.N) break;
    const float* dq = s.dq + i * C;
    // 2. top-M candidates, lexicographic (dQ, j)
    if (Mc >= C) {
      for (int j = lane; j < C; j += 32) cand[j] = j;
    } else {
      uint32_t chosen = 0;
      for (int m = 0; m < Mc; ++m) {
        float bd = INFINITY;
        int bj = 0x7FFFFFFF;
        for (int k8 = 0; k8 < 8; ++k8) {
          const int j = lane + 32 * k8;
          if (j < C && !((chosen >> k8) & 1u)) {
            const float v = dq[j];
            if (v < bd || (v == bd && j < bj)) { bd = v; bj = j; }
          }
        }
#pragma unroll
        for (int off = 16; off; off >>= 1) {
          const float od = __shfl_xor_sync(0xFFFFFFFFu, bd, off);
          const int oj = __shfl_xor_sync(0xFFFFFFFFu, bj, off);
          if (od < bd || (od == bd && oj < bj)) { bd = od; bj = oj; }
        }
        if (bj >= C) bj = C - 1;  // only reachable with non-finite inputs
        if ((bj & 31) == lane) chosen |= 1u << (bj >> 5);
        if (lane == 0) cand[m] = bj;
      }
    }
    __syncwarp();

    float xk[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) xk[e] = s.x[i * 128 + 4 * lane + e];

    // 3. QSAC score S_j = sum_g W_g R_g^2 over the candidates (Eq. 10, 12)
    float bestS = INFINITY;
    int bestj = 0x7FFFFFFF;
    for (int m = 0; m < Mc; ++m) {
      const int j = cand[m];
      const uint32_t* row = s.mu + j * MU_W;
      const uint32_t pa = row[2 * lane], pb = row[2 * lane + 1];
      const float r0 = __fsub_rn(xk[0], bf_lo(pa)), r1 = __fsub_rn(xk[1], bf_hi(pa));
      const float r2 = __fsub_rn(xk[2], bf_lo(pb)), r3 = __fsub_rn(xk[3], bf_hi(pb));
      float mx = fmaxf(fmaxf(r0, r1), fmaxf(r2, r3));
      float mn = fminf(fminf(r0, r1), fminf(r2, r3));
      for (int off = 1; off < glanes; off <<= 1) {
        mx = fmaxf(mx, __shfl_xor_sync(0xFFFFFFFFu, mx, off));
        mn = fminf(mn, __shfl_xor_sync(0xFFFFFFFFu, mn, off));
      }
      const float R = __fsub_rn(mx, mn);
      float S = 0.0f;
      for (int g = 0; g < ng; ++g) {
        const float Rg = __shfl_sync(0xFFFFFFFFu, R, g * glanes);
        S = __fadd_rn(S, __fmul_rn(s.wg[g], __fmul_rn(Rg, Rg)));
      }
      if (S < bestS || (S == bestS && j < bestj)) { bestS = S; bestj = j; }
    }
    const int id = bestj < C ? bestj : C - 1;

    // 4. INT2 residual quantization (Eq. 1-2), k0 = mu + s (q - z) (Eq. 4)
    const uint32_t* row = s.mu + id * MU_W;
    const uint32_t pa = row[2 * lane], pb = row[2 * lane + 1];
    const float mu4[4] = {bf_lo(pa), bf_hi(pa), bf_lo(pb), bf_hi(pb)};
    float res[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) res[e] = __fsub_rn(xk[e], mu4[e]);
    float lo = fminf(fminf(fminf(res[0], res[1]), fminf(res[2], res[3])), 0.0f);
    float hi = fmaxf(fmaxf(fmaxf(res[0], res[1]), fmaxf(res[2], res[3])), 0.0f);
    for (int off = 1; off < glanes; off <<= 1) {
      lo = fminf(lo, __shfl_xor_sync(0xFFFFFFFFu, lo, off));
      hi = fmaxf(hi, __shfl_xor_sync(0xFFFFFFFFu, hi, off));
    }
    const float s32 = __fdiv_rn(__fsub_rn(hi, lo), 3.0f);
    __half sh = __float2half_ru(s32);
    float sc = __half2float(sh);
    // scale format 1 (App. D.1): s = code * s2, s2 the binary16 round-up of the
    // token's largest range / 3 / 255, code the smallest byte covering range / 3
    uint32_t code = 0;
    __half s2h = __ushort_as_half(0);
    if (L.sf) {
      float smax = s32;
      for (int off = glanes; off < 32; off <<= 1) smax = fmaxf(smax, __shfl_xor_sync(0xFFFFFFFFu, smax, off));
      s2h = __float2half_ru(__fdiv_rn(smax, 255.0f));
      float s2f = __half2float(s2h);
      if (smax > 0.0f && __fmul_rn(255.0f, s2f) < smax) {
        s2h = __ushort_as_half((unsigned short)(__half_as_ushort(s2h) + 1));
        s2f = __half2float(s2h);
      }
      int c = 0;
      if (s2f > 0.0f) {
        c = (int)ceilf(__fdiv_rn(s32, s2f));
        if (c > 0 && __fmul_rn((float)(c - 1), s2f) >= s32) c -= 1;
        if (__fmul_rn((float)c, s2f) < s32) c += 1;
        c = c > 255 ? 255 : c;
      }
      code = (uint32_t)c;
      sc = __fmul_rn((float)c, s2f);
    }
    int z = 0;
    uint32_t cbyte = 0;
    float k0[4];
    if (sc == 0.0f) {
#pragma unroll
      for (int e = 0; e < 4; ++e) k0[e] = __fadd_rn(mu4[e], 0.0f);
    } else {
      const float inv = __frcp_rn(sc);
      z = (int)rintf(__fmul_rn(-lo, inv));
      z = z < 0 ? 0 : (z > 3 ? 3 : z);
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        int q = (int)rintf(__fmul_rn(res[e], inv)) + z;
        q = q < 0 ? 0 : (q > 3 ? 3 : q);
        cbyte |= (uint32_t)q << (2 * e);
        k0[e] = __fadd_rn(mu4[e], __fmul_rn((float)(q - z), sc));
      }
    }
    // the rebuilt values must stay inside the binary16 operands of attention
    if (!(fmaxf(fmaxf(fabsf(k0[0]), fabsf(k0[1])), fmaxf(fabsf(k0[2]), fabsf(k0[3]))) < 65504.0f))
      atomicCAS(reinterpret_cast<int*>(a.base), 0, (int)QWM_ERR_NONFINITE);
    uint32_t zbyte = 0;
    for (int g = 0; g < ng; ++g) zbyte |= (uint32_t)__shfl_sync(0xFFFFFFFFu, z, g * glanes) << (2 * g);

    const int64_t tile = t / kTile;
    const int rowi = (int)(t % kTile);
    uint8_t* tb = head + L.tiles_off + tile * L.tile_bytes;
    const int64_t o_codes = is_key ? L.k_codes : L.v_codes;
    const int64_t o_scales = is_key ? L.k_scales : L.v_scales;
    const int64_t o_ids = is_key ? L.k_ids : L.v_ids;
    const int64_t o_zeros = is_key ? L.k_zeros : L.v_zeros;
    // Packed codes: 16 channels per little-endian 32-bit word, even channel 2k
    // at bits 2k, odd channel 2k+1 at bits 16 + 2k (four codes per byte).
    // This lane holds channels 4*lane .. 4*lane+3 = word lane/4, pairs m, m+1
    // with m = 2*(lane % 4).
    const int csh = 4 * (lane & 3);
    uint32_t word = ((cbyte & 3u) << csh) | (((cbyte >> 2) & 3u) << (16 + csh)) |
                    (((cbyte >> 4) & 3u) << (csh + 2)) | (((cbyte >> 6) & 3u) << (16 + csh + 2));
    word |= __shfl_xor_sync(0xFFFFFFFFu, word, 1);
    word |= __shfl_xor_sync(0xFFFFFFFFu, word, 2);
    if ((lane & 3) == 0) *reinterpret_cast<uint32_t*>(tb + o_codes + rowi * 32 + lane) = word;
    if (lane % glanes == 0) {
      if (L.sf) {
        tb[o_scales + (int64_t)rowi * ng + lane / glanes] = (uint8_t)code;
        if (lane == 0) reinterpret_cast<__half*>(tb + (is_key ? L.k_s2 : L.v_s2))[rowi] = s2h;
      } else {
        reinterpret_cast<__half*>(tb + o_scales + (int64_t)rowi * ng * 2)[lane / glanes] = sh;
      }
    }
    if (lane == 0) {
      tb[o_ids + rowi] = (uint8_t)id;
      tb[o_zeros + (int64_t)rowi * L.zb] = (uint8_t)zbyte;
      for (int b = 1; b < L.zb; ++b) tb[o_zeros + (int64_t)rowi * L.zb + b] = 0;
    }

    // 5. PSAC coefficients of the remaining Key error (Eq. 13, 16) + keep rule
    if (is_key && r > 0) {
      int8_t* coef = reinterpret_cast<int8_t*>(tb + L.k_coef + (int64_t)rowi * r);
      __half* sig = reinterpret_cast<__half*>(tb + L.k_sigma) + rowi;
      if (!psac) {
        if (lane < r) coef[lane] = 0;
        if (lane == 0) *sig = __ushort_as_half(0);
      } else {
        float* se = s.e + warp * 128;
        float E[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          E[e] = __fsub_rn(xk[e], k0[e]);
          se[4 * lane + e] = E[e];
        }
        __syncwarp();
        float cj = 0.0f;
        if (lane < r)
          for (int c = 0; c < 128; ++c) cj = __fmaf_rn(se[c], bf2f(s.U[c * r + lane]), cj);
        float amax = lane < r ? fabsf(cj) : 0.0f;
#pragma unroll
        for (int off = 16; off; off >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xFFFFFFFFu, amax, off));
        const __half sgh = __float2half_ru(__fdiv_rn(amax, 127.0f));
        const float sg = __half2float(sgh);
        if (lane == 0 && !(127.0f * sg <= 65504.0f))  // C_hat = t sigma must stay a finite binary16
          atomicCAS(reinterpret_cast<int*>(a.base), 0, (int)QWM_ERR_NONFINITE);
        int tq = 0;
        float ch = 0.0f;
        if (sg != 0.0f && lane < r) {
          const float inv = __frcp_rn(sg);
          float qq = rintf(__fmul_rn(cj, inv));
          qq = fminf(fmaxf(qq, -127.0f), 127.0f);
          tq = (int)qq;
          ch = __fmul_rn(qq, sg);
        }
        float* stq = s.tq + warp * 128;
        float* st0 = s.t0 + warp * 128;
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int c = 4 * lane + e;
          float u = 0.0f;
          for (int j = 0; j < r; ++j) {
            const float chj = __shfl_sync(0xFFFFFFFFu, ch, j);
            u = __fmaf_rn(bf2f(s.U[c * r + j]), chj, u);
          }
          const float ep = __fsub_rn(E[e], u);
          stq[c] = __fmul_rn(ep, ep);
          st0[c] = __fmul_rn(E[e], E[e]);
        }
        __syncwarp();
        int keep = 0;
        if (lane == 0) {
          float errq = 0.0f, err0 = 0.0f;
          for (int c = 0; c < 128; ++c) {
            errq = __fmaf_rn(s.w[c], stq[c], errq);
            err0 = __fmaf_rn(s.w[c], st0[c], err0);
          }
          keep = errq < err0;
        }
        keep = __shfl_sync(0xFFFFFFFFu, keep, 0);
        if (lane < r) coef[lane] = (int8_t)(keep ? tq : 0);
        if (lane == 0) *sig = keep ? sgh : __ushort_as_half(0);
        if (lane == 0 && keep)
          atomicOr(reinterpret_cast<unsigned int*>(head + L.pmask + tile * 16) + (rowi >> 5), 1u << (rowi & 31));
      }
    }
    __syncwarp();
  }
}

// The dense/sparse PSAC layout of each 128-token Key tile (App. D.1), from the
// keep mask the quantize kernel left: with n_t tokens and K_t kept rows the
// tile is sparse iff 16 + K_t (r + 2) < n_t (r + 2) (a 16-byte mask plus the
// kept rows against every row).  Dense: the mask becomes the tile's full
// token mask (dropped rows already hold zeros).  Sparse: the mask stays the
// keep set and kept row i moves to entry popcount(mask below i), through
// shared memory (the moves overlap in place).  One CTA per (tile, head),
// thread = row.
__global__ void __launch_bounds__(kTile) psac_tile_finish(const AppendArgs a) {
  __shared__ uint2 srow[kTile][4];  // up to 32 code bytes per row
  __shared__ __half ssig[kTile];
  const Layout& L = a.L;
  const int tile = blockIdx.x, h = blockIdx.y, i = threadIdx.x, r = L.r;
  uint8_t* head = a.base + head_offset(L, a.slot, h);
  uint4* mp = reinterpret_cast<uint4*>(head + L.pmask + (int64_t)tile * 16);
  const uint4 m = *mp;
  const int64_t nt64 = a.N - (int64_t)tile * kTile;
  const int nt = nt64 < kTile ? (int)nt64 : kTile;
  const int K = __popc(m.x) + __popc(m.y) + __popc(m.z) + __popc(m.w);
  if (!(16 + K * (r + 2) < nt * (r + 2))) {
    if (i == 0) {
      uint32_t m4[4];
      for (int w4 = 0; w4 < 4; ++w4) {
        const int nb = nt - 32 * w4;
        m4[w4] = nb >= 32 ? 0xFFFFFFFFu : (nb > 0 ? (1u << nb) - 1u : 0u);
      }
      *mp = make_uint4(m4[0], m4[1], m4[2], m4[3]);
    }
    return;
  }
  uint8_t* tb = head + L.tiles_off + (int64_t)tile * L.tile_bytes;
  uint2* coef = reinterpret_cast<uint2*>(tb + L.k_coef);  // rows of r / 8 words
  __half* sig = reinterpret_cast<__half*>(tb + L.k_sigma);
  const int rw = r / 8;
  const int e = i < nt ? psac_entry(m, i) : -1;
  if (e >= 0) {
    for (int q = 0; q < rw; ++q) srow[i][q] = coef[i * rw + q];
    ssig[i] = sig[i];
  }
  __syncthreads();
  if (e >= 0) {
    for (int q = 0; q < rw; ++q) coef[e * rw + q] = srow[i][q];
    sig[e] = ssig[i];
  }
}

}  // namespace

cudaError_t launch_append_generic(const AppendArgs& a, cudaStream_t st) {
  const size_t smem = smem_bytes(a.L.C, a.L.r);
  cudaError_t e = cudaFuncSetAttribute(append_generic_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  const int tiles = (int)((a.N + kTile - 1) / kTile);
  if (a.L.r > 0) {  // the keep masks of this slot's heads start empty
    e = cudaMemset2DAsync(a.base + head_offset(a.L, a.slot, 0) + a.L.pmask, (size_t)a.L.head_bytes, 0,
                          (size_t)tiles * 16, (size_t)a.L.H, st);
    if (e != cudaSuccess) return e;
  }
  dim3 grid((unsigned)((a.N + TT - 1) / TT), (unsigned)a.L.H, 2);
  append_generic_kernel<<<grid, NT, smem, st>>>(a);
  e = cudaGetLastError();
  if (e != cudaSuccess || a.L.r == 0) return e;
  psac_tile_finish<<<dim3((unsigned)tiles, (unsigned)a.L.H), kTile, 0, st>>>(a);
  return cudaGetLastError();
}

}  // namespace qwm
