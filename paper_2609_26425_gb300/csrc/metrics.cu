// metrics.cu -- reconstruction of a cached chunk and the top-1 key of each
// query, the two steps of the token-selection shift measurement (the ratio of
// queries whose highest-logit key changes when the cached Keys are
// quantized; the paper's "top-1 temporal-spatial token selection shift").
//
//   dequant_kernel  warp per (token, head), lane = four channels: the values
//                   attention rebuilds, k_hat = mu_id + s (q - z) (+ U_r t sigma
//                   for Keys stored with a PSAC correction), in fp32; s is the
//                   binary16 group scale or, in scale format 1, code * s2.
//   top1_kernel     64 queries x 64 keys per step on CUDA cores (a measurement,
//                   not the hot path): every logit is the fp32 sum in channel
//                   order with one fused multiply-add per term; the largest
//                   wins, ties to the lower key index.
#include "qwm_internal.cuh"

namespace qwm {
namespace {

// Bit of channel c in a token's 32 code bytes: every 16 channels form one
// little-endian 32-bit word, even channel 2k at bits 2k, odd 2k+1 at 16 + 2k.
__global__ void __launch_bounds__(256) dequant_kernel(const DequantArgs a) {
  const Layout& L = a.L;
  const int lane = threadIdx.x & 31;
  const int64_t n = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
  const int h = blockIdx.y;
  if (n >= a.N) return;
  const uint8_t* head = a.base + head_offset(L, a.slot, h);
  const int64_t tile = n >> 7, row = n & 127;
  const uint8_t* tb = head + L.tiles_off + tile * L.tile_bytes;
  const int c0 = 4 * lane, G = L.G, ng = L.ng;
  const int g = c0 / G;
  for (int side = 0; side < 2; ++side) {
    float* out = side == 0 ? a.k_out : a.v_out;
    if (!out) continue;
    const int64_t o_codes = side ? L.v_codes : L.k_codes, o_scales = side ? L.v_scales : L.k_scales;
    const int64_t o_ids = side ? L.v_ids : L.k_ids, o_zeros = side ? L.v_zeros : L.k_zeros;
    const int id = tb[o_ids + row];
    const __half* tab = reinterpret_cast<const __half*>(head + (side ? L.vtab : L.ktab)) + (size_t)id * 128;
    const float s = L.sf ? (float)tb[o_scales + row * ng + g] *
                               __half2float(reinterpret_cast<const __half*>(tb + (side ? L.v_s2 : L.k_s2))[row])
                         : __half2float(reinterpret_cast<const __half*>(tb + o_scales + row * ng * 2)[g]);
    const int z = (tb[o_zeros + row * L.zb + (g >> 2)] >> (2 * (g & 3))) & 3;
    const uint32_t word = reinterpret_cast<const uint32_t*>(tb + o_codes + row * 32)[c0 >> 4];
    const int m = (c0 & 15) >> 2;  // channels 4m .. 4m + 3 of the word's 16
    const int qv[4] = {(int)(word >> (4 * m)) & 3, (int)(word >> (16 + 4 * m)) & 3,
                       (int)(word >> (4 * m + 2)) & 3, (int)(word >> (16 + 4 * m + 2)) & 3};
    float v[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) v[e] = __half2float(tab[c0 + e]) + s * (float)(qv[e] - z);
    const int pe = (side == 0 && a.psac && L.r > 0)
                       ? psac_entry(*reinterpret_cast<const uint4*>(head + L.pmask + tile * 16), (int)row)
                       : -1;
    if (pe >= 0) {
      const float sg = __half2float(*reinterpret_cast<const __half*>(tb + L.k_sigma + pe * 2));
      const int8_t* t = reinterpret_cast<const int8_t*>(tb + L.k_coef + pe * L.r);
      const __nv_bfloat16* Ut = reinterpret_cast<const __nv_bfloat16*>(head + L.ut);  // [r][128]
      for (int j = 0; j < L.r; ++j) {
        const float cj = (float)t[j] * sg;
#pragma unroll
        for (int e = 0; e < 4; ++e) v[e] = fmaf(cj, __bfloat162float(Ut[j * 128 + c0 + e]), v[e]);
      }
    }
    *reinterpret_cast<float4*>(out + ((size_t)n * L.H + h) * 128 + c0) = make_float4(v[0], v[1], v[2], v[3]);
  }
}

constexpr int TQ = 64, TK = 64, TP = 68;  // query / key tile, padded row of the transposed tiles

__global__ void __launch_bounds__(256) top1_kernel(const __nv_bfloat16* __restrict__ q, int64_t Nq,
                                                   const float* __restrict__ keys, int64_t Nk, int H,
                                                   int32_t* __restrict__ idx) {
  extern __shared__ float tsm[];
  float* qT = tsm;              // [128][TP]: channel-major query tile
  float* kT = tsm + 128 * TP;   // [128][TP]: channel-major key tile
  const int tid = threadIdx.x, ty = tid >> 4, tx = tid & 15;
  const int h = blockIdx.y;
  const int64_t q0 = (int64_t)blockIdx.x * TQ;
  for (int i = tid; i < TQ * 32; i += 256) {  // 4 channels at a time, lanes over queries
    const int qi = i % TQ, c4 = i / TQ;
    float4 f = make_float4(0.f, 0.f, 0.f, 0.f);
    if (q0 + qi < Nq) {
      const uint2 w = *reinterpret_cast<const uint2*>(q + ((size_t)(q0 + qi) * H + h) * 128 + 4 * c4);
      f = make_float4(__uint_as_float(w.x << 16), __uint_as_float(w.x & 0xFFFF0000u), __uint_as_float(w.y << 16),
                      __uint_as_float(w.y & 0xFFFF0000u));
    }
    qT[(4 * c4) * TP + qi] = f.x;
    qT[(4 * c4 + 1) * TP + qi] = f.y;
    qT[(4 * c4 + 2) * TP + qi] = f.z;
    qT[(4 * c4 + 3) * TP + qi] = f.w;
  }
  float best[4];
  int bj[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    best[i] = -INFINITY;
    bj[i] = 0;
  }
  for (int64_t k0 = 0; k0 < Nk; k0 += TK) {
    __syncthreads();
    for (int i = tid; i < TK * 32; i += 256) {
      const int kj = i % TK, c4 = i / TK;
      float4 f = make_float4(0.f, 0.f, 0.f, 0.f);
      if (k0 + kj < Nk) f = *reinterpret_cast<const float4*>(keys + ((size_t)(k0 + kj) * H + h) * 128 + 4 * c4);
      kT[(4 * c4) * TP + kj] = f.x;
      kT[(4 * c4 + 1) * TP + kj] = f.y;
      kT[(4 * c4 + 2) * TP + kj] = f.z;
      kT[(4 * c4 + 3) * TP + kj] = f.w;
    }
    __syncthreads();
    float acc[4][4];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int j = 0; j < 4; ++j) acc[i][j] = 0.0f;
#pragma unroll 8
    for (int c = 0; c < 128; ++c) {
      const float4 qv = *reinterpret_cast<const float4*>(qT + c * TP + 4 * ty);
      const float4 kv = *reinterpret_cast<const float4*>(kT + c * TP + 4 * tx);
      const float qa[4] = {qv.x, qv.y, qv.z, qv.w}, ka[4] = {kv.x, kv.y, kv.z, kv.w};
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(qa[i], ka[j], acc[i][j]);
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int64_t kj = k0 + 4 * tx + j;
      if (kj < Nk)
#pragma unroll
        for (int i = 0; i < 4; ++i)
          if (acc[i][j] > best[i]) {  // keys arrive in increasing order: the first of equal logits stays
            best[i] = acc[i][j];
            bj[i] = (int)kj;
          }
    }
  }
  // the 16 threads of a query group hold disjoint key subsets: reduce, ties to the lower index
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    float b = best[i];
    int j = bj[i];
#pragma unroll
    for (int o = 8; o; o >>= 1) {
      const float ob = __shfl_xor_sync(0xFFFFFFFFu, b, o);
      const int oj = __shfl_xor_sync(0xFFFFFFFFu, j, o);
      if (ob > b || (ob == b && oj < j) || (b != b && ob == ob)) {
        b = ob;
        j = oj;
      }
    }
    const int64_t qi = q0 + 4 * ty + i;
    if (tx == 0 && qi < Nq) idx[(size_t)h * Nq + qi] = j;
  }
}

}  // namespace

cudaError_t launch_dequant(const DequantArgs& a, cudaStream_t st) {
  if (a.N == 0) return cudaSuccess;
  dim3 grid((unsigned)((a.N + 7) / 8), (unsigned)a.L.H);
  dequant_kernel<<<grid, 256, 0, st>>>(a);
  return cudaGetLastError();
}

}  // namespace qwm

extern "C" QWM_API qwm_status qwm_top1_keys(const qwm_config* cfg, const void* q, int64_t Nq, const float* keys,
                                            int64_t Nk, int32_t* idx, void* stream) {
  using namespace qwm;
  if (!cfg || !q || !keys || !idx || Nq < 1 || Nk < 1) return QWM_ERR_INVALID_ARG;
  if (!config_supported(cfg)) return QWM_ERR_UNSUPPORTED;
  if ((reinterpret_cast<uintptr_t>(q) & 15u) || (reinterpret_cast<uintptr_t>(keys) & 15u) ||
      (reinterpret_cast<uintptr_t>(idx) & 3u))
    return QWM_ERR_INVALID_ARG;
  if (Nq > ((int64_t)1 << 31) / TQ || Nk > ((int64_t)1 << 31) - TK) return QWM_ERR_UNSUPPORTED;
  const int smem = 2 * 128 * TP * 4;
  if (cudaFuncSetAttribute(top1_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess)
    return QWM_ERR_CUDA;
  dim3 grid((unsigned)((Nq + TQ - 1) / TQ), (unsigned)cfg->num_heads);
  top1_kernel<<<grid, 256, smem, static_cast<cudaStream_t>(stream)>>>(
      static_cast<const __nv_bfloat16*>(q), Nq, keys, Nk, cfg->num_heads, idx);
  return cudaGetLastError() == cudaSuccess ? QWM_OK : QWM_ERR_CUDA;
}
