// append_full.cu -- the full quadratic form of the App. C.4 ablation for the
// Keys' top-M candidates (qwm_quantize_append_full).
//
// The candidate filter (append.cu) screens the Keys with the tensor cores on
// B = M mu_j and A_j = mu_j^T M mu_j under a bound that covers the full
// form's fp32 evaluation; what it cannot decide it records as a band of at
// most kBand centroids (or every centroid).  This kernel runs between the
// filter and the quantize kernel: each such Key row gets the exact full form
// of its band members in the oracle's order -- e = k - mu_j (exact for bf16
// operands), t_c = sum_c' M_cc' e_c' and d_j = sum_c e_c t_c, one fused
// multiply-add per term in index order -- and its record is rewritten as the
// decided top-M (the M smallest (d_j, j), ties to the lower index).  The QSAC
// score and everything after use w as before.
#include "ptx_sm103.cuh"
#include "qwm_internal.cuh"

namespace qwm {
namespace {

constexpr int RT = 128;  // one thread per token row of a 128-token tile

// e of the thread's row sits in shared memory as column `tid` of [128][RT]
// (conflict-free: lane i reads bank i).
__device__ __forceinline__ float exact_dq_full(const __nv_bfloat16* k, const __nv_bfloat16* mu, const float* Mh,
                                               float* es) {
#pragma unroll 4
  for (int ch = 0; ch < 16; ++ch) {
    const uint4 kv = __ldg(reinterpret_cast<const uint4*>(k + ch * 8));
    const uint4 mv = __ldg(reinterpret_cast<const uint4*>(mu + ch * 8));
    const uint32_t kw[4] = {kv.x, kv.y, kv.z, kv.w}, mw[4] = {mv.x, mv.y, mv.z, mv.w};
#pragma unroll
    for (int p = 0; p < 4; ++p) {
      es[(ch * 8 + 2 * p) * RT] = __fsub_rn(__uint_as_float(kw[p] << 16), __uint_as_float(mw[p] << 16));
      es[(ch * 8 + 2 * p + 1) * RT] =
          __fsub_rn(__uint_as_float(kw[p] & 0xFFFF0000u), __uint_as_float(mw[p] & 0xFFFF0000u));
    }
  }
  float acc = 0.0f;
#pragma unroll 1
  for (int c = 0; c < 128; c += 4) {
    // four rows of M, four independent t_c chains, each in c' order
    const float4* M0 = reinterpret_cast<const float4*>(Mh + (size_t)c * 128);
    float t0 = 0.0f, t1 = 0.0f, t2 = 0.0f, t3 = 0.0f;
#pragma unroll 8
    for (int c4 = 0; c4 < 32; ++c4) {
      const float4 a0 = __ldg(M0 + c4), a1 = __ldg(M0 + 32 + c4), a2 = __ldg(M0 + 64 + c4), a3 = __ldg(M0 + 96 + c4);
      const float e0 = es[(4 * c4) * RT], e1 = es[(4 * c4 + 1) * RT], e2 = es[(4 * c4 + 2) * RT],
                  e3 = es[(4 * c4 + 3) * RT];
      t0 = __fmaf_rn(a0.x, e0, t0); t1 = __fmaf_rn(a1.x, e0, t1); t2 = __fmaf_rn(a2.x, e0, t2); t3 = __fmaf_rn(a3.x, e0, t3);
      t0 = __fmaf_rn(a0.y, e1, t0); t1 = __fmaf_rn(a1.y, e1, t1); t2 = __fmaf_rn(a2.y, e1, t2); t3 = __fmaf_rn(a3.y, e1, t3);
      t0 = __fmaf_rn(a0.z, e2, t0); t1 = __fmaf_rn(a1.z, e2, t1); t2 = __fmaf_rn(a2.z, e2, t2); t3 = __fmaf_rn(a3.z, e2, t3);
      t0 = __fmaf_rn(a0.w, e3, t0); t1 = __fmaf_rn(a1.w, e3, t1); t2 = __fmaf_rn(a2.w, e3, t2); t3 = __fmaf_rn(a3.w, e3, t3);
    }
    acc = __fmaf_rn(es[c * RT], t0, acc);   // d = sum_c e_c t_c in c order
    acc = __fmaf_rn(es[(c + 1) * RT], t1, acc);
    acc = __fmaf_rn(es[(c + 2) * RT], t2, acc);
    acc = __fmaf_rn(es[(c + 3) * RT], t3, acc);
  }
  return acc;
}

__global__ void __launch_bounds__(RT) full_rescore(const AppendArgs a) {
  extern __shared__ float sE[];  // [128][RT]
  const Layout& L = a.L;
  const int h = blockIdx.y, tile = blockIdx.x;
  const int64_t t = (int64_t)tile * 128 + threadIdx.x;
  if (t >= a.N) return;
  uint8_t* rec = a.base + head_offset(L, a.slot, h) + L.tiles_off + (int64_t)tile * L.tile_bytes + L.k_codes +
                 threadIdx.x * 32;
  uint8_t r[32];
  *reinterpret_cast<uint4*>(r) = *reinterpret_cast<const uint4*>(rec);
  *reinterpret_cast<uint4*>(r + 16) = *reinterpret_cast<const uint4*>(rec + 16);
  const int C = L.C, Mc = a.M;
  const int n = r[0];
  if (n == Mc) return;  // decided by the filter
  const bool band = n >= Mc && n <= kBand;
  const int cnt = band ? n : C;
  const __nv_bfloat16* k = a.k + ((size_t)t * L.H + h) * 128;
  const __nv_bfloat16* tab = a.kc + (size_t)h * C * 128;
  const float* Mh = a.Mq + (size_t)h * 128 * 128;
  float bv[kMaxFilterM];
  int bj[kMaxFilterM];
#pragma unroll
  for (int s = 0; s < kMaxFilterM; ++s) { bv[s] = INFINITY; bj[s] = 0x7FFFFFFF; }
  for (int m = 0; m < cnt; ++m) {  // ascending j in both cases
    int j = m;
    if (band) {
#pragma unroll
      for (int i = 0; i < kBand; ++i)
        if (i == m) j = r[1 + i];
    }
    if (j >= C) j = C - 1;  // a record left stale by a timed-out filter stays inside the table
    float v = exact_dq_full(k, tab + (size_t)j * 128, Mh, sE + threadIdx.x);
    int jj = j;
    // insert among the Mc smallest (value, index); an equal value stays behind
#pragma unroll
    for (int s = 0; s < kMaxFilterM; ++s) {
      if (s < Mc && v < bv[s]) {
        const float ov = bv[s];
        const int oj = bj[s];
        bv[s] = v;
        bj[s] = jj;
        v = ov;
        jj = oj;
      }
    }
  }
  r[0] = (uint8_t)Mc;
#pragma unroll
  for (int s = 0; s < kMaxFilterM; ++s)
    if (s < Mc) r[1 + s] = (uint8_t)bj[s];
  *reinterpret_cast<uint4*>(rec) = *reinterpret_cast<const uint4*>(r);
  *reinterpret_cast<uint4*>(rec + 16) = *reinterpret_cast<const uint4*>(r + 16);
}

}  // namespace

cudaError_t launch_full_rescore(const AppendArgs& a, cudaStream_t st) {
  const int tiles = (int)((a.N + 127) / 128);
  constexpr int smem = 128 * RT * 4;
  cudaError_t e = cudaFuncSetAttribute(full_rescore, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  full_rescore<<<dim3((unsigned)tiles, (unsigned)a.L.H), RT, smem, st>>>(a);
  return cudaGetLastError();
}

}  // namespace qwm
