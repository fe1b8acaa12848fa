// attend.cu -- attention of new queries over the packed 2-bit cache and the
// active bf16 chunk, on the sm_103a tensor cores (tcgen05 + TMEM), one CTA
// pair (a 2-CTA cluster on two SMs) per 512 queries of one head.
//
// Each CTA of the pair owns 256 queries (two 128-row Q tiles).  The pair
// shares its K/V work through paired MMAs (cta_group::2): the leader issues
// M = 256 MMAs whose A rows are the two CTAs' Q (or P) tiles and whose B
// operand is split between the CTAs along N, so each CTA rebuilds only half
// of every 128-key tile -- keys 64c..64c+63 of K_hat0 and C_hat, channels
// 64c..64c+63 of V_hat for all 128 keys (c = the CTA's rank) -- while each
// SM still runs its full share of tensor work.  18 warps per CTA with fixed
// roles that hand work to each other through mbarriers:
//   warps 0-3, 4-7   softmax of Q tile 0 / 1: thread = query row; reads its
//                    logit row S_i from TMEM, keeps the running max and sum,
//                    writes P_i as f16 back into the same TMEM columns, and
//                    at chunk boundaries moves Q U_r of the next chunk
//                    (Sec. 4.2 Eq. 17; computed by the tensor cores into
//                    spare S_i columns) into the extra Q operand columns;
//   warps 8-11       rebuild this CTA's 64 keys of K_hat0 = mu_id + s (q - z)
//                    (Sec. 2 Eq. 4) of each 128-key tile into a 2-stage
//                    shared-memory ring, plus their r PSAC columns
//                    C_hat = t * sigma (Eq. 16), and at a chunk's first tile
//                    its U_r^T as the B operand of the Q U_r MMA;
//   warps 12-15      rebuild this CTA's 64 channels of V_hat (same
//                    reconstruction, no PSAC) for all 128 keys;
//   warp 16          allocates the pair's TMEM; in the leader it runs the
//                    issue loop and one elected lane issues every MMA:
//                    Q_i U_r once per chunk,
//                    S_i = [Q_i | Q_i U_r] [K_hat0 | C_hat]^T
//                    (the PSAC logit term rides along as extra reduction
//                    columns) and O_i += P_i V_hat with P_i read straight from
//                    TMEM; in the follower it relays the K stages' hand-offs;
//   warp 17          in the follower, relays the V stages' hand-offs.
// Rebuild and softmax warps report to the leader's mbarriers (one arrival per
// warp; the follower's softmax warps remotely, its rebuild warps through the
// relays); MMA completions are committed to the mbarriers of both CTAs.
// TMEM (512 columns per CTA): S0 | S1 | O0 | O1, 128 fp32 columns each; P_i
// aliases the first 64 columns of S_i.  MMAs of one thread execute in issue
// order, so S_i of the next tile never overtakes the P_i V_hat MMA that reads
// P_i.  The O accumulator is rescaled only when the running maximum grows by
// more than 2^8 (every P stays <= 2^8).  Operands are binary16 with fp32
// accumulation: the bf16 rate with 8x finer rounding of the rebuilt keys.
// Every mbarrier wait is bounded; a wait that runs out records
// QWM_ERR_TIMEOUT in the cache's status word and that role leaves its loop.
#include <cstring>

#include "ptx_sm103.cuh"
#include "qwm_internal.cuh"

namespace qwm {
namespace {

using namespace ptx;

constexpr int kWarps = 18;
constexpr int NT = kWarps * 32;
constexpr int W_DQV = 12, W_MMA = 16;
constexpr float kTauLog2 = 8.0f;
constexpr int BLK = 16384;               // 128 rows x 128 bytes, 128-byte swizzled
constexpr int HBLK = 8192;               // 64 rows x 128 bytes
constexpr int OFF_Q = 0;                 // Q0 (2 blocks), Q1 (2 blocks)
constexpr int OFF_QU = 4 * BLK;          // Q_i U_r at columns [i*rpad, (i+1)*rpad)
constexpr int OFF_K = 5 * BLK;           // this CTA's 64 keys of K_hat0: stage s, block kb at (2s + kb) * HBLK
constexpr int OFF_C = OFF_K + 4 * HBLK;  // their C_hat (64 rows), stage s at columns [s*rpad, (s+1)*rpad)
constexpr int OFF_V = OFF_C + HBLK;      // this CTA's 64 channels of V_hat (128 keys), stage s at s * BLK
constexpr int OFF_U = OFF_V + 2 * BLK;    // U_r^T operand of the Q U_r MMA: chunk parity p, block kb at (2p + kb) * 4 KB
constexpr int UBLK = 4096;                 // 32 rows x 128 bytes
constexpr int OFF_BAR = OFF_U + 4 * UBLK;
// B_KRDY / B_VRDY: the follower's rebuilt stages, relayed to the leader's
// B_KFULL / B_VFULL by the follower's warps 16 and 17.
enum { B_KFULL = 0, B_KEMPTY = 2, B_VFULL = 4, B_VEMPTY = 6, B_SFULL = 8, B_PFULL = 10, B_QU = 12, B_OFINAL = 14,
       B_QUMMA = 15, B_KRDY = 17, B_VRDY = 19, NBAR = 21 };
static_assert(NBAR * 8 + 16 <= 256, "barrier area");
constexpr int SMEM_BYTES = OFF_BAR + 256 + 1024;  // + alignment slack

// 8 f16 (16 bytes) of row `row`, chunk `ch` (columns 8ch..8ch+7) into a run of
// 128-byte-swizzled blocks of `rows` rows x 64 columns.
__device__ __forceinline__ void st_chunk(uint8_t* base, int row, int ch, uint4 v, int rows = 128) {
  const int kb = ch >> 3, pos = (ch & 7) ^ (row & 7);
  *reinterpret_cast<uint4*>(base + kb * rows * 128 + row * 128 + pos * 16) = v;
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

// 32-byte read-only global load (address 32-byte aligned).
__device__ __forceinline__ void ldg32B(const void* p, uint32_t (&r)[8]) {
  asm volatile("ld.global.nc.v8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7])
               : "l"(p));
}

__device__ __forceinline__ uint32_t h2u(__half2 h) { return *reinterpret_cast<uint32_t*>(&h); }
__device__ __forceinline__ __half2 u2h(uint32_t u) { return *reinterpret_cast<__half2*>(&u); }

__device__ __forceinline__ void zero_row(uint8_t* dst, int row, int ch0, int nch) {
  for (int ch = ch0; ch < ch0 + nch; ++ch) st_chunk(dst, row, ch, make_uint4(0, 0, 0, 0));
}

// A row of 128 bf16 into the f16 operand; values beyond the binary16 range
// saturate and set `bad`.
__device__ __forceinline__ void copy_row(uint8_t* dst, int row, const __nv_bfloat16* src, bool& bad) {
#pragma unroll
  for (int ch = 0; ch < 16; ++ch) st_chunk(dst, row, ch, bf16x8_to_f16x8_sat(ldg16(src + ch * 8), bad));
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
  // the units [u0, u_end) (a part's range of chunks)
  __device__ __forceinline__ void init(const AttendArgs& a, const AttendSlots& S, int h, int u0, int u_end) {
    u = u0; tl = 0; n_units = u_end; ntiles = 0;
    if (u0 < u_end) { U = unit_at(a, S, u0, h); ntiles = (U.ntok + 127) / 128; }
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

// Q_i U_r of one query row, computed by the tensor cores into TMEM columns
// [64, 64 + rpad) of S_i, as f16 into the shared Q U_r block at columns
// [i*rpad, (i+1)*rpad) (the A operand of the PSAC reduction columns).
__device__ __forceinline__ void qu_to_smem(uint8_t* sQU, int i, int row, uint32_t tqu, int rpad) {
  float v[32];
  tmem_ld32(tqu, v);
#pragma unroll
  for (int c2 = 0; c2 < 4; ++c2) {
    if (c2 * 8 < rpad) {
      uint32_t w4[4];
#pragma unroll
      for (int p = 0; p < 4; ++p) w4[p] = pack_f16(v[c2 * 8 + 2 * p], v[c2 * 8 + 2 * p + 1]);
      st_chunk(sQU, row, (i * rpad) / 8 + c2, make_uint4(w4[0], w4[1], w4[2], w4[3]));
    }
  }
}

// SF: the slot's scale format (0: binary16 group scales; 1: uint8 group codes
// times a binary16 secondary scale per token, App. D.1).
// PARTS: the launch of the tail units' parts (see plan_attend) instead of
// the whole units.
template <int SF, bool PARTS>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(NT, 1)
    attend_kernel(const AttendArgs a, const AttendSlots S) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  const Layout& L = a.L;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  // Whole units: grid x = 2 * (block of 512 queries) + rank (the CTA pair of
  // a cluster), y = head, every key (the pairs of one head run close together
  // and share its packed tiles through L2).  Parts: grid x = 2 * (part index)
  // + rank over the tail units (the units from n_whole on, nparts parts each,
  // every part over a contiguous range of the key units: cached chunks, then
  // the active chunk), whose partial results a third kernel combines.
  const int P = blockIdx.x >> 1;
  const int wunit = PARTS ? a.n_whole + P / a.nparts : (int)blockIdx.y * a.bph + P;
  const int part = PARTS ? P % a.nparts : 0;
  const int h = PARTS ? wunit / a.bph : (int)blockIdx.y;
  const int H = L.H, r = L.r;
  const int rpad = r == 8 ? 16 : r;
  const int gshift = L.G == 32 ? 5 : 6;
  const uint32_t rank = cluster_rank();  // 0: leader
  const int64_t pair0 = PARTS ? (int64_t)(wunit - h * a.bph) * 512 : (int64_t)P * 512;
  const int64_t q0 = pair0 + 256 * rank;
  // Q tiles the pair runs: the second is left out when neither CTA has a
  // query in it (the tail of the query range), halving that pair's MMA and
  // softmax work.
  const int nqt = pair0 + 128 < a.Nq ? 2 : 1;
  const int n_all = S.n + (a.Ncur > 0 ? 1 : 0);
  // this pair's key units [cu0, cu1)
  const int cu0 = PARTS ? (int)((int64_t)part * n_all / a.nparts) : 0;
  const int cu1 = PARTS ? (int)((int64_t)(part + 1) * n_all / a.nparts) : n_all;

  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + OFF_BAR);
  uint32_t* tslot = reinterpret_cast<uint32_t*>(sm + OFF_BAR + NBAR * 8);
  int* s_err = reinterpret_cast<int*>(sm + OFF_BAR + NBAR * 8 + 8);
  volatile int* s_bad = reinterpret_cast<volatile int*>(sm + OFF_BAR + NBAR * 8 + 12);  // an input beyond binary16
  auto bar = [&](int i) { return smem_u32(bars + i); };
  // One arrival per warp on the leader's copy of barrier i, after every lane's
  // writes (the caller fences them for their consumer first).
  auto arrive_leader = [&](int i) {
    __syncwarp();
    if (lane == 0) {
      if (rank == 0) mbar_arrive(bar(i));
      else mbar_arrive_cluster(mapa(bar(i), 0));
    }
  };
  // Hand-off of P_i (tensor memory the softmax warps wrote with tcgen05.st,
  // waited for and fenced before the hand-off) to the leader's MMA warp.  In
  // the leader each warp arrives on barrier b.  In the follower the four
  // warps meet at named barrier nb, which also ANDs their `ok` flags so that
  // a timed-out wait ends the role in all four warps together, and one lane
  // arrives for all of them with a relaxed cluster-scope arrive (the payload
  // needs no release of other memory accesses).  Returns the common flag.
  auto handoff = [&](int b, int nb, bool okw) -> bool {
    if (rank == 0) {
      __syncwarp();
      if (okw && lane == 0) mbar_arrive(bar(b));
      return okw;
    }
    const bool all = named_bar_and(nb, 128, okw);
    if (all && (warp & 3) == 0 && lane == 0) mbar_arrive_cluster_relaxed(mapa(bar(b), 0));
    return all;
  };

  // Hand-off of a rebuilt K/V stage: each warp arrives at CTA scope, in the
  // leader on the leader's barrier b, in the follower on the local barrier
  // rb that the follower's relay warp forwards to b (so the rebuild warps
  // never wait for a cluster-scope release).
  auto stage_done = [&](int b, int rb, bool okw) -> bool {
    __syncwarp();
    if (okw && lane == 0) mbar_arrive(bar(rank == 0 ? b : rb));
    return okw;
  };

  if (tid == 0) {
    for (int s = 0; s < 2; ++s) {
      mbar_init(bar(B_KFULL + s), 5);    // 4 leader rebuild warps + 1 follower arrival
      mbar_init(bar(B_KEMPTY + s), 1);   // pair MMA commit, both CTAs
      mbar_init(bar(B_VFULL + s), 5);
      mbar_init(bar(B_VEMPTY + s), 1);
      mbar_init(bar(B_SFULL + s), 1);
      mbar_init(bar(B_PFULL + s), 5);    // 4 leader softmax warps + 1 follower arrival
      mbar_init(bar(B_QU + s), 8);
      mbar_init(bar(B_KRDY + s), 4);     // the follower's four K rebuild warps
      mbar_init(bar(B_VRDY + s), 4);
    }
    mbar_init(bar(B_OFINAL), 1);
    mbar_init(bar(B_QUMMA), 1);         // Q_i U_r MMA commit, both CTAs
    mbar_init(bar(B_QUMMA + 1), 1);
    *s_err = 0;
    *s_bad = 0;
    fence_mbar_init();
  }
  if (warp == W_MMA) {
    tmem_alloc2(smem_u32(tslot), 512);
    tmem_relinquish2();
  }
  tc_fence_before();
  cluster_sync();  // both CTAs' barriers exist before any remote arrival
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
    bool qbad = false;
    if (qvalid) copy_row(sQi, row, qrow, qbad);
    else zero_row(sQi, row, 0, 16);
    if (qbad) *s_bad = 1;
    fence_proxy_async_smem();
    arrive_leader(B_QU + i);  // Q_i is in place
    // Q_i U_r of each chunk that carries PSAC columns: the MMA warp computes
    // it into columns 64.. of S_i (free while S_i is not in use); this group
    // moves it into the shared A operand of the extra reduction columns.
    if (i < nqt) {
    uint32_t qum = 0;  // completed Q_i U_r MMAs
    auto take_qu = [&]() -> bool {
      bool okw = __all_sync(0xFFFFFFFFu, mbar_wait(bar(B_QUMMA + i), qum & 1, a.wait_ns));
      if (okw) {
        ++qum;
        tc_fence_after();
        qu_to_smem(sm + OFF_QU, i, row, tS + 64, rpad);
        tc_fence_before();
        fence_proxy_async_smem();
      }
      if (rank == 1) okw = named_bar_and(1 + i, 128, okw);  // the group leaves together
      if (okw) arrive_leader(B_QU + i);
      return okw;
    };

    const float sl2 = a.sm_scale * 1.4426950408889634f;
    float m_run = -INFINITY, l_run = 0.0f;
    uint32_t jt = 0;
    bool ok = true;
    if (cu0 < cu1 && unit_at(a, S, cu0, h).psac) ok = take_qu();
    for (int u = cu0; u < cu1 && ok; ++u) {
      const Unit U = unit_at(a, S, u, h);
      const int ntiles = (U.ntok + 127) / 128;
      for (int tl = 0; tl < ntiles; ++tl, ++jt) {
        const int nvalid = min(128, U.ntok - tl * 128);
        const bool okw = __all_sync(0xFFFFFFFFu, mbar_wait(bar(B_SFULL + i), jt & 1, a.wait_ns));
        if (okw) {
          tc_fence_after();
          // ---- row maximum: four reducing TMEM loads and one wait
          const bool full = nvalid == 128;
          float va[32], vb[32];
          float mt = -INFINITY;
          if (full) {
            mt = tmem_max128(tS);
          } else {
  #pragma unroll 1
            for (int cp = 0; cp < 2; ++cp) {
              tmem_ld32x2(tS + 64 * cp, tS + 64 * cp + 32, va, vb);
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
  #pragma unroll 1
            for (int cb = 0; cb < 8; ++cb) {
              uint32_t t[16];
              tmem_ld16(tO + cb * 16, t);
  #pragma unroll
              for (int e = 0; e < 16; ++e) t[e] = __float_as_uint(__uint_as_float(t[e]) * alpha);
              tmem_st16(tO + cb * 16, t);
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
  #pragma unroll 1
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
        }
        ok = handoff(B_PFULL + i, 1 + i, okw);
        if (!ok) break;
      }
      if (ok && u + 1 < cu1 && unit_at(a, S, u + 1, h).psac) ok = take_qu();
    }
    if (ok) ok = __all_sync(0xFFFFFFFFu, mbar_wait(bar(B_OFINAL), 0, a.wait_ns));
    if (ok && !PARTS) {
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
    } else if (ok) {
      // a part of a tail unit: the unnormalised O row, the running maximum and
      // sum, for the combining kernel
      tc_fence_after();
      const size_t prow = ((size_t)(blockIdx.x >> 1) * 512 + 256 * rank + 128 * i + row);
      float v[32];
#pragma unroll
      for (int cb = 0; cb < 4; ++cb) {
        tmem_ld32(tO + cb * 32, v);
        if (qvalid) {
          float4* dst = reinterpret_cast<float4*>(a.part_o + prow * 128 + cb * 32);
#pragma unroll
          for (int k = 0; k < 8; ++k) dst[k] = make_float4(v[4 * k], v[4 * k + 1], v[4 * k + 2], v[4 * k + 3]);
        }
      }
      if (qvalid) *reinterpret_cast<float2*>(a.part_ml + prow * 2) = make_float2(m_run, l_run);
    } else {
      *s_err = 1;
    }
    // Off the critical path: this CTA's share of the active chunk's rows of
    // head h (the rebuild converts them with saturation) is checked for values
    // beyond the binary16 range, which only the status word reports.
    if (a.Ncur > 0 && (!PARTS || (int)(blockIdx.x >> 1) % a.nparts == 0)) {
      const int64_t gx = 2 * (int64_t)a.bph, bx = 2 * (pair0 >> 9) + rank;
      const int64_t per = (a.Ncur + gx - 1) / gx;
      const int64_t r0 = bx * per, r1 = min(a.Ncur, r0 + per);
      uint32_t mag = 0u;
      for (int64_t e = r0 * 16 + (tid & 255); e < r1 * 16; e += 256) {
        const int64_t tok = e >> 4;
        const int ch = (int)(e & 15);
        const uint4 kv = ldg16(a.kcur + ((size_t)tok * H + h) * 128 + ch * 8);
        const uint4 vv = ldg16(a.vcur + ((size_t)tok * H + h) * 128 + ch * 8);
        const uint32_t w8[8] = {kv.x, kv.y, kv.z, kv.w, vv.x, vv.y, vv.z, vv.w};
#pragma unroll
        for (int i = 0; i < 8; ++i) mag = vmax_u16x2(mag, w8[i] & 0x7FFF7FFFu);
      }
      if (bf16x2_out_of_f16(mag)) *s_bad = 1;
    }
    }
  } else if (warp < W_DQV) {
    // ------------------------------------------------------------ K_hat0 + C_hat of this CTA's 64 keys (warps 8-11)
    // Four lanes per key row: lane q of a quad rebuilds channels 16q..16q+15
    // and 64+16q..64+16q+15 (chunks 2q, 2q+1, 8+2q, 9+2q) from 32-byte
    // centroid slices, and PSAC columns 8q..8q+7.  Warp w covers local rows
    // 16w..16w+15 (tile rows 64c + local) in two passes of 8 rows, all loads
    // of the tile in one round.  Ids and zero-points of the next tile are
    // loaded one tile ahead.
    const int q = lane & 3, rr = lane >> 2;
    const int wrow = (warp & 3) * 16 + rr;  // local row of pass p: wrow + 8p
    const int tro = 64 * (int)rank;         // tile row of local row 0
    TileCursor cur;
    cur.init(a, S, h, cu0, cu1);
    auto load_ids = [&](const TileCursor& c) -> uint32_t {  // 2 ids | 2 zero bytes << 16
      uint32_t v = 0;
      if (c.valid() && c.U.hb) {
        const uint8_t* tb = c.U.hb + L.tiles_off + (int64_t)c.tl * L.tile_bytes;
        const int nv = c.nvalid();
#pragma unroll
        for (int p = 0; p < 2; ++p) {
          const int trw = tro + wrow + 8 * p;
          if (trw < nv)
            v |= ((uint32_t)tb[L.k_ids + trw] << (8 * p)) | ((uint32_t)tb[L.k_zeros + (int64_t)trw * L.zb] << (16 + 8 * p));
        }
      }
      return v;
    };
    // the tile's PSAC keep mask (which rows its code and scale arrays hold),
    // loaded one tile ahead with the ids and used only in the next tile's
    // passes, so no warp waits for it
    auto load_pm = [&](const TileCursor& c) -> uint4 {
      uint4 v = make_uint4(0u, 0u, 0u, 0u);
      if (c.valid() && c.U.hb && c.U.psac && q * 8 < r) v = ldg16(c.U.hb + L.pmask + (int64_t)c.tl * 16);
      return v;
    };
    uint32_t idn = load_ids(cur);
    uint4 pmn = load_pm(cur);
    uint32_t jt = 0;
    bool ok = true;
    const int kt = tid - 32 * 8;  // 0..127
    if (rank == 1)  // the follower's half of the U_r^T operand (rows 32..63 of N = 64) stays zero
      for (int idx = kt; idx < 4 * UBLK / 16; idx += 128)
        *reinterpret_cast<uint4*>(sm + OFF_U + 16 * idx) = make_uint4(0u, 0u, 0u, 0u);
    while (cur.valid()) {
      const uint32_t idc = idn;
      const uint4 pmc = pmn;
      TileCursor nc = cur;
      nc.next(a, S, h);
      const int st = jt & 1;
      const uint32_t ph = (jt >> 1) & 1;
      const int nv = cur.nvalid();
      const bool okw = __all_sync(0xFFFFFFFFu, mbar_wait(bar(B_KEMPTY + st), ph ^ 1, a.wait_ns));
      if (okw) {
        uint8_t* dst = sm + OFF_K + 2 * st * HBLK;
        const uint8_t* tb = cur.U.hb ? cur.U.hb + L.tiles_off + (int64_t)cur.tl * L.tile_bytes : nullptr;
        const uint8_t* tab = cur.U.hb ? cur.U.hb + L.ktab : nullptr;
        if (rank == 0 && cur.tl == 0 && cur.U.psac) {
          // U_r^T of this chunk (rows j < r, zero up to 32) as f16 into the
          // chunk-parity buffer read by the Q U_r MMA; published with this tile.
          uint8_t* sU = sm + OFF_U + (cur.u & 1) * 2 * UBLK;
          const uint8_t* ut = cur.U.hb + L.ut;
  #pragma unroll 1
          for (int idx = kt; idx < 32 * 16; idx += 128) {
            const int j = idx >> 4, ch = idx & 15;
            bool ubad = false;
            const uint4 v = j < r ? bf16x8_to_f16x8_sat(ldg16(ut + ((int64_t)j * 128 + ch * 8) * 2), ubad) : make_uint4(0u, 0u, 0u, 0u);
            if (ubad) *s_bad = 1;
            st_chunk(sU, j, ch, v, 32);
          }
        }
        const bool psac_lane = cur.U.psac && q * 8 < r;
        // entries of the lane's two rows in the tile's PSAC arrays (-1: none):
        // the rows lie in this CTA's half of the tile (mask words 2c, 2c + 1),
        // entry = kept rows below the row
        int pe0 = -1, pe1 = -1;
        if (psac_lane) {
          const uint32_t lo = rank ? pmc.z : pmc.x, hi = rank ? pmc.w : pmc.y;
          const int base = rank ? __popc(pmc.x) + __popc(pmc.y) : 0;
          const int b0 = wrow & 31, b1 = (wrow + 8) & 31;
          const uint32_t w0 = wrow >= 32 ? hi : lo, w1 = wrow + 8 >= 32 ? hi : lo;
          const int o0 = base + (wrow >= 32 ? __popc(lo) : 0), o1 = base + (wrow + 8 >= 32 ? __popc(lo) : 0);
          if ((w0 >> b0) & 1u) pe0 = o0 + __popc(w0 & ((1u << b0) - 1u));
          if ((w1 >> b1) & 1u) pe1 = o1 + __popc(w1 & ((1u << b1) - 1u));
        }
        // One row per pass (loads, then its reconstruction); the pass loop is
        // kept rolled so that the four roles' hot loops stay small enough for
        // the instruction caches.
  #pragma unroll 1
        for (int p = 0; p < 2; ++p) {
          const int lr = wrow + 8 * p, trw = tro + lr;
          const bool rv = trw < nv;
          uint32_t mv[2][8];  // [slice][words]
          uint32_t cwv[2] = {0u, 0u}, scv[2] = {0u, 0u};
          uint2 cfv = make_uint2(0u, 0u);  // PSAC INT8 codes 8q..8q+7 of the row
          uint32_t sgv = 0u;               // PSAC row scale (binary16 bits)
  #pragma unroll
          for (int sl = 0; sl < 2; ++sl)
  #pragma unroll
            for (int e = 0; e < 8; ++e) mv[sl][e] = 0u;
          if (rv) {
            if (tb) {
              const uint8_t* mu = tab + (int64_t)((idc >> (8 * p)) & 0xFFu) * 256;
              ldg32B(mu + 32 * q, mv[0]);
              ldg32B(mu + 128 + 32 * q, mv[1]);
              const uint8_t* cp = tb + L.k_codes + trw * 32;
              cwv[0] = __ldg(reinterpret_cast<const uint32_t*>(cp + 4 * q));
              cwv[1] = __ldg(reinterpret_cast<const uint32_t*>(cp + 16 + 4 * q));
              if constexpr (SF == 0) {
                const unsigned short* sp =
                    reinterpret_cast<const unsigned short*>(tb + L.k_scales + (int64_t)trw * L.ng * 2);
                scv[0] = __ldg(sp + ((16 * q) >> gshift));
                scv[1] = __ldg(sp + ((64 + 16 * q) >> gshift));
              } else {
                const uint8_t* cp8 = tb + L.k_scales + (int64_t)trw * L.ng;
                const __half s2 = __ushort_as_half(__ldg(reinterpret_cast<const unsigned short*>(tb + L.k_s2) + trw));
                scv[0] = __half_as_ushort(__hmul(__uint2half_rn(__ldg(cp8 + ((16 * q) >> gshift))), s2));
                scv[1] = __half_as_ushort(__hmul(__uint2half_rn(__ldg(cp8 + ((64 + 16 * q) >> gshift))), s2));
              }
              if (psac_lane) {
                // the tile's keep mask names the stored rows; row trw is entry e
                const int e = p ? pe1 : pe0;
                if (e >= 0) {
                  cfv = __ldg(reinterpret_cast<const uint2*>(tb + L.k_coef + (int64_t)e * r + q * 8));
                  sgv = __ldg(reinterpret_cast<const unsigned short*>(tb + L.k_sigma + e * 2));
                }
              }
            } else {
              const __nv_bfloat16* src = a.kcur + ((size_t)(cur.tl * 128 + trw) * H + h) * 128;
  #pragma unroll
              for (int sl = 0; sl < 2; ++sl) {
                const uint4 f0 = bf16x8_to_f16x8(ldg16(src + 64 * sl + 16 * q));
                const uint4 f1 = bf16x8_to_f16x8(ldg16(src + 64 * sl + 16 * q + 8));
                mv[sl][0] = f0.x; mv[sl][1] = f0.y; mv[sl][2] = f0.z; mv[sl][3] = f0.w;
                mv[sl][4] = f1.x; mv[sl][5] = f1.y; mv[sl][6] = f1.z; mv[sl][7] = f1.w;
              }
            }
          }
          const bool deq = tb && rv;
          const uint32_t zbyte = (idc >> (16 + 8 * p)) & 0xFFu;
  #pragma unroll
          for (int sl = 0; sl < 2; ++sl) {
            const int c0 = 8 * sl + 2 * q;  // first of the two chunks of this slice
            // f16 pairs mu + (q - z) s; a row of the active chunk (or a padding
            // row) passes through with s = 0 and z = q.
            const int g = (64 * sl + 16 * q) >> gshift;
            const uint32_t sb = deq ? scv[sl] : 0u;
            const __half2 s2 = u2h(sb | (sb << 16));
            const uint32_t zz = 0x6400u | ((zbyte >> (2 * g)) & 3u);
            const __half2 z2 = u2h(zz | (zz << 16));
            const uint32_t word = cwv[sl];
            uint32_t ow[8];
  #pragma unroll
            for (int k = 0; k < 8; ++k) {  // channel pairs (2k, 2k+1) of the 16-channel word
              const uint32_t qq = ((word >> (2 * k)) & 0x00030003u) | 0x64006400u;
              ow[k] = h2u(__hfma2(__hsub2(u2h(qq), z2), s2, u2h(mv[sl][k])));
            }
            st_chunk(dst, lr, c0, make_uint4(ow[0], ow[1], ow[2], ow[3]), 64);
            st_chunk(dst, lr, c0 + 1, make_uint4(ow[4], ow[5], ow[6], ow[7]), 64);
          }
          if (cur.U.psac && q * 8 < rpad) {
            // C_hat = t * sigma (Eq. 16), PSAC columns 8q..8q+7 of the row, in
            // f16: byte b of an INT8 code t becomes the f16 1024 + (t + 128)
            // (its byte XOR 0x80 under exponent bits 0x64), minus 1152 gives t
            // exactly, and one f16 multiply rounds t * sigma once.  Lanes past
            // r and padding rows hold zero codes and scale: zero columns.
            const __half2 sg2 = u2h(sgv | (sgv << 16));
            const __half2 off2 = u2h(0x64806480u);  // (1152, 1152)
            const uint32_t cwd[2] = {cfv.x ^ 0x80808080u, cfv.y ^ 0x80808080u};
            uint32_t w4[4];
  #pragma unroll
            for (int q2 = 0; q2 < 4; ++q2) {
              const uint32_t b0 = 2 * (q2 & 1);
              const uint32_t t2 = __byte_perm(cwd[q2 >> 1], 0x64646464u, b0 | (4u << 4) | ((b0 + 1) << 8) | (4u << 12));
              w4[q2] = h2u(__hmul2(__hsub2(u2h(t2), off2), sg2));
            }
            st_chunk(sm + OFF_C, lr, (st * rpad) / 8 + q, make_uint4(w4[0], w4[1], w4[2], w4[3]), 64);
          }
        }
        fence_proxy_async_smem();
      }
      if (!(ok = stage_done(B_KFULL + st, B_KRDY + st, okw))) break;
      // the next tile's ids and zero-points are fetched only now: a release
      // waits for every memory operation the thread has in flight
      idn = load_ids(nc);
      pmn = load_pm(nc);
      cur = nc;
      ++jt;
    }
    if (!ok) *s_err = 1;
  } else if (warp < W_MMA) {
    // ------------------------------------------------------------ V_hat, this CTA's 64 channels (warps 12-15)
    // Four lanes per key row: lane q rebuilds channels 64c+16q..64c+16q+15
    // (chunks 2q, 2q+1 of this CTA's V block) from one 32-byte centroid
    // slice.  Warp w covers rows 32w..32w+31 in four passes of 8 rows, two
    // passes per round of loads; ids and zero-points one tile ahead.
    const int q = lane & 3, rr = lane >> 2;
    const int wrow = (warp & 3) * 32 + rr;  // row of pass p: wrow + 8p
    const int c16 = 4 * (int)rank + q;      // this lane's 16-channel block of the row
    TileCursor cur;
    // an idle V role (the test hook of qwm_cache_set_idle_role) publishes no
    // tile: the MMA warp's bounded wait for the first one runs out
    cur.init(a, S, h, cu0, a.idle_role == QWM_ROLE_V_REBUILD ? cu0 : cu1);
    auto load_ids = [&](const TileCursor& c) -> uint64_t {  // 4 ids | 4 zero bytes << 32
      uint64_t v = 0;
      if (c.valid() && c.U.hb) {
        const uint8_t* tb = c.U.hb + L.tiles_off + (int64_t)c.tl * L.tile_bytes;
        const int nv = c.nvalid();
#pragma unroll
        for (int p = 0; p < 4; ++p) {
          const int row = wrow + 8 * p;
          if (row < nv)
            v |= ((uint64_t)tb[L.v_ids + row] << (8 * p)) | ((uint64_t)tb[L.v_zeros + (int64_t)row * L.zb] << (32 + 8 * p));
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
      const int st = jt & 1;
      const uint32_t ph = (jt >> 1) & 1;
      const int nv = cur.nvalid();
      const bool okw = __all_sync(0xFFFFFFFFu, mbar_wait(bar(B_VEMPTY + st), ph ^ 1, a.wait_ns));
      if (okw) {
        uint8_t* dst = sm + OFF_V + st * BLK;
        const uint8_t* tb = cur.U.hb ? cur.U.hb + L.tiles_off + (int64_t)cur.tl * L.tile_bytes : nullptr;
        const uint8_t* tab = cur.U.hb ? cur.U.hb + L.vtab : nullptr;
        const int g = (16 * c16) >> gshift;
  #pragma unroll 1
        for (int rd = 0; rd < 2; ++rd) {
          uint32_t mv[2][8];
          uint32_t cwv[2] = {0u, 0u}, scv[2] = {0u, 0u};
  #pragma unroll
          for (int pp = 0; pp < 2; ++pp) {
            const int p = 2 * rd + pp;
            const int row = wrow + 8 * p;
  #pragma unroll
            for (int e = 0; e < 8; ++e) mv[pp][e] = 0u;
            if (row < nv) {
              if (tb) {
                ldg32B(tab + (int64_t)((idc >> (8 * p)) & 0xFFu) * 256 + 32 * c16, mv[pp]);
                cwv[pp] = __ldg(reinterpret_cast<const uint32_t*>(tb + L.v_codes + row * 32 + 4 * c16));
                if constexpr (SF == 0) {
                  scv[pp] = __ldg(reinterpret_cast<const unsigned short*>(tb + L.v_scales + (int64_t)row * L.ng * 2) + g);
                } else {
                  const __half s2 = __ushort_as_half(__ldg(reinterpret_cast<const unsigned short*>(tb + L.v_s2) + row));
                  scv[pp] = __half_as_ushort(__hmul(__uint2half_rn(__ldg(tb + L.v_scales + (int64_t)row * L.ng + g)), s2));
                }
              } else {
                const __nv_bfloat16* src = a.vcur + ((size_t)(cur.tl * 128 + row) * H + h) * 128 + 16 * c16;
                const uint4 f0 = bf16x8_to_f16x8(ldg16(src)), f1 = bf16x8_to_f16x8(ldg16(src + 8));
                mv[pp][0] = f0.x; mv[pp][1] = f0.y; mv[pp][2] = f0.z; mv[pp][3] = f0.w;
                mv[pp][4] = f1.x; mv[pp][5] = f1.y; mv[pp][6] = f1.z; mv[pp][7] = f1.w;
              }
            }
          }
  #pragma unroll
          for (int pp = 0; pp < 2; ++pp) {
            const int p = 2 * rd + pp;
            const int row = wrow + 8 * p;
            // mu + (q - z) s; active-chunk and padding rows pass through with
            // s = 0 and zero codes and zero-points (the ids word is 0 there).
            const uint32_t zbyte = (uint32_t)((idc >> (32 + 8 * p)) & 0xFFu);
            const uint32_t sb = scv[pp];
            const __half2 s2 = u2h(sb | (sb << 16));
            const uint32_t zz = 0x6400u | ((zbyte >> (2 * g)) & 3u);
            const __half2 z2 = u2h(zz | (zz << 16));
            const uint32_t word = cwv[pp];
            uint32_t ow[8];
  #pragma unroll
            for (int k = 0; k < 8; ++k) {
              const uint32_t qq = ((word >> (2 * k)) & 0x00030003u) | 0x64006400u;
              ow[k] = h2u(__hfma2(__hsub2(u2h(qq), z2), s2, u2h(mv[pp][k])));
            }
            st_chunk(dst, row, 2 * q, make_uint4(ow[0], ow[1], ow[2], ow[3]));
            st_chunk(dst, row, 2 * q + 1, make_uint4(ow[4], ow[5], ow[6], ow[7]));
          }
        }
        fence_proxy_async_smem();
      }
      if (!(ok = stage_done(B_VFULL + st, B_VRDY + st, okw))) break;
      // the next tile's ids and zero-points are fetched only now: a release
      // waits for every memory operation the thread has in flight
      idn = load_ids(nc);
      cur = nc;
      ++jt;
    }
    if (!ok) *s_err = 1;
  } else {
    // ------------------------------------------------------------ MMA issue (leader, one warp)
    // Order per KV tile j: P0 V(j), S0(j+1), P1 V(j), S1(j+1), so that the
    // softmax of Q tile 0 on tile j+1 overlaps the softmax of Q tile 1 on
    // tile j (S_i(j+1) reuses the TMEM columns of P_i(j) after P_i V(j) has
    // read them: MMAs of one thread run in issue order).  The whole warp runs
    // the loop; one elected lane issues every MMA and commit.
    if (rank == 0 && warp == W_MMA) {
      const uint32_t e = elect_one();
      // operand descriptors: the base of each buffer once, then byte offsets
      // >> 4 added to the start-address field (every address stays below the
      // 256 KB that the 14-bit field covers)
      const uint64_t dQ = desc_sw128(smem_u32(sm + OFF_Q)), dQU = desc_sw128(smem_u32(sm + OFF_QU));
      const uint64_t dK = desc_sw128(smem_u32(sm + OFF_K)), dC = desc_sw128(smem_u32(sm + OFF_C));
      const uint64_t dV = desc_sw128(smem_u32(sm + OFF_V)), dU = desc_sw128(smem_u32(sm + OFF_U));
      auto off = [](int bytes) { return (uint64_t)(bytes >> 4); };
      constexpr uint32_t idS = idesc_f16(256, 128, false);
      constexpr uint32_t idQU = idesc_f16(256, 64, false);
      constexpr uint32_t idPV = idesc_f16(256, 128, true);
      auto wait_all = [&](int b, uint32_t ph) -> bool {
        return __all_sync(0xFFFFFFFFu, mbar_wait_cluster(bar(b), ph, a.wait_ns));
      };
      int total = 0;
      for (int u = cu0; u < cu1; ++u) total += (unit_at(a, S, u, h).ntok + 127) / 128;
      TileCursor sc;  // next tile to issue S for
      sc.init(a, S, h, cu0, cu1);
      uint32_t sjt = 0, qph[2] = {0, 0};
      bool ok = true;
      auto issue_S = [&](int i) -> bool {
        const int st = sjt & 1;
        const uint32_t ph = (sjt >> 1) & 1;
        if (i == 0 && !wait_all(B_KFULL + st, ph)) return false;
        if (sc.tl == 0 && sc.u == cu0) {  // Q_i in place
          if (!wait_all(B_QU + i, qph[i])) return false;
          qph[i] ^= 1;
        }
        if (sc.tl == 0 && sc.U.psac) {
          // Q_i U_r of this chunk into columns 64.. of S_i (N = 64: the
          // leader's 32 rows of U_r^T, the follower's zero rows): every MMA
          // that read S_i or Q_i U_r of the previous chunk was issued before.
          tc_fence_after();
          const uint64_t dUc = dU + off((sc.u & 1) * 2 * UBLK);
#pragma unroll
          for (int kb = 0; kb < 2; ++kb)
#pragma unroll
            for (int ks = 0; ks < 4; ++ks)
              umma2_ss_e(tbase + 128 * i + 64, dQ + off((2 * i + kb) * BLK + ks * 32), dUc + off(kb * UBLK + ks * 32),
                         idQU, (kb | ks) != 0, e);
          umma2_commit_both_e(bar(B_QUMMA + i), e);
          if (!wait_all(B_QU + i, qph[i])) return false;  // moved into the shared A operand
          qph[i] ^= 1;
        }
        tc_fence_after();
        const uint32_t tS = tbase + 128 * i;
#pragma unroll
        for (int kb = 0; kb < 2; ++kb)
#pragma unroll
          for (int ks = 0; ks < 4; ++ks)
            umma2_ss_e(tS, dQ + off((2 * i + kb) * BLK + ks * 32), dK + off((2 * st + kb) * HBLK + ks * 32), idS,
                       (kb | ks) != 0, e);
        if (sc.U.psac)
          for (int ks = 0; ks < rpad / 16; ++ks)
            umma2_ss_e(tS, dQU + off(i * rpad * 2 + ks * 32), dC + off(st * rpad * 2 + ks * 32), idS, 1u, e);
        umma2_commit_both_e(bar(B_SFULL + i), e);
        if (i == nqt - 1) {
          umma2_commit_both_e(bar(B_KEMPTY + st), e);
          sc.next(a, S, h);
          ++sjt;
        }
        return true;
      };
      if (total > 0) ok = issue_S(0) && (nqt == 1 || issue_S(1));
      for (int jt = 0; jt < total && ok; ++jt) {
        const int st = jt & 1;
        const uint32_t ph = (jt >> 1) & 1;
        if (!(ok = wait_all(B_VFULL + st, ph))) break;
#pragma unroll
        for (int i = 0; i < nqt; ++i) {
          if (!(ok = wait_all(B_PFULL + i, jt & 1))) break;
          tc_fence_after();
          const uint32_t tP = tbase + 128 * i, tO = tbase + 256 + 128 * i;
#pragma unroll
          for (int ks = 0; ks < 8; ++ks)
            umma2_ts_e(tO, tP + 8 * ks, dV + off(st * BLK + ks * 2048), idPV, (jt > 0 || ks > 0) ? 1u : 0u, e);
          if (i == nqt - 1) umma2_commit_both_e(bar(B_VEMPTY + st), e);
          if (jt + 1 < total && !(ok = issue_S(i))) break;
        }
      }
      umma2_commit_both_e(bar(B_OFINAL), e);
      if (!ok) {
        // a wait ran out: let the MMAs already issued finish before the
        // pair's TMEM is released
        mbar_wait(bar(B_OFINAL), 0, a.wait_ns);
        *s_err = 1;
      }
    } else if (rank == 1) {
      // ---------------------------------------------------------- hand-off relays (follower)
      // Warp 16 forwards the K stages and warp 17 the V stages: having
      // acquired the four rebuild warps' CTA-scope arrivals, one lane
      // arrives on the leader's barrier with a cluster-scope release, which
      // covers their shared-memory writes and waits for every memory access
      // the SM has in flight (hundreds to a thousand cycles) in this warp
      // instead of in the rebuild warps.
      const bool kside = warp == W_MMA;
      TileCursor c;
      c.init(a, S, h, cu0, (!kside && a.idle_role == QWM_ROLE_V_REBUILD) ? cu0 : cu1);
      bool ok = true;
      for (uint32_t jt = 0; c.valid() && ok; ++jt, c.next(a, S, h)) {
        const int st = jt & 1;
        ok = __all_sync(0xFFFFFFFFu, mbar_wait(bar((kside ? B_KRDY : B_VRDY) + st), (jt >> 1) & 1, a.wait_ns));
        if (ok && lane == 0) mbar_arrive_cluster(mapa(bar((kside ? B_KFULL : B_VFULL) + st), 0));
      }
      if (!ok) *s_err = 1;
    }
    __syncwarp();
  }

  tc_fence_before();
  __syncthreads();
  if (tid == 0 && *s_err) atomicCAS(a.status, 0, (int)QWM_ERR_TIMEOUT);
  if (tid == 0 && *s_bad) atomicCAS(a.status, 0, (int)QWM_ERR_NONFINITE);
  cluster_sync();  // neither CTA frees the pair's TMEM while the other still reads it
  if (warp == W_MMA) {
    tc_fence_after();
    tmem_dealloc2(tbase, 512);
  }
}


// The parts of a tail unit combined (the usual rescaling of partial softmax
// results: m = max_p m_p, l = sum_p l_p 2^((m_p - m) c), O = sum_p O_p
// 2^((m_p - m) c) / l with c = sm_scale log2(e)); a warp per query row, four
// channels per lane.
__global__ void __launch_bounds__(256) attend_combine(const AttendArgs a) {
  const int64_t gw = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;  // (tail unit, row)
  const int lane = threadIdx.x & 31;
  const int ntail = (a.n_units - a.n_whole);
  if (gw >= (int64_t)ntail * 512) return;
  const int tu = (int)(gw >> 9), prow = (int)(gw & 511);
  const int unit = a.n_whole + tu;
  const int h = unit / a.bph;
  const int64_t qi = (int64_t)(unit - h * a.bph) * 512 + prow;
  if (qi >= a.Nq) return;
  const float c = a.sm_scale * 1.4426950408889634f;
  float m = -INFINITY;
  for (int p = 0; p < a.nparts; ++p) m = fmaxf(m, a.part_ml[((size_t)(tu * a.nparts + p) * 512 + prow) * 2]);
  float l = 0.0f;
  float4 o = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
  for (int p = 0; p < a.nparts; ++p) {
    const size_t pr = (size_t)(tu * a.nparts + p) * 512 + prow;
    const float2 ml = *reinterpret_cast<const float2*>(a.part_ml + pr * 2);
    const float wgt = exp2f((ml.x - m) * c);
    l = fmaf(ml.y, wgt, l);
    const float4 v = *reinterpret_cast<const float4*>(a.part_o + pr * 128 + 4 * lane);
    o.x = fmaf(v.x, wgt, o.x); o.y = fmaf(v.y, wgt, o.y); o.z = fmaf(v.z, wgt, o.z); o.w = fmaf(v.w, wgt, o.w);
  }
  const float inv_l = 1.0f / l;
  uint2* dst = reinterpret_cast<uint2*>(a.out + ((size_t)qi * a.L.H + h) * 128 + 4 * lane);
  *dst = make_uint2(pack_bf16(o.x * inv_l, o.y * inv_l), pack_bf16(o.z * inv_l, o.w * inv_l));
  if (a.lse && lane == 0) a.lse[(size_t)h * a.Nq + qi] = m * a.sm_scale + logf(l);
}

}  // namespace

AttendPlan plan_attend(int64_t Nq, int H, int n_key_units, int nsm, bool split) {
  AttendPlan pl{};
  pl.bph = (int)((Nq + 511) / 512);
  pl.n_units = pl.bph * H;
  pl.n_whole = pl.n_units;
  pl.nparts = 1;
  const int slots = nsm / 2 > 0 ? nsm / 2 : 1;
  if (!split || n_key_units < 2 || pl.n_units % slots == 0) return pl;
  // whole units: full waves of the pair slots, rounded down to whole heads
  const int whole = pl.n_units / slots * slots / pl.bph * pl.bph, tail = pl.n_units - whole;
  // parts per tail unit: the fewest rounds of the tail over the pair slots
  // times the largest part (in key units), each part charged a fixed 0.15 of
  // a key unit; ties to fewer parts
  int best = 1;
  double best_cost = (double)n_key_units + 0.15;
  for (int s = 2; s <= n_key_units; ++s) {
    const int rounds = (tail * s + slots - 1) / slots;
    const int largest = (n_key_units + s - 1) / s;
    const double cost = rounds * (largest + 0.15);
    if (cost < best_cost - 1e-9) { best_cost = cost; best = s; }
  }
  if (best > 1) {
    pl.n_whole = whole;
    pl.nparts = best;
  }
  return pl;
}

size_t attend_workspace_bytes(const AttendPlan& pl) {
  if (pl.nparts <= 1) return 0;
  return (size_t)(pl.n_units - pl.n_whole) * pl.nparts * 512 * (128 + 2) * sizeof(float);
}

cudaError_t launch_attend(const AttendArgs& a, const AttendSlots& slots, cudaStream_t st) {
  auto whole = a.L.sf ? attend_kernel<1, false> : attend_kernel<0, false>;
  auto parts = a.L.sf ? attend_kernel<1, true> : attend_kernel<0, true>;
  cudaError_t e = cudaFuncSetAttribute(whole, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES);
  if (e == cudaSuccess) e = cudaFuncSetAttribute(parts, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES);
  if (e != cudaSuccess) return e;
  // the whole units are whole heads (n_whole a multiple of bph): a CTA pair
  // per block of 512 queries of each of those heads
  if (a.n_whole > 0) {
    whole<<<dim3((unsigned)(2 * a.bph), (unsigned)(a.n_whole / a.bph)), NT, SMEM_BYTES, st>>>(a, slots);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  if (a.n_units == a.n_whole) return cudaSuccess;
  const int64_t pairs = (int64_t)(a.n_units - a.n_whole) * a.nparts;
  parts<<<dim3((unsigned)(2 * pairs)), NT, SMEM_BYTES, st>>>(a, slots);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const int64_t warps = (int64_t)(a.n_units - a.n_whole) * 512;
  attend_combine<<<(unsigned)((warps * 32 + 255) / 256), 256, 0, st>>>(a);
  return cudaGetLastError();
}

}  // namespace qwm
