// qwm_internal.cuh -- shared definitions of the CUDA library: cache layout,
// kernel parameter blocks, launch entry points and sm_103a PTX helpers
// (tcgen05, mbarrier, bulk copies).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <stdint.h>

#include "../../include/qwm.h"

namespace qwm {

constexpr int kHeadDim = 128;
constexpr int kTile = 128;        // tokens per cache tile, queries per attend CTA
constexpr int kMaxSlots = 256;    // chunk slots per cache
constexpr int kHeaderBytes = 256;
constexpr int kSlotMetaBytes = 256;

__host__ __device__ inline int64_t round_up(int64_t x, int64_t a) { return (x + a - 1) / a * a; }

// Byte layout of the packed cache (see qwm_layout in qwm.h).
struct Layout {
  int H, d, C, G, r, ng, zb;
  int sf;                // scale format: 0 binary16 scales, 1 uint8 codes + binary16 secondary scale
  int64_t T;             // token capacity of a slot
  int32_t max_chunks;
  int64_t tiles;         // tiles per slot
  int64_t k_codes, k_scales, k_ids, k_zeros, k_coef, k_sigma, k_bytes;
  int64_t v_codes, v_scales, v_ids, v_zeros, v_bytes;  // from the tile start
  int64_t k_s2, v_s2;    // scale format 1: secondary scales [128] binary16
  int64_t tile_bytes;
  int64_t ktab, vtab, ut, pmask, tiles_off, head_bytes;  // pmask: [tiles][16 B] PSAC keep masks (r > 0)
  int64_t slot_bytes;
  int64_t total_bytes;
};

inline Layout make_layout(const qwm_config& c, int64_t T, int32_t max_chunks) {
  Layout L{};
  L.H = c.num_heads; L.d = c.head_dim; L.C = c.num_centroids; L.G = c.group_size; L.r = c.psac_rank;
  L.sf = c.scale_format;
  L.ng = L.d / L.G;
  L.zb = (2 * L.ng + 7) / 8;
  L.T = T; L.max_chunks = max_chunks;
  L.tiles = (T + kTile - 1) / kTile;
  int64_t o = 0;
  L.k_codes = o;  o += (int64_t)kTile * (L.d / 4);
  L.k_scales = o; o += round_up((int64_t)kTile * L.ng * (L.sf ? 1 : 2), 16);
  L.k_s2 = L.sf ? o : 0; o += L.sf ? kTile * 2 : 0;
  L.k_ids = o;    o += kTile;
  L.k_zeros = o;  o += round_up((int64_t)kTile * L.zb, 16);
  L.k_coef = o;   o += (int64_t)kTile * L.r;
  L.k_sigma = o;  o += L.r > 0 ? kTile * 2 : 0;
  L.k_bytes = round_up(o, 128);
  o = L.k_bytes;
  L.v_codes = o;  o += (int64_t)kTile * (L.d / 4);
  L.v_scales = o; o += round_up((int64_t)kTile * L.ng * (L.sf ? 1 : 2), 16);
  L.v_s2 = L.sf ? o : 0; o += L.sf ? kTile * 2 : 0;
  L.v_ids = o;    o += kTile;
  L.v_zeros = o;  o += round_up((int64_t)kTile * L.zb, 16);
  L.v_bytes = round_up(o, 128) - L.k_bytes;
  L.tile_bytes = L.k_bytes + L.v_bytes;
  o = 0;
  L.ktab = o;      o += (int64_t)L.C * L.d * 2;
  L.vtab = o;      o += (int64_t)L.C * L.d * 2;
  L.ut = o;        o += (int64_t)L.r * L.d * 2;
  L.pmask = o;     o += L.r > 0 ? L.tiles * 16 : 0;
  o = round_up(o, 1024);
  L.tiles_off = o; o += L.tiles * L.tile_bytes;
  L.head_bytes = round_up(o, 1024);
  L.slot_bytes = kSlotMetaBytes + (int64_t)L.H * L.head_bytes;
  L.total_bytes = kHeaderBytes + (int64_t)max_chunks * L.slot_bytes;
  return L;
}

// Entry of row `row` (0..127) of a tile in its PSAC code and scale arrays, or
// -1 when the tile's keep mask (4 little-endian words) does not name the row:
// the entry is the number of mask bits below the row (App. D.1 dense/sparse
// layouts; a dense tile names every row, so the entry is the row).
__device__ __forceinline__ int psac_entry(uint4 m, int row) {
  const int wi = row >> 5, bi = row & 31;
  const uint32_t w = wi == 0 ? m.x : (wi == 1 ? m.y : (wi == 2 ? m.z : m.w));
  if (!((w >> bi) & 1u)) return -1;
  return __popc(w & ((1u << bi) - 1u)) + (wi > 0 ? __popc(m.x) : 0) + (wi > 1 ? __popc(m.y) : 0) +
         (wi > 2 ? __popc(m.z) : 0);
}

__host__ __device__ inline int64_t head_offset(const Layout& L, int slot, int h) {
  return kHeaderBytes + (int64_t)slot * L.slot_bytes + kSlotMetaBytes + (int64_t)h * L.head_bytes;
}

// The configurations the library accepts (head_dim 128, group size 32 or 64,
// 1..256 centroids, PSAC rank 0/8/16/32, 1..4096 heads); qwm_api.cu.
bool config_supported(const qwm_config* c);

// ----------------------------------------------------------------------------
// TMA tensor maps (host, qwm_api.cu).
// Tokens x[N][H][128] (bf16): boxes of 64 channels x 1 head x box_rows tokens,
// 128-byte swizzle; rows past N read as zeros.
bool make_token_map(CUtensorMap* m, const void* x, int64_t N, int H, int box_rows);
// The cache buffer as rows of 256 bytes (128 binary16 values): boxes of 64
// values x 1 row, 128-byte swizzle, for tile::gather4 loads of centroid rows.
bool make_row_map(CUtensorMap* m, const void* base, int64_t rows);
// Centroid tables tab[H][C][128] (bf16): boxes of 64 channels x box_rows
// centroids x 1 head, 128-byte swizzle; rows past C read as zeros.
bool make_table_map(CUtensorMap* m, const void* tab, int C, int H, int box_rows);

// ----------------------------------------------------------------------------
// Kernel launch entry points (defined in the .cu files).
// ----------------------------------------------------------------------------
struct AppendArgs {
  Layout L;
  uint8_t* base;               // cache buffer
  int slot;
  int64_t N;
  const __nv_bfloat16* k;      // [N][H][d]
  const __nv_bfloat16* v;
  const __nv_bfloat16* kc;     // [H][C][d]
  const __nv_bfloat16* vc;
  const float* w;              // [H][d] or null
  const __nv_bfloat16* U;      // [H][d][r] or null
  int M;                       // candidates (clamped to C)
  const float* Mq;             // [H][d][d] fp32: Keys' candidates by the full quadratic form, or null
};
cudaError_t launch_append(const AppendArgs& a, cudaStream_t s);
cudaError_t launch_append_generic(const AppendArgs& a, cudaStream_t s);
cudaError_t launch_append_fused(const AppendArgs& a, cudaStream_t s);
cudaError_t launch_full_rescore(const AppendArgs& a, cudaStream_t s);

// The candidate filter's per-token record, parked in the token's 32 code
// bytes of the destination slot until the quantize kernel reads it: byte 0 =
// n, bytes 1.. = centroid ids.  n = M: the decided top-M; M <= n <= kBand:
// the band to rescore exactly; kRecAll: rescore every centroid.
constexpr int kMaxFilterM = 8;
constexpr int kBand = 16;
constexpr int kRecAll = 255;

struct AttendSlots {
  int32_t n;
  int32_t slot[kMaxSlots];
  int32_t tokens[kMaxSlots];
  int32_t psac[kMaxSlots];     // chunk stored with a PSAC correction
};
struct AttendArgs {
  Layout L;
  const uint8_t* base;
  int32_t* status;             // device status word
  const __nv_bfloat16* q;      // [Nq][H][d]
  const __nv_bfloat16* kcur;   // [Ncur][H][d]
  const __nv_bfloat16* vcur;
  int64_t Nq, Ncur;
  float sm_scale;
  __nv_bfloat16* out;          // [Nq][H][d]
  float* lse;                  // [H][Nq] or null
  uint64_t wait_ns;            // limit of every bounded wait
  int32_t idle_role;           // QWM_ROLE_*: a role that publishes nothing (test hook), 0 = none
  // work units (CTA pairs of 512 queries of one head) and their split: units
  // [0, n_whole) run over every key; each later unit runs as nparts parts over
  // contiguous ranges of the key units, combined by a second kernel from the
  // parts' unnormalised O rows and running (max, sum) in part_o / part_ml
  int32_t bph, n_units, n_whole, nparts;
  float* part_o;               // [tail units][nparts][512][128] fp32
  float* part_ml;              // [tail units][nparts][512][2] fp32
};
struct AttendPlan {
  int32_t bph, n_units, n_whole, nparts;
};
// The split of a launch: whole units in full waves of the SMs' CTA pairs, the
// remaining units in parts over the key units (split = false: no parts).
AttendPlan plan_attend(int64_t Nq, int H, int n_key_units, int nsm, bool split);
size_t attend_workspace_bytes(const AttendPlan& pl);
cudaError_t launch_attend(const AttendArgs& a, const AttendSlots& slots, cudaStream_t s);

struct FitArgs {
  int H, d, C, iters, Npad;    // Npad: C rounded up to a multiple of 16 (MMA width)
  int64_t N;
  const __nv_bfloat16* x;      // [N][H][d]
  __nv_bfloat16* out;          // [H][C][d]
  // workspace (FitWorkspace carves it)
  int32_t* status;             // device status word (a bounded wait that ran out)
  float* cent;                 // [H][C][d] fp32 centroids
  uint8_t* img;                // [H][2][Npad * 256] bf16 MMA operand images: hi, lo
  float* nrm;                  // [H][Npad] squared centroid norms
  uint32_t* nmax;              // [H] largest squared norm (fp32 bits)
  int32_t* emax;               // [H] largest bf16 exponent field of the head's tokens
  float* xn2;                  // [H][N] |x|^2 of every token (fp32, any order)
  int room;                    // fixed-point headroom bits of the exact member sums
  int32_t* counts;             // [H][C] members per cluster
  int32_t* offs;               // [H][C] first member slot
  uint8_t* asg;                // [H][N] assignment
  int32_t* list;               // [H][N] member token indices grouped by cluster
};
struct DequantArgs {
  Layout L;
  const uint8_t* base;         // cache buffer
  int slot;
  int64_t N;                   // tokens in the chunk
  int psac;                    // chunk stored with a PSAC correction
  float* k_out;                // [N][H][d] fp32 or null
  float* v_out;
};
cudaError_t launch_dequant(const DequantArgs& a, cudaStream_t s);

// Byte size of the k-means workspace for H heads of N tokens and C centroids
// (head_dim 128), and the carving of a workspace into FitArgs.
size_t fit_workspace_bytes(int H, int d, int C, int64_t N);
void fit_carve(FitArgs& a, uint8_t* ws);
cudaError_t launch_fit(const FitArgs& a, cudaStream_t s);

}  // namespace qwm
