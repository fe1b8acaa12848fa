// qwm_api.cu -- host side of the C ABI declared in include/qwm.h: argument
// validation, the cache descriptor (slot ring bookkeeping) and kernel launch.
#include <cstdlib>
#include <cstring>
#include <new>

#include <cudaTypedefs.h>

#include "qwm_internal.cuh"

namespace qwm {
namespace {
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q{};
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) !=
            cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      return (PFN_cuTensorMapEncodeTiled_v12000) nullptr;
    return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }();
  return fn;
}
}  // namespace

bool make_token_map(CUtensorMap* m, const void* x, int64_t N, int H, int box_rows) {
  PFN_cuTensorMapEncodeTiled_v12000 fn = encode_fn();
  if (!fn || N < 1) return false;
  cuuint64_t dims[3] = {128, (cuuint64_t)H, (cuuint64_t)N};
  cuuint64_t strides[2] = {256, (cuuint64_t)H * 256};
  cuuint32_t box[3] = {64, 1, (cuuint32_t)box_rows};
  cuuint32_t es[3] = {1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(x), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool make_table_map(CUtensorMap* m, const void* tab, int C, int H, int box_rows) {
  PFN_cuTensorMapEncodeTiled_v12000 fn = encode_fn();
  if (!fn || C < 1 || H < 1 || box_rows < 1 || box_rows > 256) return false;
  cuuint64_t dims[3] = {128, (cuuint64_t)C, (cuuint64_t)H};
  cuuint64_t strides[2] = {256, (cuuint64_t)C * 256};
  cuuint32_t box[3] = {64, (cuuint32_t)box_rows, 1};
  cuuint32_t es[3] = {1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(tab), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool make_row_map(CUtensorMap* m, const void* base, int64_t rows) {
  PFN_cuTensorMapEncodeTiled_v12000 fn = encode_fn();
  if (!fn || rows < 1) return false;
  cuuint64_t dims[2] = {128, (cuuint64_t)rows};
  cuuint64_t strides[1] = {256};
  cuuint32_t box[2] = {64, 1};
  cuuint32_t es[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void*>(base), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}
}  // namespace qwm

using qwm::Layout;

struct qwm_cache {
  qwm_config cfg;
  Layout L;
  uint8_t* base;
  size_t bytes;
  int32_t sliding_window;
  int64_t appended;                       // chunks appended so far
  int32_t n_tokens[qwm::kMaxSlots];       // tokens held by each slot
  int32_t psac[qwm::kMaxSlots];           // slot stored with a PSAC correction
  uint64_t wait_ns;                       // limit of the kernels' bounded waits
  int32_t idle_role;                      // qwm_cache_set_idle_role (0: none)
};

namespace {

bool supported(const qwm_config* c) { return qwm::config_supported(c); }

}  // namespace

bool qwm::config_supported(const qwm_config* c) {
  if (c->num_heads < 1 || c->num_heads > 4096) return false;
  if (c->head_dim != qwm::kHeadDim) return false;
  if (c->group_size != 32 && c->group_size != 64) return false;
  if (c->num_centroids < 1 || c->num_centroids > 256) return false;
  if (c->psac_rank != 0 && c->psac_rank != 8 && c->psac_rank != 16 && c->psac_rank != 32) return false;
  if (c->num_candidates < 1 || c->kmeans_iters < 0) return false;
  if (c->scale_format != 0 && c->scale_format != 1) return false;
  return true;
}

namespace {

bool same_shape(const qwm_config* a, const qwm_config* b) {
  return a->num_heads == b->num_heads && a->head_dim == b->head_dim && a->num_centroids == b->num_centroids &&
         a->group_size == b->group_size && a->psac_rank == b->psac_rank && a->scale_format == b->scale_format;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace

extern "C" {

const char* qwm_status_string(qwm_status s) {
  switch (s) {
    case QWM_OK: return "ok";
    case QWM_ERR_INVALID_ARG: return "invalid argument";
    case QWM_ERR_UNSUPPORTED: return "unsupported configuration";
    case QWM_ERR_CAPACITY: return "cache capacity exceeded";
    case QWM_ERR_CUDA: return "CUDA error";
    case QWM_ERR_TIMEOUT: return "device wait timed out";
    case QWM_ERR_NONFINITE: return "non-finite input";
  }
  return "unknown status";
}

size_t qwm_cache_bytes(const qwm_config* cfg, int64_t tokens_per_chunk, int32_t max_chunks) {
  if (!cfg || !supported(cfg) || tokens_per_chunk < 1 || max_chunks < 1 || max_chunks > qwm::kMaxSlots) return 0;
  return (size_t)qwm::make_layout(*cfg, tokens_per_chunk, max_chunks).total_bytes;
}

qwm_status qwm_cache_init(qwm_cache** out, const qwm_config* cfg, void* dev_buf, size_t bytes,
                          int64_t tokens_per_chunk, int32_t max_chunks, int32_t sliding_window, void* stream) {
  if (!out || !cfg || !dev_buf) return QWM_ERR_INVALID_ARG;
  *out = nullptr;
  if (!supported(cfg)) return QWM_ERR_UNSUPPORTED;
  if (tokens_per_chunk < 1 || max_chunks < 1 || max_chunks > qwm::kMaxSlots) return QWM_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(dev_buf) & 255u) != 0) return QWM_ERR_INVALID_ARG;
  Layout L = qwm::make_layout(*cfg, tokens_per_chunk, max_chunks);
  if (bytes < (size_t)L.total_bytes) return QWM_ERR_CAPACITY;
  qwm_cache* c = new (std::nothrow) qwm_cache();
  if (!c) return QWM_ERR_INVALID_ARG;
  c->cfg = *cfg;
  c->L = L;
  c->base = static_cast<uint8_t*>(dev_buf);
  c->bytes = bytes;
  c->sliding_window = sliding_window;
  c->appended = 0;
  c->wait_ns = 2000000000ull;
  c->idle_role = 0;
  if (cudaMemsetAsync(dev_buf, 0, qwm::kHeaderBytes, static_cast<cudaStream_t>(stream)) != cudaSuccess) {
    delete c;
    return QWM_ERR_CUDA;
  }
  *out = c;
  return QWM_OK;
}

void qwm_cache_free(qwm_cache* cache) { delete cache; }

int32_t qwm_cache_num_chunks(const qwm_cache* c) {
  if (!c) return 0;
  return (int32_t)(c->appended < c->L.max_chunks ? c->appended : c->L.max_chunks);
}

qwm_status qwm_cache_chunk_info(const qwm_cache* c, int32_t i, int32_t* slot, int64_t* tokens) {
  if (!c || !slot || !tokens) return QWM_ERR_INVALID_ARG;
  int32_t n = qwm_cache_num_chunks(c);
  if (i < 0 || i >= n) return QWM_ERR_INVALID_ARG;
  int64_t chunk = c->appended - n + i;  // oldest held chunk first
  int32_t s = (int32_t)(chunk % c->L.max_chunks);
  *slot = s;
  *tokens = c->n_tokens[s];
  return QWM_OK;
}

qwm_status qwm_dequant_chunk(const qwm_config* cfg, const qwm_cache* c, int32_t i, float* k_out, float* v_out,
                             void* stream) {
  if (!cfg || !c) return QWM_ERR_INVALID_ARG;
  if (!supported(cfg)) return QWM_ERR_UNSUPPORTED;
  if (!same_shape(cfg, &c->cfg)) return QWM_ERR_INVALID_ARG;
  if ((k_out && !aligned16(k_out)) || (v_out && !aligned16(v_out))) return QWM_ERR_INVALID_ARG;
  int32_t slot = 0;
  int64_t tokens = 0;
  const qwm_status st = qwm_cache_chunk_info(c, i, &slot, &tokens);
  if (st != QWM_OK) return st;
  if (!k_out && !v_out) return QWM_OK;
  qwm::DequantArgs a{};
  a.L = c->L;
  a.base = c->base;
  a.slot = slot;
  a.N = tokens;
  a.psac = c->psac[slot];
  a.k_out = k_out;
  a.v_out = v_out;
  return qwm::launch_dequant(a, static_cast<cudaStream_t>(stream)) == cudaSuccess ? QWM_OK : QWM_ERR_CUDA;
}

qwm_status qwm_cache_layout(const qwm_cache* c, qwm_layout* o) {
  if (!c || !o) return QWM_ERR_INVALID_ARG;
  const Layout& L = c->L;
  o->header_bytes = qwm::kHeaderBytes;
  o->slot_meta_bytes = qwm::kSlotMetaBytes;
  o->slot_bytes = L.slot_bytes;
  o->head_bytes = L.head_bytes;
  o->ktab_offset = L.ktab;
  o->vtab_offset = L.vtab;
  o->ut_offset = L.ut;
  o->tiles_offset = L.tiles_off;
  o->tile_tokens = qwm::kTile;
  o->tiles_per_chunk = L.tiles;
  o->tile_bytes = L.tile_bytes;
  o->k_codes = L.k_codes; o->k_scales = L.k_scales; o->k_ids = L.k_ids; o->k_zeros = L.k_zeros;
  o->k_coef = L.k_coef; o->k_sigma = L.k_sigma; o->k_bytes = L.k_bytes;
  o->v_codes = L.v_codes; o->v_scales = L.v_scales; o->v_ids = L.v_ids; o->v_zeros = L.v_zeros;
  o->v_bytes = L.v_bytes;
  o->zero_bytes = L.zb;
  o->k_s2 = L.k_s2;
  o->v_s2 = L.v_s2;
  o->pmask_offset = L.pmask;
  return QWM_OK;
}

qwm_status qwm_cache_status(qwm_cache* c, int32_t* status, void* stream) {
  if (!c || !status) return QWM_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int32_t v = 0;
  if (cudaMemcpyAsync(&v, c->base, sizeof v, cudaMemcpyDeviceToHost, s) != cudaSuccess) return QWM_ERR_CUDA;
  if (cudaStreamSynchronize(s) != cudaSuccess) return QWM_ERR_CUDA;
  if (v != 0 && cudaMemsetAsync(c->base, 0, sizeof v, s) != cudaSuccess) return QWM_ERR_CUDA;
  *status = v;
  return QWM_OK;
}

size_t qwm_fit_workspace_bytes(const qwm_config* cfg, int64_t N) {
  if (!cfg || !supported(cfg) || N < 1) return 0;
  return qwm::fit_workspace_bytes(cfg->num_heads, cfg->head_dim, cfg->num_centroids, N);
}

qwm_status qwm_fit_centroids(const qwm_config* cfg, const void* x, int64_t N, void* centroids, void* workspace,
                             size_t workspace_bytes, void* stream) {
  if (!cfg || !x || !centroids || !workspace || N < 1) return QWM_ERR_INVALID_ARG;
  if (!supported(cfg)) return QWM_ERR_UNSUPPORTED;
  if (N > (int64_t)1 << 31) return QWM_ERR_UNSUPPORTED;
  if (!aligned16(x) || !aligned16(centroids) || (reinterpret_cast<uintptr_t>(workspace) & 255u))
    return QWM_ERR_INVALID_ARG;
  if (workspace_bytes < qwm_fit_workspace_bytes(cfg, N)) return QWM_ERR_CAPACITY;
  qwm::FitArgs a{};
  a.H = cfg->num_heads; a.d = cfg->head_dim; a.C = cfg->num_centroids; a.iters = cfg->kmeans_iters;
  a.N = N;
  a.x = static_cast<const __nv_bfloat16*>(x);
  a.out = static_cast<__nv_bfloat16*>(centroids);
  qwm::fit_carve(a, static_cast<uint8_t*>(workspace));
  return qwm::launch_fit(a, static_cast<cudaStream_t>(stream)) == cudaSuccess ? QWM_OK : QWM_ERR_CUDA;
}

namespace {

qwm_status quantize_append(const qwm_config* cfg, qwm_cache* c, const void* k, const void* v, int64_t N,
                           const void* k_centroids, const void* v_centroids, const float* w, const void* U,
                           const float* Mq, void* stream) {
  if (!cfg || !c || !k || !v || !k_centroids || !v_centroids) return QWM_ERR_INVALID_ARG;
  if (!supported(cfg)) return QWM_ERR_UNSUPPORTED;
  if (!same_shape(cfg, &c->cfg)) return QWM_ERR_INVALID_ARG;
  if (N < 1) return QWM_ERR_INVALID_ARG;
  if (N > c->L.T) return QWM_ERR_CAPACITY;
  if (!aligned16(k) || !aligned16(v)) return QWM_ERR_INVALID_ARG;
  // the centroid rows are read as whole 32-byte sectors
  if ((reinterpret_cast<uintptr_t>(k_centroids) & 31u) || (reinterpret_cast<uintptr_t>(v_centroids) & 31u))
    return QWM_ERR_INVALID_ARG;
  if ((w && (reinterpret_cast<uintptr_t>(w) & 3u)) || (U && !aligned16(U))) return QWM_ERR_INVALID_ARG;
  if (c->appended >= c->L.max_chunks && !c->sliding_window) return QWM_ERR_CAPACITY;
  int slot = (int)(c->appended % c->L.max_chunks);
  qwm::AppendArgs a{};
  a.L = c->L;
  a.base = c->base;
  a.slot = slot;
  a.N = N;
  a.k = static_cast<const __nv_bfloat16*>(k);
  a.v = static_cast<const __nv_bfloat16*>(v);
  a.kc = static_cast<const __nv_bfloat16*>(k_centroids);
  a.vc = static_cast<const __nv_bfloat16*>(v_centroids);
  a.w = w;
  a.U = (cfg->psac_rank > 0) ? static_cast<const __nv_bfloat16*>(U) : nullptr;
  a.M = cfg->num_candidates < cfg->num_centroids ? cfg->num_candidates : cfg->num_centroids;
  a.Mq = Mq;
  if (qwm::launch_append(a, static_cast<cudaStream_t>(stream)) != cudaSuccess) return QWM_ERR_CUDA;
  c->n_tokens[slot] = (int32_t)N;
  c->psac[slot] = a.U != nullptr;
  c->appended += 1;
  return QWM_OK;
}

}  // namespace

qwm_status qwm_quantize_append(const qwm_config* cfg, qwm_cache* c, const void* k, const void* v, int64_t N,
                               const void* k_centroids, const void* v_centroids, const float* w, const void* U,
                               void* stream) {
  return quantize_append(cfg, c, k, v, N, k_centroids, v_centroids, w, U, nullptr, stream);
}

qwm_status qwm_quantize_append_full(const qwm_config* cfg, qwm_cache* c, const void* k, const void* v, int64_t N,
                                    const void* k_centroids, const void* v_centroids, const float* w, const void* U,
                                    const float* Mq, void* stream) {
  if (!Mq || !aligned16(Mq)) return QWM_ERR_INVALID_ARG;
  if (!cfg) return QWM_ERR_INVALID_ARG;
  // the exhaustive-distance kernel of 8 < M < C takes the diagonal form only
  if (cfg->num_candidates > 8 && cfg->num_candidates < cfg->num_centroids) return QWM_ERR_UNSUPPORTED;
  return quantize_append(cfg, c, k, v, N, k_centroids, v_centroids, w, U, Mq, stream);
}

namespace {

int device_sms() {
  int dev = 0, nsm = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return 0;
  return nsm;
}

qwm_status attend_impl(const qwm_config* cfg, const qwm_cache* c, const void* q, int64_t Nq, const void* k_cur,
                       const void* v_cur, int64_t N_cur, float sm_scale, void* out, float* lse, void* workspace,
                       size_t workspace_bytes, void* stream) {
  if (!cfg || !c || Nq < 0 || N_cur < 0) return QWM_ERR_INVALID_ARG;
  if (!supported(cfg)) return QWM_ERR_UNSUPPORTED;
  if (!same_shape(cfg, &c->cfg)) return QWM_ERR_INVALID_ARG;
  if (qwm_cache_num_chunks(c) == 0 && N_cur == 0) return QWM_ERR_INVALID_ARG;
  if (Nq == 0) return QWM_OK;
  if (!q || !out) return QWM_ERR_INVALID_ARG;
  if (N_cur > 0 && (!k_cur || !v_cur || !aligned16(k_cur) || !aligned16(v_cur))) return QWM_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(out)) return QWM_ERR_INVALID_ARG;
  if (workspace && (reinterpret_cast<uintptr_t>(workspace) & 255u)) return QWM_ERR_INVALID_ARG;
  if (!(sm_scale > 0.0f) || sm_scale > 3.0e38f) return QWM_ERR_INVALID_ARG;
  if (Nq > ((int64_t)1 << 31) || N_cur > ((int64_t)1 << 31)) return QWM_ERR_UNSUPPORTED;
  int32_t n = qwm_cache_num_chunks(c);
  qwm::AttendSlots slots{};
  slots.n = n;
  for (int32_t i = 0; i < n; ++i) {
    int64_t tok;
    int32_t s;
    qwm_cache_chunk_info(c, i, &s, &tok);
    slots.slot[i] = s;
    slots.tokens[i] = (int32_t)tok;
    slots.psac[i] = c->psac[s];
  }
  qwm::AttendArgs a{};
  a.L = c->L;
  a.base = c->base;
  a.status = reinterpret_cast<int32_t*>(c->base);
  a.q = static_cast<const __nv_bfloat16*>(q);
  a.kcur = static_cast<const __nv_bfloat16*>(k_cur);
  a.vcur = static_cast<const __nv_bfloat16*>(v_cur);
  a.Nq = Nq;
  a.Ncur = N_cur;
  a.sm_scale = sm_scale;
  a.out = static_cast<__nv_bfloat16*>(out);
  a.lse = lse;
  a.wait_ns = c->wait_ns;
  a.idle_role = c->idle_role;
  const int nsm = device_sms();
  if (nsm <= 0) return QWM_ERR_CUDA;
  qwm::AttendPlan pl = qwm::plan_attend(Nq, c->L.H, n + (N_cur > 0 ? 1 : 0), nsm, workspace != nullptr);
  const size_t need = qwm::attend_workspace_bytes(pl);
  if (need > 0 && workspace_bytes < need) pl = qwm::plan_attend(Nq, c->L.H, n + (N_cur > 0 ? 1 : 0), nsm, false);
  a.bph = pl.bph;
  a.n_units = pl.n_units;
  a.n_whole = pl.n_whole;
  a.nparts = pl.nparts;
  if (pl.nparts > 1) {
    a.part_o = static_cast<float*>(workspace);
    a.part_ml = a.part_o + (size_t)(pl.n_units - pl.n_whole) * pl.nparts * 512 * 128;
  }
  return qwm::launch_attend(a, slots, static_cast<cudaStream_t>(stream)) == cudaSuccess ? QWM_OK : QWM_ERR_CUDA;
}

}  // namespace

qwm_status qwm_attend(const qwm_config* cfg, const qwm_cache* c, const void* q, int64_t Nq, const void* k_cur,
                      const void* v_cur, int64_t N_cur, float sm_scale, void* out, float* lse, void* stream) {
  return attend_impl(cfg, c, q, Nq, k_cur, v_cur, N_cur, sm_scale, out, lse, nullptr, 0, stream);
}

size_t qwm_attend_workspace_bytes(const qwm_config* cfg, const qwm_cache* c, int64_t Nq, int64_t N_cur) {
  if (!cfg || !c || Nq < 1 || N_cur < 0 || !supported(cfg) || !same_shape(cfg, &c->cfg)) return 0;
  const int nsm = device_sms();
  if (nsm <= 0) return 0;
  const int n_key_units = qwm_cache_num_chunks(c) + (N_cur > 0 ? 1 : 0);
  return qwm::attend_workspace_bytes(qwm::plan_attend(Nq, c->L.H, n_key_units, nsm, true));
}

qwm_status qwm_attend_ws(const qwm_config* cfg, const qwm_cache* c, const void* q, int64_t Nq, const void* k_cur,
                         const void* v_cur, int64_t N_cur, float sm_scale, void* out, float* lse, void* workspace,
                         size_t workspace_bytes, void* stream) {
  return attend_impl(cfg, c, q, Nq, k_cur, v_cur, N_cur, sm_scale, out, lse, workspace, workspace_bytes, stream);
}

qwm_status qwm_cache_set_wait_limit(qwm_cache* c, uint64_t ns) {
  if (!c || ns < 1000ull || ns > 60000000000ull) return QWM_ERR_INVALID_ARG;
  c->wait_ns = ns;
  return QWM_OK;
}

qwm_status qwm_cache_set_idle_role(qwm_cache* c, int32_t role) {
  if (!c || (role != 0 && role != QWM_ROLE_V_REBUILD)) return QWM_ERR_INVALID_ARG;
  c->idle_role = role;
  return QWM_OK;
}

}  // extern "C"
