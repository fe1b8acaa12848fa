/*
 * qwm.h -- C ABI of the GB300-native QuantWM per-chunk 2-bit KV-cache path.
 *
 * QuantWM ("Temporally Consistent 2-Bit KV Cache Quantization for Video World
 * Models") stores each finished chunk of an autoregressive video model's KV
 * cache as centroid ids + INT2 residual codes (Sec. 2 Eq. 1-4), chosen by the
 * Query-sensitivity-aware QSAC rule (Sec. 4.1 Eq. 9-12), plus for Keys a
 * rank-r PSAC correction C = E U_r (Sec. 4.2 Eq. 13-17); attention then runs
 * over the packed history and the active bf16 chunk (App. D.1 "Cache
 * lifecycle").  This library implements both halves of that per-chunk path on
 * one GB300 GPU (sm_103a):
 *   qwm_fit_centroids    k-means centroids of a chunk (Sec. 2, QVG convention)
 *   qwm_quantize_append  QSAC assignment, INT2 residual quantization + packing,
 *                        PSAC coefficients, written into one chunk slot
 *   qwm_attend           softmax attention of new queries over the packed
 *                        chunks (with the PSAC logit term Q U_r C^T) and the
 *                        active bf16 chunk
 *   qwm_cache_bytes      size of the caller-owned cache buffer
 *
 * Conventions for every call:
 *   - Tensor pointers are DEVICE pointers owned by the caller; the library
 *     never allocates device memory.  bf16 tensors are token-major
 *     [tokens][heads][head_dim], contiguous, 16-byte aligned.
 *   - `stream` is a cudaStream_t (NULL = legacy default stream); every call is
 *     asynchronous on it, except qwm_cache_status, which synchronises it.
 *   - Host-detectable errors (bad arguments, unsupported shapes, capacity)
 *     are returned before anything is launched.  Errors detected on the GPU
 *     (a bounded wait that ran out; a value the binary16 operands cannot
 *     hold) are recorded in the cache's device status word, read with
 *     qwm_cache_status.
 *   - Supported: head_dim 128; group_size 32 or 64; 1 <= num_centroids <= 256;
 *     psac_rank 0, 8, 16 or 32; num_candidates >= 1 (values above
 *     num_centroids mean "all centroids"); scale_format 0 or 1.  Anything
 *     else returns QWM_ERR_UNSUPPORTED.
 */
#ifndef QWM_H
#define QWM_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define QWM_API __attribute__((visibility("default")))
#else
#define QWM_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

/* Problem statement: heads H, head_dim d, centroid count C, INT2 group size G,
 * PSAC rank r (Sec. 4.2; r = 0 disables PSAC), QSAC candidate count M
 * (App. C.5, default 4), Lloyd iterations of qwm_fit_centroids. */
typedef struct qwm_config {
  int32_t num_heads;
  int32_t head_dim;
  int32_t num_centroids;
  int32_t group_size;
  int32_t psac_rank;
  int32_t num_candidates;
  int32_t kmeans_iters;
  /* Storage of the INT2 group scales: 0 = one binary16 per group; 1 = App. D.1's
   * uint8 code per group with one binary16 secondary scale per token-head
   * (the group's scale is code * secondary).  Zero-initialise the struct. */
  int32_t scale_format;
} qwm_config;

typedef enum qwm_status {
  QWM_OK = 0,
  QWM_ERR_INVALID_ARG = 1, /* NULL pointer, negative size, mismatched config */
  QWM_ERR_UNSUPPORTED = 2, /* shape outside the supported set above */
  QWM_ERR_CAPACITY = 3,    /* chunk larger than a slot, or cache full without a window */
  QWM_ERR_CUDA = 4,        /* a CUDA runtime call failed */
  QWM_ERR_TIMEOUT = 5,     /* a bounded wait inside a kernel ran out (device status) */
  QWM_ERR_NONFINITE = 6    /* an input beyond the binary16 range or not a number (device status) */
} qwm_status;

/* Opaque host descriptor over a caller-owned device buffer. */
typedef struct qwm_cache qwm_cache;

/* Byte offsets of the packed cache, for readers of the buffer (tests, tools).
 * A slot holds one chunk: for head h, at slot_offset(s) + slot_meta_bytes +
 * h*head_bytes, come the Key centroid table [C][d] and the Value centroid
 * table [C][d], both binary16 (the chunk's bf16 tables converted exactly;
 * bf16 values outside the binary16 range are not representable there),
 * U_r^T [r][d] bf16, then tiles_per_chunk tiles of tile_tokens tokens.  Each
 * tile is a Key block followed by a Value block of structure-of-arrays fields
 * (offsets within the tile):
 *   codes [128][d/4] u8: the 2-bit codes of a token, 16 channels per
 *     little-endian 32-bit word; in word k (channels 16k..16k+15) the even
 *     channel 16k+2i sits at bits 2i and the odd channel 16k+2i+1 at bits
 *     16+2i (App. D.1 packs four codes per byte; this order is ours);
 *   scales [128][d/G] binary16; ids [128] u8;
 *   zero-points [128][zb] u8: group g in byte g/4, bits 2(g%4);
 *   Keys only: PSAC codes [128][r] int8 and row scales [128] binary16, in one
 *     of two layouts per tile (App. D.1 stores the smaller of a dense and a
 *     sparse coefficient layout): the tile's 16-byte keep mask at
 *     pmask_offset + 16 * tile (bit i of the little-endian 128-bit mask = row
 *     i) names the rows stored; row i's codes and scale are entry
 *     e = popcount(mask bits below i) of the two arrays.  Dense tiles set a
 *     bit for every token (rows whose correction was dropped hold zeros);
 *     sparse tiles set the kept rows only, so they take 16 + K (r + 2) bytes
 *     instead of n (r + 2), and are chosen when that is smaller.
 * With scale_format 1 the scale field holds [128][d/G] u8 codes and a
 * secondary scale field [128] binary16 follows it (k_s2, v_s2). */
typedef struct qwm_layout {
  int64_t header_bytes;     /* device status word + reserved, before slot 0 */
  int64_t slot_meta_bytes;  /* per-slot reserved bytes before head 0 */
  int64_t slot_bytes;       /* bytes per chunk slot */
  int64_t head_bytes;       /* bytes per head inside a slot */
  int64_t ktab_offset, vtab_offset, ut_offset, tiles_offset; /* within a head */
  int64_t tile_tokens, tiles_per_chunk, tile_bytes;
  int64_t k_codes, k_scales, k_ids, k_zeros, k_coef, k_sigma, k_bytes; /* within a tile */
  int64_t v_codes, v_scales, v_ids, v_zeros, v_bytes; /* within a tile, from its start */
  int64_t zero_bytes;       /* zb: bytes of packed zero-points per token */
  int64_t k_s2, v_s2;       /* scale_format 1: secondary scales [128] binary16 (k_scales, v_scales
                               then hold [128][d/G] uint8 codes); 0 otherwise */
  int64_t pmask_offset;     /* within a head: PSAC keep masks [tiles_per_chunk][16 B] (r > 0) */
} qwm_layout;

/* Human-readable name of a status code (static string). */
QWM_API const char* qwm_status_string(qwm_status status);

/* Bytes of device memory a cache of max_chunks slots of tokens_per_chunk
 * tokens needs (App. D.1 packed storage: per token-head d/4 code bytes, d/G
 * binary16 scales, one uint8 centroid id, 2-bit zero-points, for Keys r INT8
 * PSAC codes + one binary16 row scale; per chunk-head the two centroid
 * tables as binary16, U_r^T as bf16 and a 16-byte PSAC keep mask per tile).  Returns 0 for an invalid or
 * unsupported configuration. */
QWM_API size_t qwm_cache_bytes(const qwm_config* cfg, int64_t tokens_per_chunk, int32_t max_chunks);

/* Create a host descriptor over dev_buf (256-byte aligned, bytes >=
 * qwm_cache_bytes(...)), and
 * clear the buffer's header on `stream`.  max_chunks <= 256.  With
 * sliding_window != 0, appending to a full cache overwrites the oldest chunk
 * (slot = chunk index mod max_chunks); otherwise it returns QWM_ERR_CAPACITY.
 * The descriptor is freed with qwm_cache_free; the buffer stays the caller's. */
QWM_API qwm_status qwm_cache_init(qwm_cache** out, const qwm_config* cfg, void* dev_buf, size_t bytes,
                          int64_t tokens_per_chunk, int32_t max_chunks, int32_t sliding_window,
                          void* stream);
QWM_API void qwm_cache_free(qwm_cache* cache);

/* Number of chunks currently held; chunk i (0 = oldest) lives in *slot and
 * has *tokens tokens. */
QWM_API int32_t qwm_cache_num_chunks(const qwm_cache* cache);
QWM_API qwm_status qwm_cache_chunk_info(const qwm_cache* cache, int32_t i, int32_t* slot, int64_t* tokens);
QWM_API qwm_status qwm_cache_layout(const qwm_cache* cache, qwm_layout* out);

/* Synchronise `stream`, then read and clear the device status word: *status
 * receives QWM_OK or the first error a kernel recorded (QWM_ERR_TIMEOUT,
 * QWM_ERR_NONFINITE). */
QWM_API qwm_status qwm_cache_status(qwm_cache* cache, int32_t* status, void* stream);

/* Limit of every bounded wait inside the kernels that use this cache (an
 * mbarrier wait between the roles of a kernel); default 2 s.  A wait that
 * runs out makes its role leave its loop, the kernel finishes without further
 * work on the GPU, and QWM_ERR_TIMEOUT is recorded in the status word (the
 * outputs of that call are then incomplete).  1e3 <= ns <= 6e10, otherwise
 * QWM_ERR_INVALID_ARG.  Host-side setting; applies to the calls made after it. */
QWM_API qwm_status qwm_cache_set_wait_limit(qwm_cache* cache, uint64_t ns);

/* Test hook of the timeout path (no counterpart in the paper): with role
 * QWM_ROLE_V_REBUILD, the attention calls made afterwards leave the role that
 * rebuilds V_hat idle, so the MMA warp's bounded wait for its first tile runs
 * out (with a short qwm_cache_set_wait_limit, in milliseconds) and the call
 * records QWM_ERR_TIMEOUT instead of computing.  0 restores normal work; any
 * other role returns QWM_ERR_INVALID_ARG. */
#define QWM_ROLE_V_REBUILD 1
QWM_API qwm_status qwm_cache_set_idle_role(qwm_cache* cache, int32_t role);

/* Scratch bytes qwm_fit_centroids needs for N tokens; 0 for an invalid
 * configuration.  With P = C rounded up to a multiple of 16 (at least 16),
 * each part padded to 256 bytes: a 256-byte status word, fp32 centroids
 * H*C*d*4, bf16 operand images H*P*512, norms H*P*4, H*4, counts and offsets
 * 2*H*C*4, assignment H*N and member lists H*N*4. */
QWM_API size_t qwm_fit_workspace_bytes(const qwm_config* cfg, int64_t N);

/* k-means centroids of one chunk, per head (Sec. 2: centroid-residual form of
 * QVG, fitted with Lloyd's algorithm; App. D.1 keeps centroids in BF16).
 * x: bf16 [N][H][d] (N >= 1).  centroids (out): bf16 [H][C][d].
 * Initial centroid j is token floor(j*N/C); each of kmeans_iters iterations
 * assigns every token to its Euclidean-nearest centroid (ties to the lower
 * index) and replaces each non-empty cluster's centroid by its member mean;
 * the result is rounded to bf16.  The distance is the fp32 sum in channel
 * order of the rounded squares of the rounded differences, the mean the fp32
 * rounding of the fp64 mean: the tensor cores screen the centroids and every
 * decision is taken on these exact values.  workspace: device scratch of at
 * least qwm_fit_workspace_bytes(cfg, N) bytes, 256-byte aligned.  If a bounded
 * wait inside a kernel runs out, every output centroid is NaN. */
QWM_API qwm_status qwm_fit_centroids(const qwm_config* cfg, const void* x, int64_t N, void* centroids,
                             void* workspace, size_t workspace_bytes, void* stream);

/* Allocation-free qwm_fit_centroids (the paper has no counterpart: this is an
 * integration convenience).  For callers that cannot provide device scratch:
 * a plain C host program holding only the tensors it was given, or an engine
 * whose device memory is reserved by its own pool and which must not call
 * cudaMalloc/cudaFree mid-generation (they can synchronise the device).  The
 * k-means scratch lives in a static 16 MiB device array that every GPU which
 * loads the library keeps until process exit; calls needing more
 * (qwm_fit_workspace_bytes(cfg, N) above 16 MiB) return QWM_ERR_CAPACITY.  Same arguments and results as
 * qwm_fit_centroids without the workspace.  The first call on a device looks
 * up the array's device address on the current device, so make that first
 * call before any stream capture.  All calls share the one array: calls whose
 * work overlaps on the GPU (different streams, or several host threads) race
 * and give wrong centroids; serialise them. */
QWM_API qwm_status qwm_fit_centroids_noalloc(const qwm_config* cfg, const void* x, int64_t N, void* centroids,
                                             void* stream);

/* Quantize one finished chunk and append it to the cache (Sec. 4.1 QSAC,
 * Sec. 2 Eq. 1-4 INT2 residuals, Sec. 4.2 Eq. 13/16 PSAC, App. D.1 packing).
 * k, v: bf16 [N][H][d], 1 <= N <= tokens_per_chunk.  k_centroids,
 * v_centroids: bf16 [H][C][d], 32-byte aligned (this chunk's tables; copied
 * into the slot); a table that is only 16-byte aligned returns
 * QWM_ERR_INVALID_ARG.
 * w: fp32 [H][d] channel sensitivity weights (Eq. 8) or NULL for w = 1 (the
 * cold-start rule of App. C.3).  U: bf16 [H][d][r] principal Query basis
 * (Eq. 15) or NULL to store no PSAC correction (cold start).  Keys: top-M
 * candidates by the Query-aware distance (Eq. 9), then the lowest QSAC score
 * (Eq. 12), ties to the lower index; Values: the same with w = 1 and no PSAC.
 * The chunk goes to the next slot (oldest slot when a sliding window is full).
 * The slot holds binary16 tables and scales and attention uses binary16
 * operands: a Key, Value or centroid value of magnitude above 65504, or one
 * that is not a number, or a group whose rebuilt values mu + s (q - z) could
 * leave that range, records QWM_ERR_NONFINITE in the status word (the packed
 * records are still written as defined above; rows with such values skip the
 * tensor-core candidate filter and are decided on exact distances). */
QWM_API qwm_status qwm_quantize_append(const qwm_config* cfg, qwm_cache* cache, const void* k, const void* v,
                               int64_t N, const void* k_centroids, const void* v_centroids,
                               const float* w, const void* U, void* stream);

/* qwm_quantize_append with the Keys' top-M candidates chosen by the full
 * Query-aware quadratic form d_j = (k - mu_j)^T M (k - mu_j) instead of its
 * diagonal (Eq. 9): the ablation of App. C.4 (the QSAC score and everything
 * after still use w; Values unchanged).  Mq: fp32 [H][d][d] row-major, the
 * historical Query second moment of each head (Eq. 6) or any symmetric
 * matrix, 16-byte aligned.  As in the oracle, d_j is the fp32 evaluation
 * e = k - mu_j, t_c = sum_c' M_cc' e_c' and d = sum_c e_c t_c, one fused
 * multiply-add per term in index order; the tensor cores screen the
 * candidates (B operand M mu_j) and the undecided rows are rescored with it.
 * 8 < num_candidates < num_centroids returns QWM_ERR_UNSUPPORTED. */
QWM_API qwm_status qwm_quantize_append_full(const qwm_config* cfg, qwm_cache* cache, const void* k, const void* v,
                                            int64_t N, const void* k_centroids, const void* v_centroids,
                                            const float* w, const void* U, const float* Mq, void* stream);

/* Attention of Nq new queries over every cached chunk and the active chunk
 * (Sec. 3.3 Eq. 5 logits; Sec. 4.2 Eq. 17: Q K_hat^T = Q K_hat0^T +
 * (Q U_r) C^T with each chunk's own U_r; Values rebuilt without PSAC).
 * q: bf16 [Nq][H][d]; k_cur, v_cur: bf16 [N_cur][H][d] of the active chunk
 * (N_cur = 0 allowed, then they may be NULL).  No mask: cached chunks are in
 * the past.  sm_scale > 0 (usually 1/sqrt(d)).
 * out: bf16 [Nq][H][d] = softmax(sm_scale * logits) V.
 * lse: fp32 [H][Nq] natural-log sum-exp of the scaled logits, or NULL.
 * The tensor-core operands are binary16 with fp32 accumulation, so q, k_cur
 * and v_cur must lie within the binary16 range (|x| <= 65504): a finite value
 * beyond it saturates to +-65504 (the output stays finite) and a NaN
 * propagates; either records QWM_ERR_NONFINITE in the status word.  The
 * rebuilt cache values are in range for every chunk whose append did not
 * report QWM_ERR_NONFINITE.
 * At least one key (a cached chunk or N_cur > 0) is required. */
QWM_API qwm_status qwm_attend(const qwm_config* cfg, const qwm_cache* cache, const void* q, int64_t Nq,
                      const void* k_cur, const void* v_cur, int64_t N_cur, float sm_scale,
                      void* out, float* lse, void* stream);

/* Bytes of the scratch buffer that lets qwm_attend_ws balance a launch over
 * the GPU (0: the launch needs none), for Nq queries over the cache's current
 * chunks and N_cur active tokens on the current device; 0 for invalid
 * arguments.  Not part of the paper's method: the launch's CTA pairs work on
 * 512 queries of one head each, and when their count leaves the last wave of
 * the SMs partly idle, the work units of that wave are split along the keys
 * (whole chunks per part, cached chunks then the active chunk) and their
 * partial results combined -- the usual rescaling of partial softmax sums,
 * as for attention over several key blocks. */
QWM_API size_t qwm_attend_workspace_bytes(const qwm_config* cfg, const qwm_cache* cache, int64_t Nq, int64_t N_cur);

/* qwm_attend with a caller-owned device scratch buffer (256-byte aligned) of
 * at least qwm_attend_workspace_bytes bytes for the same arguments: the same
 * result within the attention tolerance (the parts of a split unit are
 * combined in fp32; the bf16 output and the lse may differ from
 * qwm_attend's in the last bits).  workspace = NULL, or a buffer too small,
 * runs qwm_attend.  Calls sharing a buffer must not overlap on the GPU. */
QWM_API qwm_status qwm_attend_ws(const qwm_config* cfg, const qwm_cache* cache, const void* q, int64_t Nq,
                                 const void* k_cur, const void* v_cur, int64_t N_cur, float sm_scale,
                                 void* out, float* lse, void* workspace, size_t workspace_bytes, void* stream);

/* ---------------------------------------------------------------------------
 * Historical Query statistics and the principal Query basis, kept on the GPU
 * (Sec. 4.1 Eq. 6 and 8, Sec. 4.2 Eq. 15; App. C.3 cold start; App. D.1: the
 * per-head statistics are updated incrementally, the basis is recomputed at
 * chunk boundaries, past Queries are not kept).  They produce the w and U
 * arguments of qwm_quantize_append without a host round trip.
 *
 * A statistics buffer is caller-owned device memory of
 * qwm_query_stats_bytes(cfg) bytes, 256-byte aligned:
 *   byte 0    int32 device status word (QWM_OK or the first kernel error)
 *   byte 8    uint64 Query count N_<t (tokens folded in so far)
 *   byte 16   int32 Jacobi sweeps of the last qwm_query_basis (maximum over heads)
 *   byte 256  fp32 sums S_h = sum over past Queries of q q^T, [H][d][d] row-major.
 * --------------------------------------------------------------------------- */

/* Size of a statistics buffer; 0 for an invalid configuration. */
QWM_API size_t qwm_query_stats_bytes(const qwm_config* cfg);

/* Zero a statistics buffer (no Query seen yet). */
QWM_API qwm_status qwm_query_stats_reset(const qwm_config* cfg, void* stats, void* stream);

/* Fold one chunk's Queries into the statistics (Eq. 6 numerator):
 * S_h += sum_n q[n,h] q[n,h]^T and count += N.  q: bf16 [N][H][d], 16-byte
 * aligned; N = 0 is a no-op.  Products are exact and accumulate in fp32 (tensor
 * cores); the same inputs always give the same bits. */
QWM_API qwm_status qwm_query_stats_update(const qwm_config* cfg, void* stats, const void* q, int64_t N,
                                          void* stream);

/* Channel weights and principal basis from the statistics, M_h = S_h / count.
 *   w: fp32 [H][d], w_c = M_cc / mean_c' M_c'c' (Eq. 8); 1 for every channel
 *      when count = 0 or the mean is 0 (App. C.3 cold start).
 *   U: bf16 [H][d][r], r = cfg->psac_rank (not written when r = 0): the
 *      eigenvectors of M_h for its r largest eigenvalues (Eq. 15), column j
 *      for the j-th largest (equal eigenvalues in increasing index order), each
 *      signed so that its largest-magnitude entry (the first such) is positive;
 *      0 when count = 0.
 *   eigenvalues: fp32 [H][d], all eigenvalues of M_h in decreasing order.
 * Any of w, U, eigenvalues may be NULL.  The eigen-solver is cyclic Jacobi in
 * fp32 on the whole 128 x 128 matrix, run until a sweep finds no off-diagonal
 * entry above 2^-20 of the Frobenius norm (at most 30 sweeps). */
QWM_API qwm_status qwm_query_basis(const qwm_config* cfg, const void* stats, float* w, void* U, float* eigenvalues,
                                   void* stream);

/* Synchronise `stream`, then read and clear the statistics' device status
 * word (*status) and read the Query count (*count, may be NULL). */
QWM_API qwm_status qwm_query_stats_read(void* stats, int32_t* status, int64_t* count, void* stream);

/* ---------------------------------------------------------------------------
 * Token-selection shift measurement (Sec. 5, table "top1_shift": the share of
 * queries whose highest-logit key changes when the cached Keys are quantized).
 * --------------------------------------------------------------------------- */

/* Reconstruction of cached chunk i (0 = oldest held; N = its token count from
 * qwm_cache_chunk_info), the values attention rebuilds (App. D.1 on-demand
 * reconstruction, Sec. 2 Eq. 3 and Sec. 4.2 Eq. 17):
 * k_hat_c = mu_id,c + s_g (q_c - z_g) + sum_j t_j sigma U_r[c][j] for Keys (the PSAC
 * term only when the chunk was stored with one), v_hat without it, in fp32
 * (s (q - z) and t sigma exact, one fused multiply-add per PSAC term).
 * k_out, v_out: fp32 [N][H][d], 16-byte aligned; either may be NULL. */
QWM_API qwm_status qwm_dequant_chunk(const qwm_config* cfg, const qwm_cache* cache, int32_t i, float* k_out,
                                     float* v_out, void* stream);

/* Top-1 key of every query and head: idx[h][n] = argmax_j q[n,h] . keys[j,h],
 * each logit the fp32 sum over channels in order with one fused multiply-add
 * per term, ties to the lower key index.  q: bf16 [Nq][H][d]; keys: fp32
 * [Nk][H][d] (16-byte aligned); idx: int32 [H][Nq].  Nq, Nk >= 1. */
QWM_API qwm_status qwm_top1_keys(const qwm_config* cfg, const void* q, int64_t Nq, const float* keys, int64_t Nk,
                                 int32_t* idx, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* QWM_H */
