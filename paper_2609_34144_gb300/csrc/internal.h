// Internal declarations shared by the translation units of libcast.
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>

#include <atomic>
#include <cstddef>
#include <cstdint>

#include "cast.h"

namespace cast {

// Records a printf-style message for cast_last_error_detail() and returns `s`.
cast_status fail(cast_status s, const char* fmt, ...);
// Empties the message cast_last_error_detail() returns (at the start of every entry point).
void clear_error_detail();
// Converts a pending launch error into CAST_ERR_CUDA.
cast_status check_launch(const char* what);

// cuTensorMapEncodeTiled fetched from the driver through the runtime (no libcuda link);
// nullptr if unavailable.
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeTiledFn tensor_map_encoder();

// Runs setup() for the current device unless it already succeeded there: kernel attributes
// (the dynamic shared-memory limit) belong to one device's context, so a process that drives
// several devices sets them once per device.  Concurrent first calls may both run setup().
template <class F>
bool once_per_device(std::atomic<uint64_t>& done, F&& setup) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return setup();
  const uint64_t bit = 1ull << dev;
  if (done.load(std::memory_order_acquire) & bit) return true;
  if (!setup()) return false;
  done.fetch_or(bit, std::memory_order_acq_rel);
  return true;
}

constexpr size_t kWsAlign = 256;
inline size_t align_up(size_t x, size_t a = kWsAlign) { return (x + a - 1) / a * a; }

// ------------------------------------------------------------------ history layout
// Geometry of CAST_HIST_FRAMES: (1, 8, 8) blocks over frames of an Hg x Wg token grid.
constexpr int kSpatialBlock = 8;
struct HistGeom {
  bool spatial;
  int frames, Hg, Wg, nby, nbx;   // nby x nbx blocks per frame
  int64_t blocks() const { return (int64_t)frames * nby * nbx; }
};
inline HistGeom hist_geom(const cast_hist_layout& h) {
  HistGeom g{};
  g.spatial = h.kind == CAST_HIST_FRAMES;
  if (g.spatial) {
    g.frames = h.frames;
    g.Hg = h.Hg;
    g.Wg = h.Wg;
    g.nby = h.Hg > 0 ? (h.Hg + kSpatialBlock - 1) / kSpatialBlock : 0;
    g.nbx = h.Wg > 0 ? (h.Wg + kSpatialBlock - 1) / kSpatialBlock : 0;
  }
  return g;
}

// ------------------------------------------------------------------ routing
struct RoutePlan {
  int n_seg;        // n_anchors + 2 M pooled segments
  int nsplit_q;     // row splits of an anchor-frame segment (CTAs of one cluster)
  int nsplit_kv;    // row splits of a history-block segment
  bool wide;        // per-head statistics spread over a cluster of CTAs (large M)
  int cl;           // CTAs per head in the wide form
  size_t pooled_bytes, total_bytes;
};
RoutePlan route_plan(const cast_route_args& a);
// shared memory of the pooling kernel (column sums of one CTA) and of the per-head kernel
// (pooled query, o_bar, pi, keys and masks of every anchor of one head)
size_t route_pool_smem_bytes(const cast_route_args& a);
size_t route_head_smem_bytes(const cast_route_args& a);
// Arguments must have been validated; ws holds at least route_plan(a).total_bytes.
cast_status launch_route(const cast_route_args& a, void* ws, cudaStream_t st);
// Nonzero when a routing kernel met a candidate index outside [0, M) or repeated in its set.
unsigned int route_error_word(cudaStream_t st, bool clear);

// ------------------------------------------------------------------ attention
struct AttnPlan {
  int n_pairs, n_single, n_cur_tiles, tiles_per_block;
  int n_hist_tiles;   // K/V tiles of the routed history (two (1,8,8) blocks per tile when spatial)
  int n_full, n_tail, n_split, chunk, grid;
  size_t part_o_bytes, part_ml_bytes, counter_bytes, total_bytes;
};
AttnPlan attention_plan(const cast_attn_args& a);
// o_frame_of_anchor: 0 -> output frame i for anchor i (o is [n_anchors, S, H*d]);
//                    1 -> output frame anchors[i] (o is [n_frames, S, H*d], block step).
// ws holds attention_plan(a).total_bytes (may be null when that is 0).
// after_route: launched right behind the routing kernels as a programmatic dependent (history
// tiles wait on the grid dependency); the caller has run attention_reset_counters() on the
// stream before routing.
cast_status launch_attention(const cast_attn_args& a, int o_frame_of_anchor, void* ws,
                             cudaStream_t st, bool after_route = false);
cast_status attention_reset_counters(const cast_attn_args& a, void* ws, cudaStream_t st);
unsigned int attention_error_word(cudaStream_t st, bool clear);
// A kernel whose only wait can never be satisfied and so runs into its deadline (limit_ns).
cast_status launch_bounded_wait_selftest(uint64_t limit_ns, cudaStream_t st);

// ------------------------------------------------------------------ PAR
struct ParPlan {
  int n_anchor, n_pair, n_target;
  int tiles_y, tiles_x, n_tile;
  int n_full, n_edge;   // 8x8 tiles / truncated (or non-8x8) tiles
  int chunk;        // channels per CTA (= threads per CTA)
  int n_chunk;      // channel chunks per tile
  int n_tseg_full, n_tseg_edge;   // time segments (runs of anchor pairs) per tile, per kind
  size_t rec_bytes, trans_bytes, img_bytes, total_bytes;   // workspace: chunk records, theta and g,
                                                          // blend matrices (bf16)
};
ParPlan par_plan(const cast_par_args& a);
cast_status launch_par(const cast_par_args& a, void* ws, cudaStream_t st);
unsigned int par_error_word(cudaStream_t st, bool clear);

// ------------------------------------------------------------------ dense projections
// C[anchor i, row r, :] = act(A[a_frame[i], r, :] W[N, K]^T + bias[N]) for r < S: A, W bf16
// (16-byte aligned rows, lda / ldw multiples of 8), row r of anchor i of A at
// a + (a_frame[i] * a_frame_stride + r * lda), of C at c + (c_frame[i] * S + r) * ldc; C and
// bias of their dtypes; act = GELU (tanh form) when gelu.  One tcgen05 kernel per call.
struct AnchorGemm {
  const void* a;
  int64_t lda, a_frame_stride;
  int a_frames;                  // frames the A tensor holds (its tensor map depth)
  const void* w;
  int64_t ldw;
  const void* bias;
  int bias_dtype;
  void* c;
  int64_t ldc;
  int c_dtype;
  int S, N, K, n_anchors;
  int a_frame[CAST_MAX_ANCHORS], c_frame[CAST_MAX_ANCHORS];
  bool gelu;
};
cast_status gemm_anchor_rows(const AnchorGemm& g, cudaStream_t st);
unsigned int dense_error_word(cudaStream_t st, bool clear);

// ------------------------------------------------------------------ residual update
cast_status launch_residual_add(void* x, const void* r, int dtype, size_t n, cudaStream_t st);

}  // namespace cast
