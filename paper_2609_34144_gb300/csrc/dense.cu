// Dense projections of the residual sites beyond the attention output (App. B.1, B.4): the
// output projection W_O of the anchor rows and the two GEMMs of the anchor FFN, as one
// persistent tcgen05 kernel per GEMM over the rows of every anchor.
//
//   C[anchor i, row r, :] = act(A[a_frame[i], r, :] W^T + bias),  r < S,
//
// bf16 A and W (K contiguous), f32 accumulation in TMEM, bias (+ GELU, tanh form) in the
// epilogue, C in bf16 or f32.  Tiles of 128 rows x 256 columns; a tile never spans anchors
// (rows past S read as zero through the 3-D tensor map [frame][row][k] and are not written).
// Persistent CTAs, one per SM, each loading its own A and W k-slices (no clusters): CTAs that
// run at the same time take neighbouring column tiles of one row tile, so the A tile and the
// W matrix (a few MB) are served from L2.
// Warp roles (384 threads, one CTA per SM, 193 KB shared memory, 512 TMEM columns):
//   warp 0      TMA producer: A (128 x 64) and W (256 x 64) k-slices into a 4-stage ring
//   warp 1      TMEM owner and single-thread UMMA issuer (kind::f16, M = 128, N = 256, K = 16),
//               accumulating each tile in one of two 256-column TMEM buffers
//   warps 4..11 epilogue: one output row per thread and half of the tile's columns per warp
//               (warps 4-7 columns 0-127, warps 8-11 columns 128-255), tcgen05.ld of 32
//               columns at a time, bias (vector loads issued before the TMEM load), GELU,
//               conversion and vector stores; the buffer is handed back to the issuer, so the
//               next tile's mainloop overlaps this tile's epilogue.
// Every wait is bounded; on a timeout the CTA records an error word, drains its UMMAs and
// frees TMEM before leaving.
#include <cuda_bf16.h>

#include "internal.h"
#include "ptx.cuh"

namespace cast {
namespace {

__device__ unsigned int g_dense_error;

constexpr int GBM = 128, GBN = 256, GBK = 64, kGStages = 4;
constexpr int kGThreads = 384;
constexpr int kEpiThreads = 256;
constexpr int kABytes = GBM * GBK * 2, kBBytes = GBN * GBK * 2, kStageBytes = kABytes + kBBytes;
constexpr int kGSmem = kGStages * kStageBytes + 256 + 1024;   // ring + barriers + alignment slack

struct GemmKArgs {
  int S, N, K, n_anchors, m_tiles, n_tiles, n_k;
  int total_tiles;   // n_anchors * m_tiles * n_tiles
  const void* bias;
  void* c;
  int64_t ldc;
  int c_f32, bias_f32, gelu;
  unsigned long long wait_ns;
  int a_frame[CAST_MAX_ANCHORS];
  int c_frame[CAST_MAX_ANCHORS];
};

struct GBars {
  uint64_t full[kGStages], empty[kGStages];
  uint64_t acc_full[2], acc_empty[2];
  uint64_t fin;
  uint32_t tmem_base;
  int abort;
};

__device__ __forceinline__ bool g_aborted(const GBars* b) {
  return *reinterpret_cast<const volatile int*>(&b->abort) != 0;
}
__device__ __forceinline__ void g_set_abort(GBars* b) {
  atomicExch(&b->abort, 1);
  atomicExch(&g_dense_error, 1u);
}
__device__ __forceinline__ void g_end_barrier() {
  asm volatile("barrier.sync 1, %0;" ::"n"(kGThreads) : "memory");
}

// GELU in its tanh form, 0.5 x (1 + tanh(sqrt(2/pi) (x + 0.044715 x^3))), with the hardware
// tanh approximation
__device__ __forceinline__ float gelu_tanh(float x) {
  const float u = 0.7978845608028654f * fmaf(0.044715f * x, x * x, x);
  float t;
  asm("tanh.approx.f32 %0, %1;" : "=f"(t) : "f"(u));
  return 0.5f * x * (1.f + t);
}

// Tile t -> (anchor i, row tile mt, column tile nt), column tiles innermost; a row tile past
// the anchor's rows reads zeros and writes nothing.
__device__ __forceinline__ void tile_of(const GemmKArgs& a, int t, int& i, int& mt, int& nt) {
  const int per_anchor = a.m_tiles * a.n_tiles;
  i = t / per_anchor;
  const int rem = t - i * per_anchor;
  mt = rem / a.n_tiles;
  nt = rem - mt * a.n_tiles;
}

__global__ void __launch_bounds__(kGThreads, 1)
    k_gemm(const __grid_constant__ CUtensorMap tm_a, const __grid_constant__ CUtensorMap tm_w,
           const __grid_constant__ GemmKArgs a) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  uint8_t* smem = smem_raw + (((raw + 1023u) & ~1023u) - raw);
  GBars* bars = reinterpret_cast<GBars*>(smem + kGStages * kStageBytes);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint64_t lim = a.wait_ns;
  const int first = blockIdx.x, stride = gridDim.x;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kGStages; ++s) {
      mbar_init(&bars->full[s], 1);
      mbar_init(&bars->empty[s], 1);   // released by the UMMA issuer
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&bars->acc_full[b], 1);
      mbar_init(&bars->acc_empty[b], kEpiThreads);
    }
    mbar_init(&bars->fin, 1);
    bars->abort = 0;
    fence_barrier_init();
  }
  if (warp == 1) {
    tmem_alloc(&bars->tmem_base, 512);
    tmem_relinquish();
    tc_fence_before();
  }
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bars->tmem_base;

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------------------ TMA producer
      tma_prefetch_desc(&tm_a);
      tma_prefetch_desc(&tm_w);
      int it = 0;
      bool ok = true;
      for (int t = first; ok && t < a.total_tiles; t += stride) {
        int i, mt, nt;
        tile_of(a, t, i, mt, nt);
        for (int ks = 0; ks < a.n_k; ++ks, ++it) {
          const int s = it % kGStages;
          // the UMMAs that read this stage have completed
          if (g_aborted(bars) || !mbar_wait(&bars->empty[s], ((uint32_t)(it / kGStages) & 1u) ^ 1u, lim)) {
            g_set_abort(bars);
            ok = false;
            break;
          }
          uint8_t* st = smem + s * kStageBytes;
          mbar_arrive_expect_tx(&bars->full[s], kStageBytes);   // A + W k-slices
          tma_load_3d(st, &tm_a, &bars->full[s], ks * GBK, mt * GBM, a.a_frame[i]);
          tma_load_2d(st + kABytes, &tm_w, &bars->full[s], ks * GBK, nt * GBN);
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ------------------------------------------------------------ UMMA issuer
      constexpr uint32_t idesc = idesc_bf16_f32(GBM, GBN, false, false);
      const uint32_t base = smem_u32(smem);
      int it = 0, lt = 0;
      bool ok = true;
      for (int t = first; ok && t < a.total_tiles; t += stride, ++lt) {
        const int buf = lt & 1;
        if (g_aborted(bars) || !mbar_wait(&bars->acc_empty[buf], ((uint32_t)(lt >> 1) & 1u) ^ 1u, lim)) {
          ok = false;
          break;
        }
        tc_fence_after();
        for (int ks = 0; ks < a.n_k; ++ks, ++it) {
          const int s = it % kGStages;
          if (g_aborted(bars) || !mbar_wait(&bars->full[s], (uint32_t)(it / kGStages) & 1u, lim)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sa = base + s * kStageBytes, sb = sa + kABytes;
#pragma unroll
          for (int kk = 0; kk < GBK / 16; ++kk)
            umma_bf16_ss(tmem + buf * GBN, sdesc_sw128(sa + kk * 32, 16, 1024),
                         sdesc_sw128(sb + kk * 32, 16, 1024), idesc, (ks > 0 || kk > 0) ? 1u : 0u);
          umma_commit(&bars->empty[s]);   // the stage is free once these UMMAs have read it
        }
        if (!ok) break;
        umma_commit(&bars->acc_full[buf]);
      }
      if (!ok) g_set_abort(bars);
      // every issued UMMA has completed before TMEM is released
      umma_commit(&bars->fin);
      mbar_wait(&bars->fin, 0, lim);
    }
  } else if (warp >= 4) {
    // ------------------------------------------------------------ epilogue
    const int q4 = warp & 3, half = (warp - 4) >> 2;
    const int row = q4 * 32 + lane;
    int lt = 0;
    for (int t = first; t < a.total_tiles; t += stride, ++lt) {
      const int buf = lt & 1;
      const bool w = !g_aborted(bars) && mbar_wait(&bars->acc_full[buf], (uint32_t)(lt >> 1) & 1u, lim);
      if (!__all_sync(0xffffffffu, w)) {
        g_set_abort(bars);
        break;
      }
      tc_fence_after();
      int i, mt, nt;
      tile_of(a, t, i, mt, nt);
      const int r = mt * GBM + row;
      const bool live = r < a.S;
      const uint32_t tl = tmem + buf * GBN + ((uint32_t)(q4 * 32) << 16);
      const int64_t crow = ((int64_t)a.c_frame[i] * a.S + r) * a.ldc;
#pragma unroll 1
      for (int ch = half * 4; ch < half * 4 + 4; ++ch) {
        const int n0 = nt * GBN + ch * 32;
        // bias of the 32 columns (the same for every row): vector loads in flight before the
        // TMEM load
        float bv[32];
        const bool full = n0 + 32 <= a.N;
        if (a.bias && full) {
          if (a.bias_f32) {
            const float4* bp = reinterpret_cast<const float4*>(static_cast<const float*>(a.bias) + n0);
#pragma unroll
            for (int q = 0; q < 8; ++q) {
              const float4 v4 = __ldg(bp + q);
              bv[4 * q] = v4.x; bv[4 * q + 1] = v4.y; bv[4 * q + 2] = v4.z; bv[4 * q + 3] = v4.w;
            }
          } else {
            const uint4* bp = reinterpret_cast<const uint4*>(static_cast<const __nv_bfloat16*>(a.bias) + n0);
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              const uint4 u4 = __ldg(bp + q);
              const uint32_t wds[4] = {u4.x, u4.y, u4.z, u4.w};
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                bv[8 * q + 2 * e] = __uint_as_float(wds[e] << 16);
                bv[8 * q + 2 * e + 1] = __uint_as_float(wds[e] & 0xFFFF0000u);
              }
            }
          }
        } else {
#pragma unroll
          for (int c = 0; c < 32; ++c) {
            const int n = n0 + c;
            bv[c] = 0.f;
            if (a.bias && n < a.N)
              bv[c] = a.bias_f32 ? __ldg(static_cast<const float*>(a.bias) + n)
                                 : __bfloat162float(__ldg(static_cast<const __nv_bfloat16*>(a.bias) + n));
          }
        }
        uint32_t v[32];
        tmem_ld_x32(tl + ch * 32, v);   // warp-collective: every lane loads
        if (!live || n0 >= a.N) continue;
        float y[32];
#pragma unroll
        for (int c = 0; c < 32; ++c) {
          const float x = __uint_as_float(v[c]) + bv[c];
          y[c] = a.gelu ? gelu_tanh(x) : x;
        }
        if (a.c_f32) {
          float* dst = static_cast<float*>(a.c) + crow + n0;
          if (full) {
#pragma unroll
            for (int c = 0; c < 32; c += 4)
              *reinterpret_cast<float4*>(dst + c) = make_float4(y[c], y[c + 1], y[c + 2], y[c + 3]);
          } else {
#pragma unroll
            for (int c = 0; c < 32; ++c)
              if (n0 + c < a.N) dst[c] = y[c];
          }
        } else {
          __nv_bfloat16* dst = static_cast<__nv_bfloat16*>(a.c) + crow + n0;
          if (full) {
#pragma unroll
            for (int c = 0; c < 32; c += 8) {
              uint32_t pk[4];
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                __nv_bfloat162 b2 = __floats2bfloat162_rn(y[c + 2 * e], y[c + 2 * e + 1]);
                pk[e] = *reinterpret_cast<uint32_t*>(&b2);
              }
              *reinterpret_cast<uint4*>(dst + c) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
            }
          } else {
#pragma unroll
            for (int c = 0; c < 32; ++c)
              if (n0 + c < a.N) dst[c] = __float2bfloat16_rn(y[c]);
          }
        }
      }
      // the accumulator buffer is free for the tile after next
      tc_fence_before();
      mbar_arrive(&bars->acc_empty[buf]);
    }
  }
  // the last UMMA has completed (fin) and every epilogue thread has read TMEM
  tc_fence_before();
  g_end_barrier();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// bf16 [depth][rows][inner] (rank 2 when depth == 0), box 64 x box_rows (x 1), 128-B swizzle
bool make_gemm_map(CUtensorMap* m, const void* base, uint64_t inner, uint64_t rows,
                   uint64_t row_stride_bytes, uint64_t depth, uint64_t depth_stride_bytes,
                   uint32_t box_rows) {
  EncodeTiledFn fn = tensor_map_encoder();
  if (!fn) return false;
  cuuint64_t dims[3] = {inner, rows, depth};
  cuuint64_t strides[2] = {row_stride_bytes, depth_stride_bytes};
  cuuint32_t box[3] = {64, box_rows, 1};
  cuuint32_t es[3] = {1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, depth ? 3 : 2, const_cast<void*>(base), dims, strides,
            box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

cast_status gemm_anchor_rows(const AnchorGemm& g, cudaStream_t st) {
  if (g.n_anchors < 1 || g.S < 1 || g.N < 1 || g.K < 1) return CAST_OK;
  CUtensorMap ma, mw;
  if (!make_gemm_map(&ma, g.a, (uint64_t)g.K, (uint64_t)g.S, (uint64_t)g.lda * 2, (uint64_t)g.a_frames,
                     (uint64_t)g.a_frame_stride * 2, GBM) ||
      !make_gemm_map(&mw, g.w, (uint64_t)g.K, (uint64_t)g.N, (uint64_t)g.ldw * 2, 0, 0, GBN))
    return fail(CAST_ERR_CUDA, "dense: cuTensorMapEncodeTiled failed");
  GemmKArgs k{};
  k.S = g.S;
  k.N = g.N;
  k.K = g.K;
  k.n_anchors = g.n_anchors;
  k.m_tiles = (g.S + GBM - 1) / GBM;
  k.n_tiles = (g.N + GBN - 1) / GBN;
  k.n_k = (g.K + GBK - 1) / GBK;
  k.total_tiles = g.n_anchors * k.m_tiles * k.n_tiles;
  k.bias = g.bias;
  k.c = g.c;
  k.ldc = g.ldc;
  k.c_f32 = g.c_dtype == CAST_F32;
  k.bias_f32 = g.bias_dtype == CAST_F32;
  k.gelu = g.gelu ? 1 : 0;
  k.wait_ns = 2000000000ull;
  for (int j = 0; j < g.n_anchors; ++j) {
    k.a_frame[j] = g.a_frame[j];
    k.c_frame[j] = g.c_frame[j];
  }
  static std::atomic<uint64_t> attr_done{0};
  if (!once_per_device(attr_done, [] {
        return cudaFuncSetAttribute(k_gemm, cudaFuncAttributeMaxDynamicSharedMemorySize, kGSmem) ==
               cudaSuccess;
      }))
    return check_launch("dense GEMM smem attribute");
  int dev = 0, nsm = 148;
  if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
  const int grid = k.total_tiles < nsm ? k.total_tiles : nsm;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(grid > 0 ? grid : 1, 1, 1);
  cfg.blockDim = dim3(kGThreads, 1, 1);
  cfg.dynamicSmemBytes = kGSmem;
  cfg.stream = st;
  cfg.numAttrs = 0;
  if (cudaLaunchKernelEx(&cfg, k_gemm, ma, mw, k) != cudaSuccess) return check_launch("dense GEMM kernel");
  return check_launch("dense GEMM kernel");
}

unsigned int dense_error_word(cudaStream_t st, bool clear) {
  unsigned int v = 0;
  cudaMemcpyFromSymbolAsync(&v, g_dense_error, sizeof(v), 0, cudaMemcpyDeviceToHost, st);
  cudaStreamSynchronize(st);
  if (clear && v) {
    const unsigned int z = 0;
    cudaMemcpyToSymbolAsync(g_dense_error, &z, sizeof(z), 0, cudaMemcpyHostToDevice, st);
    cudaStreamSynchronize(st);
  }
  return v;
}

}  // namespace cast
