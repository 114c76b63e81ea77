// Dense projections of the residual sites beyond the attention output (App. B.1, B.4): the
// output projection W_O of the anchor rows and the two GEMMs of the anchor FFN.  These are
// plain GEMMs, run through cuBLASLt (bf16 operands, f32 accumulation, bias / GELU-bias
// epilogues, the caller's workspace); everything around them (routing, attention, PAR) stays
// in this library's kernels.
#include <cublasLt.h>

#include <mutex>

#include "internal.h"

namespace cast {
namespace {

cast_status lt_handle(cublasLtHandle_t* out) {
  static std::mutex mu;
  static cublasLtHandle_t per_dev[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return check_launch("cuBLASLt device");
  std::lock_guard<std::mutex> lock(mu);
  if (!per_dev[dev] && cublasLtCreate(&per_dev[dev]) != CUBLAS_STATUS_SUCCESS)
    return fail(CAST_ERR_CUDA, "cublasLtCreate failed");
  *out = per_dev[dev];
  return CAST_OK;
}

#define LT_CHECK(x, what)                                                          \
  do {                                                                             \
    const cublasStatus_t st_ = (x);                                                \
    if (st_ != CUBLAS_STATUS_SUCCESS) {                                            \
      ok = fail(CAST_ERR_CUDA, "cuBLASLt %s failed (status %d)", what, (int)st_); \
      goto done;                                                                   \
    }                                                                              \
  } while (0)

}  // namespace

// Row-major C[M, N] = act(A[M, K] W[N, K]^T + bias[N]): A, W bf16; C and bias of c_dtype.
// cuBLASLt works column-major, so it computes C^T = W A^T with W transposed.
cast_status gemm_rows(const GemmRows& g, cudaStream_t st) {
  cublasLtHandle_t h;
  cast_status ok = lt_handle(&h);
  if (ok) return ok;
  cublasLtMatmulDesc_t op = nullptr;
  cublasLtMatrixLayout_t la = nullptr, lb = nullptr, lc = nullptr;
  cublasLtMatmulPreference_t pref = nullptr;
  const cudaDataType_t ct = g.c_dtype == CAST_BF16 ? CUDA_R_16BF : CUDA_R_32F;
  const cublasOperation_t tA = CUBLAS_OP_T, tB = CUBLAS_OP_N;
  cublasLtEpilogue_t epi = g.gelu ? (g.bias ? CUBLASLT_EPILOGUE_GELU_BIAS : CUBLASLT_EPILOGUE_GELU)
                                  : (g.bias ? CUBLASLT_EPILOGUE_BIAS : CUBLASLT_EPILOGUE_DEFAULT);
  const float alpha = 1.f, beta = 0.f;
  cublasLtMatmulHeuristicResult_t heur{};
  int n_res = 0;
  LT_CHECK(cublasLtMatmulDescCreate(&op, CUBLAS_COMPUTE_32F, CUDA_R_32F), "descriptor");
  LT_CHECK(cublasLtMatmulDescSetAttribute(op, CUBLASLT_MATMUL_DESC_TRANSA, &tA, sizeof(tA)), "transa");
  LT_CHECK(cublasLtMatmulDescSetAttribute(op, CUBLASLT_MATMUL_DESC_TRANSB, &tB, sizeof(tB)), "transb");
  LT_CHECK(cublasLtMatmulDescSetAttribute(op, CUBLASLT_MATMUL_DESC_EPILOGUE, &epi, sizeof(epi)), "epilogue");
  if (g.bias) {
    LT_CHECK(cublasLtMatmulDescSetAttribute(op, CUBLASLT_MATMUL_DESC_BIAS_POINTER, &g.bias, sizeof(g.bias)),
             "bias pointer");
    LT_CHECK(cublasLtMatmulDescSetAttribute(op, CUBLASLT_MATMUL_DESC_BIAS_DATA_TYPE, &ct, sizeof(ct)),
             "bias type");
  }
  // column-major views: W^T is [K, N] (ld ldw), A^T is [K, M] (ld lda), C^T is [N, M] (ld ldc)
  LT_CHECK(cublasLtMatrixLayoutCreate(&la, CUDA_R_16BF, g.K, g.N, g.ldw), "layout W");
  LT_CHECK(cublasLtMatrixLayoutCreate(&lb, CUDA_R_16BF, g.K, g.M, g.lda), "layout A");
  LT_CHECK(cublasLtMatrixLayoutCreate(&lc, ct, g.N, g.M, g.ldc), "layout C");
  LT_CHECK(cublasLtMatmulPreferenceCreate(&pref), "preference");
  LT_CHECK(cublasLtMatmulPreferenceSetAttribute(pref, CUBLASLT_MATMUL_PREF_MAX_WORKSPACE_BYTES,
                                                &g.ws_bytes, sizeof(g.ws_bytes)), "workspace preference");
  LT_CHECK(cublasLtMatmulAlgoGetHeuristic(h, op, la, lb, lc, lc, pref, 1, &heur, &n_res), "heuristic");
  if (n_res < 1) {
    ok = fail(CAST_ERR_UNSUPPORTED, "cuBLASLt has no algorithm for %d x %d x %d", g.M, g.N, g.K);
    goto done;
  }
  LT_CHECK(cublasLtMatmul(h, op, &alpha, g.w, la, g.a, lb, &beta, g.c, lc, g.c, lc, &heur.algo, g.ws,
                          g.ws_bytes, st), "matmul");
  ok = check_launch("cuBLASLt matmul");
done:
  if (pref) cublasLtMatmulPreferenceDestroy(pref);
  if (lc) cublasLtMatrixLayoutDestroy(lc);
  if (lb) cublasLtMatrixLayoutDestroy(lb);
  if (la) cublasLtMatrixLayoutDestroy(la);
  if (op) cublasLtMatmulDescDestroy(op);
  return ok;
}

}  // namespace cast
