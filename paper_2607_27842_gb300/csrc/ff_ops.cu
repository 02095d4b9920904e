// C ABI of include/featfix_ops.h: the hot-path kernels on caller buffers.
#include "featfix_ops.h"
#include "ff_common.cuh"

using namespace ff;

namespace {

bool dt_ok(int dt) { return dt == FEATFIX_DTYPE_F32 || dt == FEATFIX_DTYPE_BF16; }
bool al16(const void* p) { return ((uintptr_t)p & 15) == 0; }
featfix_status st(cudaError_t e) {
  if (e == cudaSuccess) return FEATFIX_OK;
  if (e == cudaErrorInvalidValue) return FEATFIX_ERR_INVALID_ARG;
  if (e == cudaErrorNotSupported) return FEATFIX_ERR_UNSUPPORTED;
  return FEATFIX_ERR_CUDA;
}

}  // namespace

extern "C" {

featfix_status featfix_op_draft(int dtype, void* dev_x, const void* const* dev_hist, const double* w, int n_terms,
                                long long n, void* stream) {
  if (!dt_ok(dtype) || !dev_x || !dev_hist || !w || n_terms < 1 || n_terms > 4 || n < 0) return FEATFIX_ERR_INVALID_ARG;
  Hist4 h = {{nullptr, nullptr, nullptr, nullptr}};
  float wf[4] = {0, 0, 0, 0};
  if (!al16(dev_x)) return FEATFIX_ERR_INVALID_ARG;
  for (int j = 0; j < n_terms; ++j) {
    if (!dev_hist[j] || !al16(dev_hist[j])) return FEATFIX_ERR_INVALID_ARG;
    h.p[j] = dev_hist[j];
    wf[j] = (float)w[j];
  }
  return st(launch_draft((DType)dtype, dev_x, h, wf, n_terms, n, (cudaStream_t)stream));
}

size_t featfix_op_verify_workspace(long long n) { return verify_workspace_bytes(n); }

featfix_status featfix_op_verify(int dtype, void* dev_u, const void* const* dev_hist, const double* w, int n_terms,
                                 const void* dev_hf, long long n, int write_draft, double* dev_sums,
                                 void* dev_workspace, size_t ws_bytes, void* stream) {
  if (!dt_ok(dtype) || !dev_u || !dev_hist || !w || !dev_hf || !dev_sums || !dev_workspace || n_terms < 1 ||
      n_terms > 4 || n <= 0)
    return FEATFIX_ERR_INVALID_ARG;
  if (ws_bytes < verify_workspace_bytes(n)) return FEATFIX_ERR_INVALID_ARG;
  if (!al16(dev_u) || !al16(dev_hf) || !al16(dev_workspace)) return FEATFIX_ERR_INVALID_ARG;
  Hist4 h = {{nullptr, nullptr, nullptr, nullptr}};
  float wf[4] = {0, 0, 0, 0};
  for (int j = 0; j < n_terms; ++j) {
    if (!dev_hist[j] || !al16(dev_hist[j])) return FEATFIX_ERR_INVALID_ARG;
    h.p[j] = dev_hist[j];
    wf[j] = (float)w[j];
  }
  return st(launch_verify((DType)dtype, dev_u, h, wf, n_terms, dev_hf, n, write_draft, dev_sums, dev_workspace,
                          (cudaStream_t)stream));
}

featfix_status featfix_op_ln_modulate(int dtype, const void* dev_x, void* dev_out, long long rows, int C,
                                      const float* dev_shift, const float* dev_scale, int mod_stride,
                                      int rows_per_batch, void* stream) {
  if (!dt_ok(dtype) || !dev_x || !dev_out || !dev_shift || !dev_scale || rows < 0 || C <= 0 || rows_per_batch <= 0)
    return FEATFIX_ERR_INVALID_ARG;
  if (C % (dtype == FEATFIX_DTYPE_F32 ? 4 : 8)) return FEATFIX_ERR_INVALID_ARG;
  return st(launch_ln_mod((DType)dtype, dev_x, dev_out, rows, C, dev_shift, dev_scale, mod_stride, 0, 1,
                          rows_per_batch, (cudaStream_t)stream));
}

featfix_status featfix_op_gemm(int dtype, int M, int N, int K, const void* dev_a, const void* dev_w,
                               const void* dev_bias, int act, const float* dev_gate, int gate_stride,
                               int rows_per_batch, const void* dev_resid, void* dev_out, const void* dev_hist_base,
                               void* dev_hist_out, void* stream) {
  if (!dt_ok(dtype) || M < 0 || N <= 0 || K <= 0 || !dev_a || !dev_w || !dev_out) return FEATFIX_ERR_INVALID_ARG;
  if (act != 0 && act != 1) return FEATFIX_ERR_INVALID_ARG;
  if ((dev_gate != nullptr) && (rows_per_batch <= 0 || gate_stride < N)) return FEATFIX_ERR_INVALID_ARG;
  if ((dev_hist_out != nullptr) != (dev_hist_base != nullptr)) return FEATFIX_ERR_INVALID_ARG;
  if (N % (dtype == FEATFIX_DTYPE_F32 ? 4 : 8)) return FEATFIX_ERR_INVALID_ARG;
  EpiArgs e = epi_plain(dev_out, N);
  e.bias = dev_bias;
  e.act = act;
  e.gate = dev_gate;
  e.gate_stride = gate_stride;
  e.rpb1 = rows_per_batch > 0 ? rows_per_batch : 1;
  e.resid = dev_resid;
  e.ld_resid = N;
  e.hist_base = dev_hist_base;
  e.hist_out = dev_hist_out;
  if (dtype == FEATFIX_DTYPE_BF16) return st(gemm_tc(M, N, K, dev_a, K, dev_w, K, e, (cudaStream_t)stream));
  return st(gemm_simt(F32, M, N, K, dev_a, K, dev_w, K, e, (cudaStream_t)stream));
}

featfix_status featfix_op_attention(int dtype, const void* dev_qkv, int ld_qkv, void* dev_out, int ld_out, int batch,
                                    int n_txt, int n_img, int heads, int head_dim, void* stream) {
  if (!dt_ok(dtype) || !dev_qkv || !dev_out || batch <= 0 || n_txt < 0 || n_img < 0 || heads <= 0 ||
      head_dim <= 0 || head_dim % 8 || head_dim > 128)
    return FEATFIX_ERR_INVALID_ARG;
  const int C = heads * head_dim;
  if (ld_qkv < 3 * C || ld_out < C) return FEATFIX_ERR_INVALID_ARG;
  const int es = dtype == FEATFIX_DTYPE_F32 ? 4 : 2;
  const char* base = reinterpret_cast<const char*>(dev_qkv);
  AttnArgs a;
  a.q = base;
  a.k = base + (size_t)C * es;
  a.v = base + (size_t)2 * C * es;
  a.ld_qkv = ld_qkv;
  a.out = dev_out;
  a.ld_out = ld_out;
  a.B = batch;
  a.Nt = n_txt;
  a.Ni = n_img;
  a.H = heads;
  a.hd = head_dim;
  return st(attention((DType)dtype, a, (cudaStream_t)stream));
}

}  // extern "C"
