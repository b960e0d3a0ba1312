// One training step of a ShiftQuant-quantized linear layer through the library's own entry
// points: the range pass, grouping and quantization of X (round to nearest) and dY
// (stochastic rounding), the two weight roles with the ShiftMM shifts folded in, and the
// three GEMMs as one launch -- the operand roles of the paper's setup (Sec. 5.1; Eq. 4;
// App. D).  The host variant also moves the step's inputs in from host memory and its
// results back, inside the same stream order, so that a caller holding its data in host
// memory drives the whole path with one call per layer and step.
//
// Host code only: every arithmetic step is a kernel of sq_quant.cu or sq_gemm.cu.
#include <cuda_runtime.h>

#include "sq_host.h"

namespace sq {

// every pointer a step reads or writes, checked once before the first launch
static int check_step(const sq_layer_step* L) {
  if (L == nullptr) return fail(SQ_EINVAL, "layer_step: args is NULL");
  if (!bits_ok(L->bits) || !groups_ok(L->n_groups))
    return fail(SQ_EINVAL, "layer_step: bits must be in [2, 8] and n_groups in [1, 8]");
  if (L->M < 0 || L->K < 0 || L->N < 0) return fail(SQ_EINVAL, "layer_step: negative size");
  if (L->dev_status == nullptr) return fail(SQ_EINVAL, "layer_step: dev_status is required");
  if (L->M == 0 || L->K == 0 || L->N == 0) return SQ_OK;
  const void* need[] = {L->x, L->w, L->dy, L->x_codes, L->x_range, L->x_tau0,
                        L->x_scale, L->x_exp, L->g_codes, L->g_range, L->g_tau0,
                        L->g_scale, L->g_exp, L->wf_codes, L->wf_range, L->wf_scale,
                        L->wd_codes, L->wd_range, L->wd_scale, L->y, L->dx, L->dw};
  for (const void* p : need)
    if (p == nullptr) return fail(SQ_EINVAL, "layer_step: a required buffer is NULL");
  return SQ_OK;
}

// the device part of the step, in stream order on s
static int run_step(const sq_layer_step* L, uint64_t seed, void* s) {
  const int64_t M = L->M, K = L->K, N = L->N;
  const int b = L->bits, G = L->n_groups;
  int st;
  // activation: range pass + grouping, then codes and (if asked for) the transposed copy
  // (RN); without the copy the weight gradient reads the codes MN-major
  if ((st = shiftquant_calibrate(L->x, M, K, K, SQ_GRAN_SHIFT, G, L->x_range, L->x_tau0,
                                 L->x_exp, L->dev_status, s)) != SQ_OK)
    return st;
  if ((st = shiftquant_quantize(L->x, M, K, K, SQ_GRAN_SHIFT, b, G, L->x_tau0, L->x_exp, nullptr,
                                SQ_ROUND_NEAREST_EVEN, 0, 0, L->x_codes, L->ld_x, L->xt_codes,
                                L->ld_xt, L->x_scale, s)) != SQ_OK)
    return st;
  // gradient: the same with stochastic rounding
  if ((st = shiftquant_calibrate(L->dy, M, N, N, SQ_GRAN_SHIFT, G, L->g_range, L->g_tau0,
                                 L->g_exp, L->dev_status, s)) != SQ_OK)
    return st;
  if ((st = shiftquant_quantize(L->dy, M, N, N, SQ_GRAN_SHIFT, b, G, L->g_tau0, L->g_exp, nullptr,
                                SQ_ROUND_STOCHASTIC, seed, 0, L->g_codes, L->ld_g, L->gt_codes,
                                L->ld_gt, L->g_scale, s)) != SQ_OK)
    return st;
  // weight, both roles from two passes over it: forward per out-channel (column), written
  // transposed [N, K], X's shifts in; loss propagation per in-channel (row), natural layout,
  // dY's shifts in
  if ((st = shiftquant_calibrate_weight(L->w, K, N, N, L->wf_range, L->wd_range, L->dev_status,
                                        s)) != SQ_OK)
    return st;
  if ((st = shiftquant_quantize_weight(L->w, K, N, N, b, G, L->wf_range, L->wd_range, L->x_exp,
                                       L->g_exp, L->wf_codes, L->ld_wf, L->wf_scale, L->wd_codes,
                                       L->ld_wd, L->wd_scale, s)) != SQ_OK)
    return st;
  // the three GEMMs, one persistent launch
  sq_layer_gemms g = {};
  g.x_codes = L->x_codes;   g.ld_x = L->ld_x;
  g.xt_codes = L->xt_codes; g.ld_xt = L->ld_xt;
  g.x_scale = L->x_scale;   g.x_exp = L->x_exp;
  g.g_codes = L->g_codes;   g.ld_g = L->ld_g;
  g.gt_codes = L->gt_codes; g.ld_gt = L->ld_gt;
  g.g_scale = L->g_scale;   g.g_exp = L->g_exp;
  g.wf_codes = L->wf_codes; g.ld_wf = L->ld_wf; g.wf_scale = L->wf_scale;
  g.wd_codes = L->wd_codes; g.ld_wd = L->ld_wd; g.wd_scale = L->wd_scale;
  g.M = M; g.K = K; g.N = N;
  g.bits = b; g.n_groups = G;
  g.y = L->y;   g.ld_y = N;
  g.dx = L->dx; g.ld_dx = K;
  g.dw = L->dw; g.ld_dw = N;
  return shiftquant_gemm_layer(&g, L->workspace, L->workspace_bytes, L->dev_status, s);
}

// one host<->device copy of n floats, skipped when the host pointer is NULL
static int copy(void* dst, const void* src, int64_t n, cudaMemcpyKind kind, cudaStream_t s) {
  if (src == nullptr || dst == nullptr || n == 0) return SQ_OK;
  const cudaError_t err = cudaMemcpyAsync(dst, src, static_cast<size_t>(n) * sizeof(float), kind, s);
  return err == cudaSuccess ? SQ_OK : cuda_fail(err, "cudaMemcpyAsync");
}

}  // namespace sq

using namespace sq;

extern "C" sq_status shiftquant_layer_step(const sq_layer_step* args, uint64_t seed, void* stream) {
  fail(SQ_OK, "");
  int st = check_step(args);
  if (st != SQ_OK || args->M == 0 || args->K == 0 || args->N == 0) return st;
  return run_step(args, seed, stream);
}

extern "C" sq_status shiftquant_layer_step_host(const sq_layer_step* args, const float* x_host,
                                                const float* w_host, const float* dy_host,
                                                float* y_host, float* dx_host, float* dw_host,
                                                uint64_t seed, void* inputs_queued,
                                                void* stream) {
  fail(SQ_OK, "");
  int st = check_step(args);
  if (st != SQ_OK || args->M == 0 || args->K == 0 || args->N == 0) return st;
  const int64_t M = args->M, K = args->K, N = args->N;
  cudaStream_t s = as_stream(stream);
  if ((st = copy(args->x, x_host, M * K, cudaMemcpyHostToDevice, s)) != SQ_OK) return st;
  if ((st = copy(args->w, w_host, K * N, cudaMemcpyHostToDevice, s)) != SQ_OK) return st;
  if ((st = copy(args->dy, dy_host, M * N, cudaMemcpyHostToDevice, s)) != SQ_OK) return st;
  if (inputs_queued != nullptr) {
    const cudaError_t err = cudaEventRecord(static_cast<cudaEvent_t>(inputs_queued), s);
    if (err != cudaSuccess) return cuda_fail(err, "cudaEventRecord");
  }
  if ((st = run_step(args, seed, stream)) != SQ_OK) return st;
  if ((st = copy(y_host, args->y, M * N, cudaMemcpyDeviceToHost, s)) != SQ_OK) return st;
  if ((st = copy(dx_host, args->dx, M * K, cudaMemcpyDeviceToHost, s)) != SQ_OK) return st;
  return copy(dw_host, args->dw, K * N, cudaMemcpyDeviceToHost, s);
}

extern "C" sq_status shiftquant_layer_step_host_split(const sq_layer_step* args, const float* x_host,
                                                      const float* w_host, const float* dy_host,
                                                      float* y_host, float* dx_host, float* dw_host,
                                                      uint64_t seed, void* copy_in_stream,
                                                      void* stream, void* copy_out_stream,
                                                      void* buffers_free, void* inputs_in,
                                                      void* step_done, void* outputs_out) {
  fail(SQ_OK, "");
  int st = check_step(args);
  if (st != SQ_OK) return st;
  if (inputs_in == nullptr || step_done == nullptr || outputs_out == nullptr)
    return fail(SQ_EINVAL, "layer_step_host_split: inputs_in, step_done and outputs_out are required");
  const int64_t M = args->M, K = args->K, N = args->N;
  const bool empty = M == 0 || K == 0 || N == 0;
  cudaStream_t si = as_stream(copy_in_stream), sc = as_stream(stream), so = as_stream(copy_out_stream);
  cudaEvent_t ev_in = static_cast<cudaEvent_t>(inputs_in);
  cudaEvent_t ev_done = static_cast<cudaEvent_t>(step_done);
  cudaEvent_t ev_out = static_cast<cudaEvent_t>(outputs_out);
  cudaError_t err;
  if (buffers_free != nullptr &&
      (err = cudaStreamWaitEvent(si, static_cast<cudaEvent_t>(buffers_free), 0)) != cudaSuccess)
    return cuda_fail(err, "cudaStreamWaitEvent");
  if (!empty) {
    if ((st = copy(args->x, x_host, M * K, cudaMemcpyHostToDevice, si)) != SQ_OK) return st;
    if ((st = copy(args->w, w_host, K * N, cudaMemcpyHostToDevice, si)) != SQ_OK) return st;
    if ((st = copy(args->dy, dy_host, M * N, cudaMemcpyHostToDevice, si)) != SQ_OK) return st;
  }
  if ((err = cudaEventRecord(ev_in, si)) != cudaSuccess) return cuda_fail(err, "cudaEventRecord");
  if ((err = cudaStreamWaitEvent(sc, ev_in, 0)) != cudaSuccess) return cuda_fail(err, "cudaStreamWaitEvent");
  if (!empty && (st = run_step(args, seed, stream)) != SQ_OK) return st;
  if ((err = cudaEventRecord(ev_done, sc)) != cudaSuccess) return cuda_fail(err, "cudaEventRecord");
  if ((err = cudaStreamWaitEvent(so, ev_done, 0)) != cudaSuccess)
    return cuda_fail(err, "cudaStreamWaitEvent");
  if (!empty) {
    if ((st = copy(y_host, args->y, M * N, cudaMemcpyDeviceToHost, so)) != SQ_OK) return st;
    if ((st = copy(dx_host, args->dx, M * K, cudaMemcpyDeviceToHost, so)) != SQ_OK) return st;
    if ((st = copy(dw_host, args->dw, K * N, cudaMemcpyDeviceToHost, so)) != SQ_OK) return st;
  }
  if ((err = cudaEventRecord(ev_out, so)) != cudaSuccess) return cuda_fail(err, "cudaEventRecord");
  return SQ_OK;
}
