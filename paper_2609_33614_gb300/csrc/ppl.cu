// The perplexity signal of §3.3's performance-based adjustment, computed on the device from the
// model's token negative log-likelihoods, and the layer-wise policy of §5.2 as parameters.
//
//  ppl_update_kernel: one block.  PPL_curr = exp(mean NLL over the window's n tokens) in fp64 (the
//      fp32 likelihoods summed in fp64, each thread over a fixed stride, then a fixed tree), the
//      sign of PPL_curr - PPL_prev (+1 when it is > 0, -1 otherwise, 0 without a previous value
//      or for a NaN perplexity) written to the device, and PPL_curr stored as the next window's
//      PPL_prev.  A layer handle attached to the sign (eat_set_ppl_sign_source) reads it inside its
//      selection kernel, so a model loop feeds the adjustment without a host synchronisation.
#include "eat_internal.cuh"

#include <string>

namespace eat {

namespace {

constexpr int kPplThreads = 256;

__global__ void __launch_bounds__(kPplThreads)
ppl_update_kernel(const float* __restrict__ nll, int n, double* __restrict__ state,
                  int32_t* __restrict__ sign) {
  __shared__ double red[kPplThreads];
  pdl_wait();
  pdl_launch_dependents();
  double acc = 0.0;
  for (int i = threadIdx.x; i < n; i += kPplThreads) acc += (double)nll[i];
  red[threadIdx.x] = acc;
  __syncthreads();
#pragma unroll
  for (int w = kPplThreads / 2; w > 0; w >>= 1) {
    if (threadIdx.x < w) red[threadIdx.x] += red[threadIdx.x + w];
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    const double curr = exp(red[0] / (double)n);
    const double prev = *state;
    int32_t s = 0;
    if (!isnan(prev) && !isnan(curr)) s = curr - prev > 0.0 ? 1 : -1;
    *sign = s;
    *state = curr;
  }
}

}  // namespace

cudaError_t launch_ppl_update(const float* nll, int n, double* state, int32_t* sign,
                              cudaStream_t st) {
  return launch_pdl(ppl_update_kernel, dim3(1), dim3(kPplThreads), 0, st, nll, n, state, sign);
}

}  // namespace eat

extern "C" eat_status eat_ppl_update(const float* nll, int32_t n, double* ppl_state,
                                     int32_t* sign, void* stream) {
  if (!nll || !ppl_state || !sign) {
    eat::set_thread_error("eat_ppl_update: nll, ppl_state and sign must be non-NULL");
    return EAT_ERR_INVALID_ARG;
  }
  if (n < 1) {
    eat::set_thread_error("eat_ppl_update: the window needs at least one token (n >= 1)");
    return EAT_ERR_INVALID_ARG;
  }
  if (((uintptr_t)ppl_state & 7) != 0 || ((uintptr_t)sign & 3) != 0 || ((uintptr_t)nll & 3) != 0) {
    eat::set_thread_error("eat_ppl_update: misaligned pointer");
    return EAT_ERR_INVALID_ARG;
  }
  const cudaError_t e = eat::launch_ppl_update(nll, n, ppl_state, sign, (cudaStream_t)stream);
  if (e != cudaSuccess) {
    eat::set_thread_error((std::string("eat_ppl_update launch: ") + cudaGetErrorString(e)).c_str());
    return EAT_ERR_CUDA;
  }
  return EAT_OK;
}

extern "C" eat_status eat_layer_policy(int32_t layer, int32_t n_layers, eat_params* p) {
  if (!p || n_layers < 1 || layer < 0 || layer >= n_layers) {
    eat::set_thread_error("eat_layer_policy: need params and 0 <= layer < n_layers");
    return EAT_ERR_INVALID_ARG;
  }
  // §5.2: the lower three quarters of the stack (layers 0-23 of Mixtral's 32) tolerate far
  // sparser routing; the upper quarter keeps the full K
  if (layer < (3 * n_layers) / 4) {
    p->max_k = p->max_k / 3 > 1 ? p->max_k / 3 : 1;
    p->alpha1 = 2.0 * p->alpha1;
  }
  return EAT_OK;
}
