// eat_route_noalloc: the routing call (router scores, softmax, history score, adaptive threshold,
// variable-k selection, renormalised gates) for callers that cannot allocate device memory.
//
// Some callers cannot call cudaMalloc at all: a serving process that has reserved nearly all of
// HBM for its own memory pool up front (where a fresh cudaMalloc fails or fragments the pool),
// a latency-critical decode loop that must not pay cudaMalloc's implicit device synchronisation,
// or a host framework whose rules route every device allocation through its own allocator.  They
// cannot create an eat_handle (eat_create allocates the accounts and the workspace).  This entry
// point takes every input and output from the caller and keeps its only scratch -- the partial
// router scores, as compensated fp32 pairs -- in a fixed array compiled into the library below.
#include "eat_internal.cuh"

#include <cuda.h>
#include <cudaTypedefs.h>

#include <mutex>
#include <string>

namespace {

// Scratch of the partial router scores: [split][T][E] compensated fp32 pairs (hi, lo) of 8 bytes
// each, 131072 pairs in all.  Every GPU that loads the library holds these 1 MiB until the process
// exits.  Calls share the array and it keeps the previous call's contents; nothing in it needs to
// start at zero (the scores kernel writes every entry it later reads).  Two calls that overlap on
// the GPU (different streams, or threads) race on it.
constexpr size_t kScratchScores = EAT_NOALLOC_SCRATCH_BYTES / sizeof(float2);
static __device__ __align__(256) float2 g_route_scratch[kScratchScores];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
// Per device: the scratch's device address and the unique id of the context it was looked up in.
struct Cached {
  unsigned long long ctx_id = 0;
  void* ptr = nullptr;
};
Cached g_scratch[kMaxDevices];

// Unique id of the context current on this thread (driver entry points fetched through the
// runtime, so the library needs no link against the driver library); false if there is none or
// the driver cannot tell.
bool current_context_id(unsigned long long* id) {
  static PFN_cuCtxGetCurrent_v4000 get_cur = nullptr;
  static PFN_cuCtxGetId_v12000 get_id = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 4000, cudaEnableDefault, &q) ==
            cudaSuccess && q == cudaDriverEntryPointSuccess)
      get_cur = (PFN_cuCtxGetCurrent_v4000)p;
    p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess && q == cudaDriverEntryPointSuccess)
      get_id = (PFN_cuCtxGetId_v12000)p;
  });
  CUcontext c = nullptr;
  if (!get_cur || !get_id || get_cur(&c) != CUDA_SUCCESS || !c) return false;
  return get_id(c, id) == CUDA_SUCCESS;
}

// Device address of the scratch in the current device's current context.  In host code
// g_route_scratch names a host-side stand-in, not device memory, so only this address may be
// handed to a kernel.  It is looked up once per device, with that device current, and again
// whenever the device's current context is another one than at the last look-up (after
// cudaDeviceReset the module is loaded anew and the array may move).
eat_status scratch_address(float2** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) {
    eat::set_thread_error((std::string("cudaGetDevice: ") + cudaGetErrorString(e)).c_str());
    return EAT_ERR_CUDA;
  }
  if (dev < 0 || dev >= kMaxDevices) {
    eat::set_thread_error("device index beyond the 64 devices eat_route_noalloc supports");
    return EAT_ERR_UNSUPPORTED;
  }
  std::lock_guard<std::mutex> lock(g_mu);
  unsigned long long id = 0;
  if (g_scratch[dev].ptr && current_context_id(&id) && id == g_scratch[dev].ctx_id) {
    *out = (float2*)g_scratch[dev].ptr;
    return EAT_OK;
  }
  void* p = nullptr;
  e = cudaGetSymbolAddress(&p, g_route_scratch);
  if (e != cudaSuccess || !p) {
    eat::set_thread_error((std::string("cudaGetSymbolAddress of the routing scratch: ") +
                           cudaGetErrorString(e)).c_str());
    return EAT_ERR_CUDA;
  }
  // the look-up made the device's primary context current if none was; a context the driver
  // cannot identify is not cached (then every call looks the address up)
  if (current_context_id(&id)) g_scratch[dev] = {id, p};
  else g_scratch[dev] = {};
  *out = (float2*)p;
  return EAT_OK;
}

eat_status bad(const char* msg) {
  eat::set_thread_error(msg);
  return EAT_ERR_INVALID_ARG;
}

}  // namespace

extern "C" eat_status eat_route_noalloc(const void* x, int32_t T, int32_t d_model,
                                        int32_t n_experts, int32_t xdtype, const float* w_router,
                                        const float* b_router, const int64_t* N, const double* P,
                                        const double* C, const eat_params* params,
                                        int32_t ppl_sign, int32_t* idx, float* w, int32_t* k,
                                        void* stream) {
  if (!x || !w_router || !N || !P || !C || !params || !idx || !w || !k)
    return bad("eat_route_noalloc: a required pointer is NULL");
  if (T < 1 || d_model < 1) return bad("eat_route_noalloc: T and d_model must be >= 1");
  if (n_experts < 1 || n_experts > eat::kMaxExperts)
    return bad("eat_route_noalloc: n_experts must be in [1, 256]");
  if (xdtype != EAT_F32 && xdtype != EAT_BF16)
    return bad("eat_route_noalloc: xdtype must be EAT_F32 or EAT_BF16");
  if (ppl_sign < -1 || ppl_sign > 1) return bad("eat_route_noalloc: ppl_sign must be -1, 0, +1");
  const eat_params& p = *params;
  if (p.max_k < 1 || p.max_k > eat::kMaxK || p.max_k > n_experts)
    return bad("eat_route_noalloc: max_k must be in [1, min(E, 16)]");
  if (!(p.temperature > 0.0)) return bad("eat_route_noalloc: temperature <= 0");
  if (!(p.q_lo >= 0.0 && p.q_lo <= p.q_hi && p.q_hi <= 1.0))
    return bad("eat_route_noalloc: need 0 <= q_lo <= q_hi <= 1");
  if (p.c_mode != EAT_C_SUM && p.c_mode != EAT_C_RAW) return bad("eat_route_noalloc: bad c_mode");
  if (p.router_mode < EAT_ROUTER_EAT || p.router_mode > EAT_ROUTER_TOPP ||
      (p.router_mode == EAT_ROUTER_TOPP && !(p.top_p > 0.0 && p.top_p <= 1.0)))
    return bad("eat_route_noalloc: bad router_mode or top_p");
  if ((size_t)T * (size_t)n_experts > kScratchScores)
    return bad("eat_route_noalloc: T * n_experts exceeds the 131072 router scores its fixed "
               "1 MiB scratch holds; split the call into smaller token batches");

  float2* scratch = nullptr;
  const eat_status s = scratch_address(&scratch);
  if (s != EAT_OK) return s;

  int split = eat::router_split(T, d_model, n_experts);
  while (split > 1 && (size_t)split * T * n_experts > kScratchScores) split /= 2;

  eat::RouteParams rp;
  rp.w1 = (float)p.w1;
  rp.w2 = (float)p.w2;
  rp.w3 = (float)p.w3;
  rp.beta = (float)p.beta;
  rp.alpha1 = (float)p.alpha1;
  rp.alpha2 = (float)p.alpha2;
  rp.kappa1 = (float)p.kappa1;
  rp.kappa2 = (float)p.kappa2;
  rp.ppl_factor = ppl_sign > 0 ? (float)p.ppl_up : (ppl_sign < 0 ? (float)p.ppl_down : 1.0f);
  rp.q_lo = (float)p.q_lo;
  rp.q_hi = (float)p.q_hi;
  rp.eps = (float)p.eps;
  rp.temperature = (float)p.temperature;
  rp.clamp = p.clamp_enabled;
  rp.c_mode = p.c_mode;
  rp.mode = p.router_mode;
  rp.top_p = (float)p.top_p;
  rp.smoothing = EAT_SMOOTH_CALL;  // no per-stream state without a handle
  rp.opd_scale = nullptr;
  rp.tau_in = nullptr;
  rp.tau_out = nullptr;
  rp.ppl_sign_dev = nullptr;
  rp.ppl_up = (float)p.ppl_up;
  rp.ppl_down = (float)p.ppl_down;

  cudaStream_t st = (cudaStream_t)stream;
  cudaError_t e = eat::launch_router_logits(x, xdtype == EAT_BF16, w_router, T, d_model,
                                            n_experts, split, scratch, st);
  if (e == cudaSuccess)
    e = eat::launch_route_select(scratch, split, b_router, T, n_experts, p.max_k, N, P, C, rp,
                                 idx, w, k, nullptr, st);
  if (e != cudaSuccess) {
    eat::set_thread_error((std::string("eat_route_noalloc launch: ") + cudaGetErrorString(e))
                              .c_str());
    return EAT_ERR_CUDA;
  }
  return EAT_OK;
}
