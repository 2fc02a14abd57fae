// Weighted combine / unpermute (§3.4: the layer output is the g_norm-weighted sum of the activated
// experts' outputs) and the expert-account update (§3.2).
//
//  combine_kernel: one block per token.  For each of the token's k_t slots it sums the expert
//      output partials (split-K slices, fixed order), accumulates g_norm * o into y in the order
//      j = 0..k_t-1, adds the always-on shared experts with weight 1, and reduces ||o||_2 of every
//      slot (the unweighted expert output that feeds C_s).
//  account_kernel: one block per expert.  Sums p and ||o||_2 over the expert's slots (tokens
//      ascending, a fixed tree) in fp64 and applies N += n_e, P_total += sum p,
//      C_s <- (1 - alpha) C_s + alpha * mean ||o||_2 when n_e > 0.
#include "eat_internal.cuh"

namespace eat {

namespace {

constexpr int kCombThreads = 256;
constexpr int kAccThreads = 128;

__device__ __forceinline__ void store_y(float* y, size_t i, float v) { y[i] = v; }
__device__ __forceinline__ void store_y(__nv_bfloat16* y, size_t i, float v) {
  y[i] = __float2bfloat16_rn(v);
}

template <typename TY>
__global__ void __launch_bounds__(kCombThreads)
combine_kernel(const float* __restrict__ opart, int n_split, size_t split_stride,
               const int32_t* __restrict__ slot_of, const float* __restrict__ w,
               const int32_t* __restrict__ kk, const float* __restrict__ sout, int S, int T, int K,
               int d, TY* __restrict__ y, float* __restrict__ onorm) {
  __shared__ int slots[kMaxK];
  __shared__ float gw[kMaxK];
  __shared__ float red[kCombThreads / 32][kMaxK];
  const int t = blockIdx.x;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int kt = kk[t];
  if (tid < K) {
    slots[tid] = tid < kt ? slot_of[(size_t)t * K + tid] : -1;
    gw[tid] = tid < kt ? w[(size_t)t * K + tid] : 0.f;
  }
  __syncthreads();
  float nrm[kMaxK];
#pragma unroll
  for (int j = 0; j < kMaxK; ++j) nrm[j] = 0.f;
  for (int c = tid; c < d; c += kCombThreads) {
    float acc = 0.f;
#pragma unroll
    for (int j = 0; j < kMaxK; ++j) {
      if (j < kt) {
        const size_t base = (size_t)slots[j] * d + c;
        float o = 0.f;
        for (int sp = 0; sp < n_split; ++sp) o += opart[sp * split_stride + base];
        acc = fmaf(gw[j], o, acc);
        nrm[j] = fmaf(o, o, nrm[j]);
      }
    }
    for (int s = 0; s < S; ++s) acc += sout[((size_t)s * T + t) * d + c];
    store_y(y, (size_t)t * d + c, acc);
  }
#pragma unroll
  for (int j = 0; j < kMaxK; ++j) {
    if (j < kt) {
      float v = nrm[j];
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
      if (lane == 0) red[warp][j] = v;
    }
  }
  __syncthreads();
  if (tid < kt) {
    float v = 0.f;
    for (int wi = 0; wi < kCombThreads / 32; ++wi) v += red[wi][tid];
    onorm[slots[tid]] = sqrtf(v);
  }
}

__global__ void __launch_bounds__(kAccThreads)
account_kernel(const int32_t* __restrict__ offs, const float* __restrict__ perm_p,
               const float* __restrict__ onorm, double alpha, int64_t* __restrict__ N,
               double* __restrict__ P, double* __restrict__ C, int32_t* __restrict__ st_n,
               double* __restrict__ st_p, double* __restrict__ st_norm,
               unsigned long long* __restrict__ counters) {
  __shared__ double rp[kAccThreads / 32], rn[kAccThreads / 32];
  const int e = blockIdx.x;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int beg = offs[e], end = offs[e + 1];
  double sp = 0.0, sn = 0.0;
  for (int i = beg + tid; i < end; i += kAccThreads) {
    sp += (double)perm_p[i];
    sn += (double)onorm[i];
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    sp += __shfl_xor_sync(0xffffffffu, sp, o);
    sn += __shfl_xor_sync(0xffffffffu, sn, o);
  }
  if (lane == 0) { rp[warp] = sp; rn[warp] = sn; }
  __syncthreads();
  if (tid == 0) {
    double a = 0.0, b = 0.0;
    for (int wi = 0; wi < kAccThreads / 32; ++wi) { a += rp[wi]; b += rn[wi]; }
    const int n = end - beg;
    N[e] += n;
    P[e] += a;
    if (n > 0) C[e] = (1.0 - alpha) * C[e] + alpha * (b / (double)n);
    st_n[e] = n;
    st_p[e] = a;
    st_norm[e] = b;
    if (n > 0) atomicAdd(&counters[1], 1ull);
    atomicAdd(&counters[2], (unsigned long long)n);
    if (e == 0) atomicAdd(&counters[0], 1ull);
  }
}

}  // namespace

cudaError_t launch_combine(int y_bf16, const float* opart, int n_split, int split_stride_rows,
                           const int32_t* slot_of, const float* w, const int32_t* k,
                           const float* sout, int S, int T, int K, int d, void* y, float* onorm,
                           cudaStream_t st) {
  const size_t stride = (size_t)split_stride_rows * d;
  if (y_bf16)
    combine_kernel<__nv_bfloat16><<<T, kCombThreads, 0, st>>>(
        opart, n_split, stride, slot_of, w, k, sout, S, T, K, d, (__nv_bfloat16*)y, onorm);
  else
    combine_kernel<float><<<T, kCombThreads, 0, st>>>(opart, n_split, stride, slot_of, w, k,
                                                       sout, S, T, K, d, (float*)y, onorm);
  return cudaGetLastError();
}

cudaError_t launch_account(const int32_t* offs, const float* perm_p, const float* onorm, int E,
                           double alpha, int64_t* N, double* P, double* C, int32_t* st_n,
                           double* st_p, double* st_norm, long long* counters, cudaStream_t st) {
  account_kernel<<<E, kAccThreads, 0, st>>>(offs, perm_p, onorm, alpha, N, P, C, st_n, st_p,
                                            st_norm, (unsigned long long*)counters);
  return cudaGetLastError();
}

}  // namespace eat
