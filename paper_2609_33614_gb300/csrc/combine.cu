// Weighted combine / unpermute (§3.4: the layer output is the g_norm-weighted sum of the activated
// experts' outputs) and the expert-account update (§3.2).
//
//  combine_kernel: one block per (token, 1024-column block).  For each of the token's k_t slots
//      it sums the expert output partials (split-K slices, fixed order), accumulates g_norm * o into
//      y in the order j = 0..k_t-1, adds the always-on shared experts with weight 1, and writes the
//      partial sum of squares of every slot (||o||_2 of the unweighted expert output feeds C_s).
//  account_kernel: one block per expert.  Finishes ||o||_2 of each slot from the column-block
//      partials, sums p and ||o||_2 over the expert's slots (tokens ascending, a fixed tree) in
//      fp64 and applies N += n_e, P_total += sum p,
//      C_s <- (1 - alpha) C_s + alpha * mean ||o||_2 when n_e > 0.
#include "eat_internal.cuh"

namespace eat {

namespace {

constexpr int kCombThreads = 256;
constexpr int kAccThreads = 128;

__device__ __forceinline__ void store_y4(float* y, float4 v) { *(float4*)y = v; }
__device__ __forceinline__ void store_y4(__nv_bfloat16* y, float4 v) {
  __nv_bfloat162 a = __floats2bfloat162_rn(v.x, v.y);
  __nv_bfloat162 b = __floats2bfloat162_rn(v.z, v.w);
  uint2 u;
  u.x = *(uint32_t*)&a;
  u.y = *(uint32_t*)&b;
  *(uint2*)y = u;
}

// Column block of one token: 4 consecutive columns per thread (float4 loads), so a token's row
// is spread over ceil(d / 1024) blocks; every block writes the partial sum of squares of each of
// the token's slots over its columns (nrm_part[slot][block]), which the account kernel sums.
template <typename TY>
__global__ void __launch_bounds__(kCombThreads)
combine_kernel(const float* __restrict__ opart, int n_split, size_t split_stride,
               const int32_t* __restrict__ slot_of, const float* __restrict__ w,
               const int32_t* __restrict__ kk, const float* __restrict__ sout, int S, int T, int K,
               int d, TY* __restrict__ y, float* __restrict__ nrm_part) {
  __shared__ int slots[kMaxK];
  __shared__ float gw[kMaxK];
  __shared__ float red[kCombThreads / 32][kMaxK];
  pdl_wait();
  pdl_launch_dependents();
  const int t = blockIdx.x;
  const int nb = gridDim.y, cb = blockIdx.y;
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
  const int c = (cb * kCombThreads + tid) * 4;
  if (c < d) {
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int j = 0; j < kMaxK; ++j) {
      if (j < kt) {
        const float* src = opart + (size_t)slots[j] * d + c;
        float4 o = *(const float4*)src;
        for (int sp = 1; sp < n_split; ++sp) {
          const float4 q = *(const float4*)(src + sp * split_stride);
          o.x += q.x;
          o.y += q.y;
          o.z += q.z;
          o.w += q.w;
        }
        const float g = gw[j];
        acc.x = fmaf(g, o.x, acc.x);
        acc.y = fmaf(g, o.y, acc.y);
        acc.z = fmaf(g, o.z, acc.z);
        acc.w = fmaf(g, o.w, acc.w);
        nrm[j] = fmaf(o.x, o.x, fmaf(o.y, o.y, fmaf(o.z, o.z, fmaf(o.w, o.w, nrm[j]))));
      }
    }
    for (int s = 0; s < S; ++s) {
      const float4 q = *(const float4*)(sout + ((size_t)s * T + t) * d + c);
      acc.x += q.x;
      acc.y += q.y;
      acc.z += q.z;
      acc.w += q.w;
    }
    store_y4(y + (size_t)t * d + c, acc);
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
    nrm_part[(size_t)slots[tid] * nb + cb] = v;
  }
}

__global__ void __launch_bounds__(kAccThreads)
account_kernel(const int32_t* __restrict__ offs, const float* __restrict__ perm_p,
               const float* __restrict__ nrm_part, int nb, double alpha, int64_t* __restrict__ N,
               double* __restrict__ P, double* __restrict__ C, int32_t* __restrict__ st_n,
               double* __restrict__ st_p, double* __restrict__ st_norm,
               unsigned long long* __restrict__ counters) {
  __shared__ double rp[kAccThreads / 32], rn[kAccThreads / 32];
  pdl_wait();
  pdl_launch_dependents();
  const int e = blockIdx.x;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int beg = offs[e], end = offs[e + 1];
  double sp = 0.0, sn = 0.0;
  for (int i = beg + tid; i < end; i += kAccThreads) {
    sp += (double)perm_p[i];
    double sq = 0.0;
    for (int b = 0; b < nb; ++b) sq += (double)nrm_part[(size_t)i * nb + b];
    sn += sqrt(sq);
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

int combine_col_blocks(int d) { return (d + 4 * kCombThreads - 1) / (4 * kCombThreads); }

cudaError_t launch_combine(int y_bf16, const float* opart, int n_split, int split_stride_rows,
                           const int32_t* slot_of, const float* w, const int32_t* k,
                           const float* sout, int S, int T, int K, int d, void* y,
                           float* nrm_part, cudaStream_t st) {
  const size_t stride = (size_t)split_stride_rows * d;
  dim3 grid(T, combine_col_blocks(d));
  if (y_bf16)
    return launch_pdl(combine_kernel<__nv_bfloat16>, grid, dim3(kCombThreads), 0, st, opart,
                      n_split, stride, slot_of, w, k, sout, S, T, K, d, (__nv_bfloat16*)y,
                      nrm_part);
  return launch_pdl(combine_kernel<float>, grid, dim3(kCombThreads), 0, st, opart, n_split,
                    stride, slot_of, w, k, sout, S, T, K, d, (float*)y, nrm_part);
}

cudaError_t launch_account(const int32_t* offs, const float* perm_p, const float* nrm_part, int nb,
                           int E, double alpha, int64_t* N, double* P, double* C, int32_t* st_n,
                           double* st_p, double* st_norm, long long* counters, cudaStream_t st) {
  return launch_pdl(account_kernel, dim3(E), dim3(kAccThreads), 0, st, offs, perm_p, nrm_part,
                    nb, alpha, N, P, C, st_n, st_p, st_norm, (unsigned long long*)counters);
}

}  // namespace eat
