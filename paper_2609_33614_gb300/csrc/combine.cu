// Weighted combine / unpermute (§3.4: the layer output is the g_norm-weighted sum of the activated
// experts' outputs) and the expert-account update (§3.2).
//
//  combine_kernel: one block per (token, 2048-column block).  For each of the token's k_t slots
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
constexpr int kAccThreads = 512;


// 8 consecutive values as fp32, from fp32 (two 16-byte loads) or bf16 (one 16-byte load).
struct V8 {
  float v[8];
};
__device__ __forceinline__ V8 load8(const void* base, bool bf16, size_t i) {
  V8 r;
  if (bf16) {
    const uint4 u = *(const uint4*)((const __nv_bfloat16*)base + i);
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float2 f = __bfloat1622float2(*(const __nv_bfloat162*)&w[q]);
      r.v[2 * q] = f.x;
      r.v[2 * q + 1] = f.y;
    }
  } else {
    const float4 a = *(const float4*)((const float*)base + i);
    const float4 b = *(const float4*)((const float*)base + i + 4);
    r.v[0] = a.x; r.v[1] = a.y; r.v[2] = a.z; r.v[3] = a.w;
    r.v[4] = b.x; r.v[5] = b.y; r.v[6] = b.z; r.v[7] = b.w;
  }
  return r;
}
__device__ __forceinline__ void store8(float* y, const float (&a)[8]) {
  *(float4*)y = make_float4(a[0], a[1], a[2], a[3]);
  *(float4*)(y + 4) = make_float4(a[4], a[5], a[6], a[7]);
}
__device__ __forceinline__ void store8(__nv_bfloat16* y, const float (&a)[8]) {
  uint4 u;
  uint32_t* w = (uint32_t*)&u;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const __nv_bfloat162 h = __floats2bfloat162_rn(a[2 * q], a[2 * q + 1]);
    w[q] = *(const uint32_t*)&h;
  }
  *(uint4*)y = u;
}

// Column block of one token: 8 consecutive columns per thread (16-byte loads), so a token's row
// spans ceil(d / 2048) blocks; every block writes the partial sum of squares of each of the
// token's slots over its columns (nrm_part[slot][block]), which the account kernel sums.  Expert
// outputs are fp32 split-K partials (o_bf16 = 0) or, without split-K, bf16 rows; the shared
// experts' outputs likewise (s_bf16).  All of a token's slot rows are loaded before any use.
template <typename TY, int KM>
__global__ void __launch_bounds__(kCombThreads)
combine_kernel(const void* __restrict__ opart, int o_bf16, int n_split, size_t split_stride,
               const int32_t* __restrict__ slot_of, const float* __restrict__ w,
               const int32_t* __restrict__ kk, const void* __restrict__ sout, int s_bf16, int S,
               int T, int K, int d, TY* __restrict__ y, float* __restrict__ nrm_part) {
  __shared__ int slots[KM];
  __shared__ float gw[KM];
  __shared__ float red[kCombThreads / 32][KM];
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
  float nrm[KM];
#pragma unroll
  for (int j = 0; j < KM; ++j) nrm[j] = 0.f;
  const int c = (cb * kCombThreads + tid) * 8;
  if (c < d) {
    V8 o[KM];
#pragma unroll
    for (int j = 0; j < KM; ++j)
      if (j < kt) o[j] = load8(opart, o_bf16, (size_t)slots[j] * d + c);
    for (int sp = 1; sp < n_split; ++sp) {
#pragma unroll
      for (int j = 0; j < KM; ++j) {
        if (j < kt) {
          const V8 q = load8(opart, false, sp * split_stride + (size_t)slots[j] * d + c);
#pragma unroll
          for (int i = 0; i < 8; ++i) o[j].v[i] += q.v[i];
        }
      }
    }
    float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int j = 0; j < KM; ++j) {
      if (j < kt) {
        const float g = gw[j];
        float n = 0.f;
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          acc[i] = fmaf(g, o[j].v[i], acc[i]);
          n = fmaf(o[j].v[i], o[j].v[i], n);
        }
        nrm[j] = n;
      }
    }
    for (int s = 0; s < S; ++s) {
      const V8 q = load8(sout, s_bf16, ((size_t)s * T + t) * d + c);
#pragma unroll
      for (int i = 0; i < 8; ++i) acc[i] += q.v[i];
    }
    store8(y + (size_t)t * d + c, acc);
  }
#pragma unroll
  for (int j = 0; j < KM; ++j) {
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
  // four independent slot streams per thread keep enough loads in flight for an expert that
  // holds most of a large call's tokens
  double sp4[4] = {0.0, 0.0, 0.0, 0.0}, sn4[4] = {0.0, 0.0, 0.0, 0.0};
  for (int i0 = beg + tid; i0 < end; i0 += 4 * kAccThreads) {
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int i = i0 + u * kAccThreads;
      if (i < end) {
        sp4[u] += (double)perm_p[i];
        double sq = 0.0;
        for (int b = 0; b < nb; ++b) sq += (double)nrm_part[(size_t)i * nb + b];
        sn4[u] += sqrt(sq);
      }
    }
  }
  double sp = (sp4[0] + sp4[1]) + (sp4[2] + sp4[3]);
  double sn = (sn4[0] + sn4[1]) + (sn4[2] + sn4[3]);
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

int combine_col_blocks(int d) { return (d + 8 * kCombThreads - 1) / (8 * kCombThreads); }

namespace {

template <typename TY, int KM>
cudaError_t launch_combine_t(dim3 grid, cudaStream_t st, const void* opart, int o_bf16,
                             int n_split, size_t stride, const int32_t* slot_of, const float* w,
                             const int32_t* k, const void* sout, int s_bf16, int S, int T, int K,
                             int d, void* y, float* nrm_part) {
  return launch_pdl(combine_kernel<TY, KM>, grid, dim3(kCombThreads), 0, st, opart, o_bf16,
                    n_split, stride, slot_of, w, k, sout, s_bf16, S, T, K, d, (TY*)y, nrm_part);
}

template <typename TY>
cudaError_t launch_combine_k(dim3 grid, cudaStream_t st, const void* opart, int o_bf16,
                             int n_split, size_t stride, const int32_t* slot_of, const float* w,
                             const int32_t* k, const void* sout, int s_bf16, int S, int T, int K,
                             int d, void* y, float* nrm_part) {
#define EAT_COMB(KM)                                                                            \
  launch_combine_t<TY, KM>(grid, st, opart, o_bf16, n_split, stride, slot_of, w, k, sout, s_bf16, \
                           S, T, K, d, y, nrm_part)
  if (K <= 2) return EAT_COMB(2);
  if (K <= 4) return EAT_COMB(4);
  if (K <= 8) return EAT_COMB(8);
  return EAT_COMB(16);
#undef EAT_COMB
}

}  // namespace

cudaError_t launch_combine(int y_bf16, const void* opart, int o_bf16, int n_split,
                           int split_stride_rows, const int32_t* slot_of, const float* w,
                           const int32_t* k, const void* sout, int s_bf16, int S, int T, int K,
                           int d, void* y, float* nrm_part, cudaStream_t st) {
  const size_t stride = (size_t)split_stride_rows * d;
  dim3 grid(T, combine_col_blocks(d));
  if (y_bf16)
    return launch_combine_k<__nv_bfloat16>(grid, st, opart, o_bf16, n_split, stride, slot_of, w,
                                           k, sout, s_bf16, S, T, K, d, y, nrm_part);
  return launch_combine_k<float>(grid, st, opart, o_bf16, n_split, stride, slot_of, w, k, sout,
                                 s_bf16, S, T, K, d, y, nrm_part);
}

cudaError_t launch_account(const int32_t* offs, const float* perm_p, const float* nrm_part, int nb,
                           int E, double alpha, int64_t* N, double* P, double* C, int32_t* st_n,
                           double* st_p, double* st_norm, long long* counters, cudaStream_t st) {
  return launch_pdl(account_kernel, dim3(E), dim3(kAccThreads), 0, st, offs, perm_p, nrm_part,
                    nb, alpha, N, P, C, st_n, st_p, st_norm, (unsigned long long*)counters);
}

}  // namespace eat
