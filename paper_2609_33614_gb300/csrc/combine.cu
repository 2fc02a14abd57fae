// Weighted combine / unpermute (§3.4: the layer output is the g_norm-weighted sum of the activated
// experts' outputs) and the expert-account update (§3.2).
//
//  combine_kernel: one warp per (token, 256-column segment), 8 columns per lane, no shared memory
//      and no block barrier, so each warp's loads go out as soon as it starts.  For each of the
//      token's k_t slots it sums the expert output partials (split-K slices, fixed order),
//      accumulates g_norm * o into y in the order j = 0..k_t-1, adds the always-on shared experts
//      with weight 1, and writes the segment's sum of squares of every slot (||o||_2 of the
//      unweighted expert output feeds C_s) to nrm_part[slot][segment].
//  account_kernel: blocks (e, c) over each expert's slots in chunks of 1024.  Finishes ||o||_2 of
//      each slot from its segment sums (fp32, fixed order), sums p and ||o||_2 over the chunk with
//      compensated fp32 additions (a fixed tree; about fp64 accuracy); an expert of one chunk is
//      finished by its block, a larger one by the last of its blocks to arrive (a ticket per
//      expert, reset by that block), which adds the chunks' compensated sums in chunk order.  The
//      finishing block applies, in fp64 on one thread, N += n_e, P_total += sum p and
//      C_s <- (1 - alpha) C_s + alpha * mean ||o||_2 when n_e > 0.  Per-slot work stays off
//      GB300's narrow fp64 pipe, and no block walks more than one chunk: one block per expert
//      left the most popular expert's block (~4000 slots at a 4096-token call) the longest of
//      the step.
//  Both read the device status word: when an earlier kernel of the call gave up on a bounded wait
//  (its outputs are then invalid), the combine writes NaN rows and the account update leaves N,
//  P_total and C_s as they were, so one expired wait cannot feed invalid norms into the accounts
//  that every later call routes by.  The block that finishes expert 0 copies the word to a
//  host-mapped mirror, which the entry points read without synchronising.
#include "eat_internal.cuh"

namespace eat {

namespace {

constexpr int kCombThreads = 256;  // 8 warps: 8 (token, segment) tasks per block
constexpr int kSegCols = 256;      // columns per warp task, 8 per lane
constexpr int kAccThreads = 256;
constexpr int kAccChunk = 4 * kAccThreads;  // slots of one account block

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

// Sum over the warp of v[0..N) (N a power of two <= 32), fixed order.  Each step exchanges half
// of the remaining values with the partner lane, so N sums take N - 1 + 5 - log2 N shuffles
// instead of 5 N.  On return every lane holds the total of value j = lane / (32 / N).
template <int N>
__device__ __forceinline__ float warp_sum_many(float (&v)[N], int lane) {
  const unsigned full = 0xffffffffu;
#pragma unroll
  for (int n = N, m = 16; n > 1; n >>= 1, m >>= 1) {
    const bool upper = (lane & m) != 0;
#pragma unroll
    for (int i = 0; i < n / 2; ++i) {
      const float send = upper ? v[i] : v[i + n / 2];
      const float keep = upper ? v[i + n / 2] : v[i];
      v[i] = keep + __shfl_xor_sync(full, send, m);
    }
  }
  float r = v[0];
#pragma unroll
  for (int m = 16 / N; m > 0; m >>= 1) r += __shfl_xor_sync(full, r, m);
  return r;
}

// Expert outputs are bf16 rows (OB, no split-K) or fp32 split-K partials; the shared experts'
// outputs bf16 (s_bf16) or fp32.  Slots past k_t are -1 with gate 0.  All of a token's slot rows
// are loaded before any use.  A token with no selected expert (k_t = 0, which only a NaN routing
// probability produces) gets a NaN row.
// (bf16 expert rows, the large calls: at most 64 registers, so four blocks share an SM and keep
// more row loads in flight)
template <typename TY, int KM, bool OB>
__global__ void __launch_bounds__(kCombThreads, OB ? 4 : 1)
combine_kernel(const void* __restrict__ opart, int n_split, size_t split_stride,
               const int32_t* __restrict__ slot_of, const float* __restrict__ w,
               const void* __restrict__ sout, int s_bf16, int S, int T, int K, int d, int nseg,
               TY* __restrict__ y, float* __restrict__ nrm_part,
               const unsigned int* __restrict__ status) {
  pdl_wait();
  pdl_launch_dependents();
  const unsigned full = 0xffffffffu;
  const int lane = threadIdx.x & 31;
  const int task = blockIdx.x * (kCombThreads / 32) + (threadIdx.x >> 5);
  if (task >= T * nseg) return;
  const int t = task / nseg, sg = task - t * nseg;
  int my_slot = -1;
  float my_w = 0.f;
  if (lane < K) {
    my_slot = slot_of[(size_t)t * K + lane];
    my_w = w[(size_t)t * K + lane];
  }
  int slots[KM];
  float g[KM];
#pragma unroll
  for (int j = 0; j < KM; ++j) {
    slots[j] = __shfl_sync(full, my_slot, j);
    g[j] = __shfl_sync(full, my_w, j);
  }
  const int c = sg * kSegCols + lane * 8;
  const bool in = c < d;
  float nrm[KM];
  float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  if constexpr (OB) {
    uint4 raw[KM];
#pragma unroll
    for (int j = 0; j < KM; ++j)
      if (in && slots[j] >= 0)
        raw[j] = *(const uint4*)((const __nv_bfloat16*)opart + (size_t)slots[j] * d + c);
#pragma unroll
    for (int j = 0; j < KM; ++j) {
      nrm[j] = 0.f;
      if (in && slots[j] >= 0) {
        const uint32_t wd[4] = {raw[j].x, raw[j].y, raw[j].z, raw[j].w};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const float2 f = __bfloat1622float2(*(const __nv_bfloat162*)&wd[q]);
          acc[2 * q] = fmaf(g[j], f.x, acc[2 * q]);
          acc[2 * q + 1] = fmaf(g[j], f.y, acc[2 * q + 1]);
          nrm[j] = fmaf(f.x, f.x, nrm[j]);
          nrm[j] = fmaf(f.y, f.y, nrm[j]);
        }
      }
    }
  } else {
    V8 o[KM];
#pragma unroll
    for (int j = 0; j < KM; ++j)
      if (in && slots[j] >= 0) o[j] = load8(opart, false, (size_t)slots[j] * d + c);
    for (int sp = 1; sp < n_split; ++sp) {
#pragma unroll
      for (int j = 0; j < KM; ++j) {
        if (in && slots[j] >= 0) {
          const V8 q = load8(opart, false, sp * split_stride + (size_t)slots[j] * d + c);
#pragma unroll
          for (int i = 0; i < 8; ++i) o[j].v[i] += q.v[i];
        }
      }
    }
#pragma unroll
    for (int j = 0; j < KM; ++j) {
      nrm[j] = 0.f;
      if (in && slots[j] >= 0) {
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          acc[i] = fmaf(g[j], o[j].v[i], acc[i]);
          nrm[j] = fmaf(o[j].v[i], o[j].v[i], nrm[j]);
        }
      }
    }
  }
  if (in) {
    for (int s = 0; s < S; ++s) {
      const V8 q = load8(sout, s_bf16, ((size_t)s * T + t) * d + c);
#pragma unroll
      for (int i = 0; i < 8; ++i) acc[i] += q.v[i];
    }
    // no expert selected (the token's routing was not finite), or an expert kernel of this call
    // gave up on a wait (its outputs are invalid): a NaN row
    if (slots[0] < 0 || __ldcg(status) != 0u) {
#pragma unroll
      for (int i = 0; i < 8; ++i) acc[i] = __int_as_float(0x7fc00000);
    }
    store8(y + (size_t)t * d + c, acc);
  }
  const float r = warp_sum_many<KM>(nrm, lane);
  const int jm = lane / (32 / KM);
  const int sm = __shfl_sync(full, my_slot, jm);
  if (lane % (32 / KM) == 0 && sm >= 0) nrm_part[(size_t)sm * nseg + sg] = r;
}

__global__ void __launch_bounds__(kAccThreads)
account_kernel(const int32_t* __restrict__ offs, const float* __restrict__ perm_p,
               const float* __restrict__ nrm_part, int nb, double alpha, int64_t* __restrict__ N,
               double* __restrict__ P, double* __restrict__ C, int32_t* __restrict__ st_n,
               double* __restrict__ st_p, double* __restrict__ st_norm,
               unsigned long long* __restrict__ counters, float4* __restrict__ chunk_sums,
               unsigned int* __restrict__ tickets, const unsigned int* __restrict__ status,
               unsigned int* __restrict__ status_mirror) {
  __shared__ float red[4][kAccThreads / 32];
  pdl_wait();
  pdl_launch_dependents();
  const int e = blockIdx.x, c = blockIdx.y;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int beg = offs[e], end = offs[e + 1];
  const int n = end - beg;
  const int n_chunks = n > 0 ? (n + kAccChunk - 1) / kAccChunk : 1;
  if (c >= n_chunks) return;
  const bool vec = (nb & 3) == 0;
  float p_hi = 0.f, p_lo = 0.f, n_hi = 0.f, n_lo = 0.f;
  {
    // four slots per thread, all loads issued before the sums
    const int i0 = beg + c * kAccChunk + tid;
    float pv[4], nv[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int i = i0 + u * kAccThreads;
      pv[u] = 0.f;
      nv[u] = 0.f;
      if (i < end) {
        pv[u] = perm_p[i];
        const float* np = nrm_part + (size_t)i * nb;
        float sq = 0.f;
        if (vec) {
          for (int b = 0; b < nb; b += 4) {
            const float4 q = *(const float4*)(np + b);
            sq += q.x;
            sq += q.y;
            sq += q.z;
            sq += q.w;
          }
        } else {
          for (int b = 0; b < nb; ++b) sq += np[b];
        }
        nv[u] = sq;
      }
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      df_add(p_hi, p_lo, pv[u]);
      df_add(n_hi, n_lo, sqrtf(nv[u]));
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float a = __shfl_xor_sync(0xffffffffu, p_hi, o);
    const float b = __shfl_xor_sync(0xffffffffu, p_lo, o);
    const float cc = __shfl_xor_sync(0xffffffffu, n_hi, o);
    const float dd = __shfl_xor_sync(0xffffffffu, n_lo, o);
    df_add(p_hi, p_lo, a, b);
    df_add(n_hi, n_lo, cc, dd);
  }
  if (lane == 0) {
    red[0][warp] = p_hi;
    red[1][warp] = p_lo;
    red[2][warp] = n_hi;
    red[3][warp] = n_lo;
  }
  __syncthreads();
  if (tid != 0) return;
  float ah = 0.f, al = 0.f, bh = 0.f, bl = 0.f;
  for (int wi = 0; wi < kAccThreads / 32; ++wi) {
    df_add(ah, al, red[0][wi], red[1][wi]);
    df_add(bh, bl, red[2][wi], red[3][wi]);
  }
  if (n_chunks > 1) {
    // publish this chunk's sums; the last block of the expert to arrive adds all chunks in order
    float4* cs = chunk_sums + (size_t)e * gridDim.y;
    cs[c] = make_float4(ah, al, bh, bl);
    __threadfence();
    if (atomicAdd(&tickets[e], 1u) != (unsigned)(n_chunks - 1)) return;
    __threadfence();
    tickets[e] = 0u;  // for the next call (which starts after this kernel has completed)
    ah = al = bh = bl = 0.f;
    for (int ci = 0; ci < n_chunks; ++ci) {
      const float4 v = __ldcg(cs + ci);
      df_add(ah, al, v.x, v.y);
      df_add(bh, bl, v.z, v.w);
    }
  }
  const double a = (double)ah + (double)al, b = (double)bh + (double)bl;
  const unsigned int sw = __ldcg(status);
  if (sw == 0u) {  // every kernel of the call completed its work
    N[e] += n;
    P[e] += a;
    if (n > 0) C[e] = (1.0 - alpha) * C[e] + alpha * (b / (double)n);
    if (n > 0) atomicAdd(&counters[1], 1ull);
    atomicAdd(&counters[2], (unsigned long long)n);
    if (e == 0) atomicAdd(&counters[0], 1ull);
  }
  st_n[e] = n;
  st_p[e] = a;
  st_norm[e] = b;
  if (e == 0 && status_mirror) *(volatile unsigned int*)status_mirror = sw;
}

}  // namespace

int combine_col_blocks(int d) { return (d + kSegCols - 1) / kSegCols; }

namespace {

template <typename TY, int KM>
cudaError_t launch_combine_t(int o_bf16, cudaStream_t st, const void* opart, int n_split,
                             size_t stride, const int32_t* slot_of, const float* w,
                             const void* sout, int s_bf16, int S, int T, int K, int d, void* y,
                             float* nrm_part, const unsigned int* status) {
  const int nseg = combine_col_blocks(d);
  const long long tasks = (long long)T * nseg;
  const dim3 grid((unsigned)((tasks + kCombThreads / 32 - 1) / (kCombThreads / 32)));
  if (o_bf16)
    return launch_pdl(combine_kernel<TY, KM, true>, grid, dim3(kCombThreads), 0, st, opart,
                      n_split, stride, slot_of, w, sout, s_bf16, S, T, K, d, nseg, (TY*)y,
                      nrm_part, status);
  return launch_pdl(combine_kernel<TY, KM, false>, grid, dim3(kCombThreads), 0, st, opart,
                    n_split, stride, slot_of, w, sout, s_bf16, S, T, K, d, nseg, (TY*)y,
                    nrm_part, status);
}

template <typename TY>
cudaError_t launch_combine_k(int o_bf16, cudaStream_t st, const void* opart, int n_split,
                             size_t stride, const int32_t* slot_of, const float* w,
                             const void* sout, int s_bf16, int S, int T, int K, int d, void* y,
                             float* nrm_part, const unsigned int* status) {
#define EAT_COMB(KM)                                                                           \
  launch_combine_t<TY, KM>(o_bf16, st, opart, n_split, stride, slot_of, w, sout, s_bf16, S, T, \
                           K, d, y, nrm_part, status)
  if (K <= 2) return EAT_COMB(2);
  if (K <= 4) return EAT_COMB(4);
  if (K <= 8) return EAT_COMB(8);
  return EAT_COMB(16);
#undef EAT_COMB
}

}  // namespace

cudaError_t launch_combine(int y_bf16, const void* opart, int o_bf16, int n_split,
                           int split_stride_rows, const int32_t* slot_of, const float* w,
                           const void* sout, int s_bf16, int S, int T, int K, int d, void* y,
                           float* nrm_part, const unsigned int* status, cudaStream_t st) {
  const size_t stride = (size_t)split_stride_rows * d;
  if (y_bf16)
    return launch_combine_k<__nv_bfloat16>(o_bf16, st, opart, n_split, stride, slot_of, w, sout,
                                           s_bf16, S, T, K, d, y, nrm_part, status);
  return launch_combine_k<float>(o_bf16, st, opart, n_split, stride, slot_of, w, sout, s_bf16, S,
                                 T, K, d, y, nrm_part, status);
}

int account_chunks(long long rows) {
  return rows > kAccChunk ? (int)((rows + kAccChunk - 1) / kAccChunk) : 1;
}

cudaError_t launch_account(const int32_t* offs, const float* perm_p, const float* nrm_part, int nb,
                           int E, long long rows, double alpha, int64_t* N, double* P, double* C,
                           int32_t* st_n, double* st_p, double* st_norm, long long* counters,
                           float4* chunk_sums, unsigned int* tickets, const unsigned int* status,
                           unsigned int* status_mirror, cudaStream_t st) {
  return launch_pdl(account_kernel, dim3(E, account_chunks(rows)), dim3(kAccThreads), 0, st, offs,
                    perm_p, nrm_part, nb, alpha, N, P, C, st_n, st_p, st_norm,
                    (unsigned long long*)counters, chunk_sums, tickets, status, status_mirror);
}

}  // namespace eat
