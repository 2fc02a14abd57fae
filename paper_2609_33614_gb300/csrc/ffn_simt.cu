// CUDA-core expert FFN kernels: the path for fp32 layers (full fp32 arithmetic, no tensor-core
// rounding) over grouped, gathered rows.  SwiGLU experts (§3.1 expert FFN; the configurations use
// SwiGLU): act = silu(x Wg^T) * (x Wu^T) fused in the first kernel's epilogue; the second kernel
// is the down projection act Wd^T, written per slot in fp32 for the combine.
//
// Tile: 32 rows x 64 output features, K in chunks of 32 staged through shared memory; 256
// threads, each owning 2 rows x 4 features (x2 for gate and up).  Blocks map to (feature tile,
// row tile); a row tile belongs to one group (expert), found from the tile prefix.
#include "eat_internal.cuh"

namespace eat {

namespace {

constexpr int BR = kSimtTileRows;  // rows per tile
constexpr int BF = 64;             // output features per tile
constexpr int BK = 32;
constexpr int kThreads = 256;

__device__ __forceinline__ float ld(const float* p, size_t i) { return p[i]; }
__device__ __forceinline__ float ld(const __nv_bfloat16* p, size_t i) {
  return __bfloat162float(p[i]);
}
__device__ __forceinline__ void st(float* p, size_t i, float v) { p[i] = v; }
__device__ __forceinline__ void st(__nv_bfloat16* p, size_t i, float v) {
  p[i] = __float2bfloat16_rn(v);
}

struct TileInfo {
  int g, row0, nrows, slot0;
  bool ok;
};

__device__ __forceinline__ TileInfo find_tile(const GroupMap& gm, int u) {
  TileInfo ti;
  ti.ok = false;
  if (gm.tile_offs) {
    if (u >= gm.tile_offs[gm.n_groups]) return ti;
    int lo = 0, hi = gm.n_groups - 1;  // last g with tile_offs[g] <= u
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (gm.tile_offs[mid] <= u) lo = mid;
      else hi = mid - 1;
    }
    ti.g = lo;
    ti.row0 = (u - gm.tile_offs[lo]) * BR;
  } else {
    const int tpg = (gm.uniform_rows + BR - 1) / BR;
    if (u >= tpg * gm.n_groups) return ti;
    ti.g = u / tpg;
    ti.row0 = (u % tpg) * BR;
  }
  const int beg = gm.row_offs ? gm.row_offs[ti.g] : ti.g * gm.uniform_rows;
  const int end = gm.row_offs ? gm.row_offs[ti.g + 1] : (ti.g + 1) * gm.uniform_rows;
  ti.slot0 = beg + ti.row0;
  ti.nrows = min(BR, end - ti.slot0);
  ti.ok = ti.nrows > 0;
  return ti;
}

__device__ __forceinline__ int in_row(const GroupMap& gm, int g, int s) {
  if (gm.row_mode == kRowGather) return gm.row_tok[s];
  if (gm.row_mode == kRowSlot) return s;
  return s - g * gm.uniform_rows;
}

template <typename TW, bool GATEUP>
__global__ void __launch_bounds__(kThreads)
ffn_simt_kernel(const TW* __restrict__ in, const TW* __restrict__ w0, const TW* __restrict__ w1,
                int Fout, int Kdim, GroupMap gm, void* __restrict__ outp) {
  __shared__ float as[BR][BK + 1];
  __shared__ float ws0[BF][BK + 1];
  __shared__ float ws1[GATEUP ? BF : 1][BK + 1];
  __shared__ int rows[BR];
  pdl_wait();
  pdl_launch_dependents();
  const TileInfo ti = find_tile(gm, blockIdx.y);
  if (!ti.ok) return;
  const int f0 = blockIdx.x * BF;
  const int tid = threadIdx.x;
  if (tid < BR) rows[tid] = tid < ti.nrows ? in_row(gm, ti.g, ti.slot0 + tid) : -1;
  __syncthreads();
  const size_t wbase = (size_t)ti.g * Fout * Kdim;
  const int tr = tid >> 4;   // 0..15 -> rows tr, tr + 16
  const int tf = tid & 15;   // 0..15 -> features tf + 16 q
  float acc0[2][4] = {}, acc1[2][4] = {};
  for (int k0 = 0; k0 < Kdim; k0 += BK) {
    for (int i = tid; i < BR * BK; i += kThreads) {
      const int r = i / BK, kk = i % BK;
      const int row = rows[r];
      as[r][kk] = row >= 0 ? ld(in, (size_t)row * Kdim + k0 + kk) : 0.f;
    }
    for (int i = tid; i < BF * BK; i += kThreads) {
      const int f = i / BK, kk = i % BK;
      const bool okf = f0 + f < Fout;
      ws0[f][kk] = okf ? ld(w0, wbase + (size_t)(f0 + f) * Kdim + k0 + kk) : 0.f;
      if (GATEUP) ws1[f][kk] = okf ? ld(w1, wbase + (size_t)(f0 + f) * Kdim + k0 + kk) : 0.f;
    }
    __syncthreads();
#pragma unroll 8
    for (int kk = 0; kk < BK; ++kk) {
      const float a0 = as[tr][kk], a1 = as[tr + 16][kk];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const float b0 = ws0[tf + 16 * q][kk];
        acc0[0][q] = fmaf(a0, b0, acc0[0][q]);
        acc0[1][q] = fmaf(a1, b0, acc0[1][q]);
        if (GATEUP) {
          const float b1 = ws1[tf + 16 * q][kk];
          acc1[0][q] = fmaf(a0, b1, acc1[0][q]);
          acc1[1][q] = fmaf(a1, b1, acc1[1][q]);
        }
      }
    }
    __syncthreads();
  }
#pragma unroll
  for (int rr = 0; rr < 2; ++rr) {
    const int r = tr + 16 * rr;
    if (r >= ti.nrows) continue;
    const size_t slot = (size_t)ti.slot0 + r;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int f = f0 + tf + 16 * q;
      if (f >= Fout) continue;
      if (GATEUP) {
        const float g = acc0[rr][q];
        const float silu = g / (1.0f + expf(-g));
        st((TW*)outp, slot * Fout + f, silu * acc1[rr][q]);
      } else {
        ((float*)outp)[slot * Fout + f] = acc0[rr][q];
      }
    }
  }
}

}  // namespace

cudaError_t launch_ffn_gateup_simt(int dtype_bf16, const void* in, const void* wg, const void* wu,
                                   int Fout, int Kdim, GroupMap gm, void* act, cudaStream_t st) {
  dim3 grid((Fout + BF - 1) / BF, gm.max_tiles);
  if (grid.y == 0) return cudaSuccess;
  if (dtype_bf16)
    return launch_pdl(ffn_simt_kernel<__nv_bfloat16, true>, grid, dim3(kThreads), 0, st,
                      (const __nv_bfloat16*)in, (const __nv_bfloat16*)wg,
                      (const __nv_bfloat16*)wu, Fout, Kdim, gm, act);
  return launch_pdl(ffn_simt_kernel<float, true>, grid, dim3(kThreads), 0, st, (const float*)in,
                    (const float*)wg, (const float*)wu, Fout, Kdim, gm, act);
}

cudaError_t launch_ffn_down_simt(int dtype_bf16, const void* act, const void* wd, int Dout,
                                 int Kdim, GroupMap gm, float* out, cudaStream_t st) {
  dim3 grid((Dout + BF - 1) / BF, gm.max_tiles);
  if (grid.y == 0) return cudaSuccess;
  GroupMap g2 = gm;
  g2.row_mode = kRowSlot;  // the down projection reads act rows in slot order
  if (dtype_bf16)
    return launch_pdl(ffn_simt_kernel<__nv_bfloat16, false>, grid, dim3(kThreads), 0, st,
                      (const __nv_bfloat16*)act, (const __nv_bfloat16*)wd,
                      (const __nv_bfloat16*)nullptr, Dout, Kdim, g2, (void*)out);
  return launch_pdl(ffn_simt_kernel<float, false>, grid, dim3(kThreads), 0, st,
                    (const float*)act, (const float*)wd, (const float*)nullptr, Dout, Kdim, g2,
                    (void*)out);
}

}  // namespace eat
