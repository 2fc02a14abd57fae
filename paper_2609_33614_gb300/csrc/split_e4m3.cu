// fp8 layers: the split of a GEMM's bf16 B operand into e4m3 hi/lo planes with per-row
// power-of-two scales (the operand format of the e4m3 x e4m3 tensor-core MMAs in ffn_tc.cu).
#include "ffn_tc.cuh"

#include <algorithm>

namespace eat {

namespace {

// fp8 layers: the B operand of an expert GEMM as two e4m3 planes.  Output row r (r < *n_dev, or
// n_host without a count) takes source row map[r] (or r) of a bf16 matrix, picks the power of two
// s_r that puts the row's largest magnitude in [128, 256) (the e4m3 range ends at 448), and stores
// hi = e4m3(v / s_r) in plane 0 and lo = e4m3(v / s_r - hi) in plane 1, and s_r in scale[r].  A
// bf16 value keeps 8 significant bits, hi the leading 4 and the remainder at most 4 more, so
// hi + lo equals v / s_r exactly where that remainder stays on the e4m3 grid: scaled magnitudes of
// at least 1/4, i.e. every value within 2^-9 of the row's largest magnitude; below, the error is
// at most half the e4m3 subnormal step (2^-10 after scaling).  A row with an infinite or NaN largest
// magnitude gets a NaN scale, so the outputs it feeds are NaN.
// Two floats -> two e4m3 bytes, `first` in the low byte (the lower address); the conversion puts
// its first source operand in the upper byte.
__device__ __forceinline__ uint16_t e4m3x2_of(float first, float second) {
  uint16_t r;
  asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(r) : "f"(second), "f"(first));
  return r;
}
__device__ __forceinline__ float2 f32x2_of_e4m3x2(uint16_t v) {
  uint32_t h;
  asm("cvt.rn.f16x2.e4m3x2 %0, %1;" : "=r"(h) : "h"(v));
  return __half22float2(*(const __half2*)&h);
}

// 8 bf16 values -> their 8 hi and 8 lo e4m3 bytes (v * inv = hi + lo + remainder).
__device__ __forceinline__ void split8(const uint4& u, float inv, uint2& hi, uint2& lo) {
  const uint32_t w[4] = {u.x, u.y, u.z, u.w};
  uint32_t hw[2] = {0u, 0u}, lw[2] = {0u, 0u};
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    // a bf16 is the upper half of the float with the same value
    const float a = __uint_as_float(w[q] << 16) * inv;  // exact: a power of two
    const float b = __uint_as_float(w[q] & 0xffff0000u) * inv;
    const uint16_t h = e4m3x2_of(a, b);
    const float2 hf = f32x2_of_e4m3x2(h);
    const uint16_t l = e4m3x2_of(a - hf.x, b - hf.y);  // exact differences
    hw[q >> 1] |= (uint32_t)h << (16 * (q & 1));
    lw[q >> 1] |= (uint32_t)l << (16 * (q & 1));
  }
  hi = make_uint2(hw[0], hw[1]);
  lo = make_uint2(lw[0], lw[1]);
}
__device__ __forceinline__ float amax8(const uint4& u, float m) {
  const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
  for (int q = 0; q < 4; ++q)
    m = fmaxf(m, fmaxf(fabsf(__uint_as_float(w[q] << 16)),
                       fabsf(__uint_as_float(w[q] & 0xffff0000u))));
  return m;
}

// The row's power-of-two scale from its largest magnitude m: s with m / s in [128, 256), its
// inverse, and a NaN scale for a non-finite m (rows below 2^-119 keep scale 1).
__device__ __forceinline__ void split_scale(float m, float& s, float& inv) {
  const uint32_t ex = (__float_as_uint(m) >> 23) & 0xffu;  // m in [2^(ex-127), 2^(ex-126))
  s = 1.0f;
  inv = 1.0f;
  if (ex == 0xffu) {
    s = __uint_as_float(0x7fc00000u);
  } else if (ex >= 8u) {
    s = __uint_as_float((ex - 7u) << 23);     // 2^(ex - 134)
    inv = __uint_as_float((261u - ex) << 23);  // 2^(134 - ex)
  }
}

// Rows of at most 32 x VPL 16-byte vectors (256 bf16 per VPL): one warp per row, the row held in
// registers and reduced with shuffles, eight rows per 256-thread CTA and no block barrier, so a
// prefill call keeps thousands of rows in flight.
template <int VPL>
__global__ void __launch_bounds__(256)
split_e4m3_warp_kernel(const __nv_bfloat16* __restrict__ src, const int32_t* __restrict__ map,
                       const int32_t* __restrict__ n_dev, int n_host, int cols,
                       uint8_t* __restrict__ dst, long long plane, float* __restrict__ scale) {
  pdl_wait();
  pdl_launch_dependents();
  const int n = n_dev ? *n_dev : n_host;
  const int lane = threadIdx.x & 31;
  const int r = blockIdx.x * 8 + (threadIdx.x >> 5);
  if (r >= n) return;
  const int vecs = cols >> 3;
  const int sr = map ? map[r] : r;
  const uint4* row = (const uint4*)(src + (size_t)sr * cols);
  uint4 v[VPL];
  float m = 0.0f;
#pragma unroll
  for (int j = 0; j < VPL; ++j) {
    const int i = lane + 32 * j;
    v[j] = i < vecs ? row[i] : make_uint4(0u, 0u, 0u, 0u);
  }
#pragma unroll
  for (int j = 0; j < VPL; ++j) m = amax8(v[j], m);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
  float s, inv;
  split_scale(m, s, inv);
  if (lane == 0) scale[r] = s;
  uint2* hi_row = (uint2*)(dst + (size_t)r * cols);
  uint2* lo_row = (uint2*)(dst + plane + (size_t)r * cols);
#pragma unroll
  for (int j = 0; j < VPL; ++j) {
    const int i = lane + 32 * j;
    if (i < vecs) {
      uint2 h, l;
      split8(v[j], inv, h, l);
      hi_row[i] = h;
      lo_row[i] = l;
    }
  }
}

// Longer rows: one CTA per row; rows of up to 256 x kSplitRegs 16-byte vectors (16384 bf16) are
// read once and kept in registers, longer ones are read twice.
constexpr int kSplitRegs = 8;

__global__ void __launch_bounds__(256)
split_e4m3_kernel(const __nv_bfloat16* __restrict__ src, const int32_t* __restrict__ map,
                  const int32_t* __restrict__ n_dev, int n_host, int cols,
                  uint8_t* __restrict__ dst, long long plane, float* __restrict__ scale) {
  __shared__ float red[8];
  pdl_wait();
  pdl_launch_dependents();
  const int n = n_dev ? *n_dev : n_host;
  const int vecs = cols >> 3;
  const bool in_regs = vecs <= 256 * kSplitRegs;
  const int tid = threadIdx.x;
  for (int r = blockIdx.x; r < n; r += gridDim.x) {
    const int sr = map ? map[r] : r;
    const uint4* row = (const uint4*)(src + (size_t)sr * cols);
    uint4 v[kSplitRegs];
    float m = 0.0f;
    if (in_regs) {
#pragma unroll
      for (int j = 0; j < kSplitRegs; ++j) {
        const int i = tid + 256 * j;
        v[j] = i < vecs ? row[i] : make_uint4(0u, 0u, 0u, 0u);
      }
#pragma unroll
      for (int j = 0; j < kSplitRegs; ++j) m = amax8(v[j], m);
    } else {
      for (int i = tid; i < vecs; i += 256) m = amax8(row[i], m);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
    if ((tid & 31) == 0) red[tid >> 5] = m;
    __syncthreads();
    m = red[0];
#pragma unroll
    for (int i = 1; i < 8; ++i) m = fmaxf(m, red[i]);
    __syncthreads();  // red is rewritten for the next row
    float s, inv;
    split_scale(m, s, inv);
    if (tid == 0) scale[r] = s;
    uint2* hi_row = (uint2*)(dst + (size_t)r * cols);
    uint2* lo_row = (uint2*)(dst + plane + (size_t)r * cols);
    uint2 h, l;
    if (in_regs) {
#pragma unroll
      for (int j = 0; j < kSplitRegs; ++j) {
        const int i = tid + 256 * j;
        if (i < vecs) {
          split8(v[j], inv, h, l);
          hi_row[i] = h;
          lo_row[i] = l;
        }
      }
    } else {
      for (int i = tid; i < vecs; i += 256) {
        split8(row[i], inv, h, l);
        hi_row[i] = h;
        lo_row[i] = l;
      }
    }
  }
}

}  // namespace

cudaError_t tc_launch_split(const TcLayer& L, const TcCall& c, TcSplit which, cudaStream_t st) {
  const long long rows = (long long)L.Tmax * L.K;
  const __nv_bfloat16* src = nullptr;
  const int32_t* map = nullptr;
  const int32_t* n_dev = nullptr;
  int n_host = 0, cols = 0;
  uint8_t* dst = nullptr;
  float* scale = nullptr;
  long long plane_rows = 0;
  switch (which) {
    case TcSplit::kSlotX:  // routed gate/up: x rows in slot order
      src = (const __nv_bfloat16*)c.x, map = c.perm_tok, n_dev = c.offs + L.E;
      n_host = c.T * L.K, cols = L.d, dst = L.q.xq, scale = L.q.xq_s, plane_rows = rows;
      break;
    case TcSplit::kTokenX:  // shared gate/up: x rows in token order
      src = (const __nv_bfloat16*)c.x, n_host = c.T, cols = L.d;
      dst = L.q.xqt, scale = L.q.xqt_s, plane_rows = L.Tmax;
      break;
    case TcSplit::kAct:  // routed down: the gate/up activations of the call's slots
      src = (const __nv_bfloat16*)c.act, n_dev = c.offs + L.E, n_host = c.T * L.K, cols = L.F;
      dst = L.q.aq, scale = L.q.aq_s, plane_rows = rows;
      break;
    case TcSplit::kSharedAct:  // shared down: rows g * T + t
      src = (const __nv_bfloat16*)c.sact, n_host = L.S * c.T, cols = L.Fs;
      dst = L.q.saq, scale = L.q.saq_s, plane_rows = (long long)L.S * L.Tmax;
      break;
  }
  if (n_host <= 0) return cudaSuccess;
  const int vecs = cols / 8;
  const dim3 wgrid((n_host + 7) / 8);
  if (vecs <= 32 * 8)
    return launch_pdl(split_e4m3_warp_kernel<8>, wgrid, dim3(256), 0, st, src, map, n_dev, n_host,
                      cols, dst, plane_rows * cols, scale);
  if (vecs <= 32 * 16)
    return launch_pdl(split_e4m3_warp_kernel<16>, wgrid, dim3(256), 0, st, src, map, n_dev,
                      n_host, cols, dst, plane_rows * cols, scale);
  const int grid = std::min(n_host, 4 * L.num_sms);
  return launch_pdl(split_e4m3_kernel, dim3(grid), dim3(256), 0, st, src, map, n_dev, n_host,
                    cols, dst, plane_rows * cols, scale);
}


}  // namespace eat
