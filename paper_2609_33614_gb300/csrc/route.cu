// Router and EAT selection (§3.1-§3.4 of the EAT paper, Eq. 1-8).
//
//  router_logits_small_kernel (T <= 128, decode) / router_logits_sk_kernel (bf16 x, larger calls;
//      stream-K over tiles and chunks of d) / router_logits_kernel (other large calls; both tiled
//      through shared memory): partial router scores x . w_r over slices of d: fp32 FMA inside
//      16- or 32-wide chunks, chunk sums accumulated in Kahan-compensated fp32, so the
//      logits carry ~1e-7 absolute error (the selection compares I against tau at 1e-5 and P_total
//      sums p at 1e-6 relative).  The scores stay off the tensor cores: their fp32 accumulation
//      biased the scores enough to move P_total by ~1e-6 relative.
//  route_select_kernel: one warp per token.  Each lane owns experts lane, lane+32, ...; the warp
//      does the softmax (§3.2), importance (Eq. 2), mean / population std (Eq. 3-4), tau (Eq. 5),
//      PPL factor and smoothing (§3.3), the clamp to the type-7 q_lo / q_hi quantiles of p
//      (order statistics from a warp-wide bitonic sort of (value, index) pairs), the candidate
//      set and K cap (Eq. 6, ties to the lower index; the K-th pair of the same sort) and the
//      renormalised gates (Eq. 7-8), with shuffles only.
//      The history score S_h (Eq. 1) is computed once per block from the accounts.
#include "eat_internal.cuh"

#include <math.h>

#include <algorithm>
#include <atomic>

namespace eat {

namespace {

constexpr int kLogitThreads = 256;

__device__ __forceinline__ float load_x(const float* p, size_t i) { return p[i]; }
__device__ __forceinline__ float load_x(const __nv_bfloat16* p, size_t i) {
  return __bfloat162float(p[i]);
}


// Router scores for large T: CTA tile of 64 tokens x 64 experts over one slice of d, 256 threads
// with 4 tokens x 4 experts each.  x and W_r chunks of 32 columns are staged transposed in shared
// memory; every output takes 32 fp32 FMAs per chunk and the chunk sums are added with Kahan
// compensation (fp32), so the score carries about the error of an fp64 sum of fp32 products.
constexpr int kTileT = 64, kTileE = 64, kChunkK = 32;

__device__ __forceinline__ void kahan_add(float& sum, float& comp, float v) {
  const float y = v - comp;
  const float t = sum + y;
  comp = (t - sum) - y;
  sum = t;
}

template <typename TX>
__global__ void __launch_bounds__(kLogitThreads)
router_logits_kernel(const TX* __restrict__ x, const float* __restrict__ wr, int T, int d, int E,
                     int d_per_split, float2* __restrict__ part) {
  __shared__ float xs[kChunkK][kTileT + 4];
  __shared__ float ws[kChunkK][kTileE + 4];
  pdl_wait();
  pdl_launch_dependents();
  const int tid = threadIdx.x;
  const int tx = tid & 15, ty = tid >> 4;
  const int t0 = blockIdx.x * kTileT, e0 = blockIdx.y * kTileE;
  const int dbeg = blockIdx.z * d_per_split;
  const int dend = min(d, dbeg + d_per_split);
  float sum[4][4], comp[4][4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) sum[i][j] = comp[i][j] = 0.f;

  for (int k0 = dbeg; k0 < dend; k0 += kChunkK) {
    // stage: 64 rows x 32 columns of x and of W_r, transposed (column-major in shared memory)
    for (int i = tid; i < kTileT * kChunkK; i += kLogitThreads) {
      const int r = i / kChunkK, kk = i % kChunkK;
      const int t = t0 + r, k = k0 + kk;
      xs[kk][r] = (t < T && k < dend) ? load_x(x, (size_t)t * d + k) : 0.f;
      const int e = e0 + r;
      ws[kk][r] = (e < E && k < dend) ? wr[(size_t)e * d + k] : 0.f;
    }
    __syncthreads();
    float acc[4][4];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
#pragma unroll 8
    for (int kk = 0; kk < kChunkK; ++kk) {
      const float4 a = *(const float4*)&xs[kk][ty * 4];
      const float4 b = *(const float4*)&ws[kk][tx * 4];
      const float av[4] = {a.x, a.y, a.z, a.w}, bv[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(av[i], bv[j], acc[i][j]);
    }
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int j = 0; j < 4; ++j) kahan_add(sum[i][j], comp[i][j], acc[i][j]);
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int t = t0 + ty * 4 + i;
    if (t >= T) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int e = e0 + tx * 4 + j;
      if (e < E)
        part[((size_t)blockIdx.z * T + t) * E + e] = make_float2(sum[i][j], -comp[i][j]);
    }
  }
}

// Router scores for small T (decode): block (t, s, z) computes part[s][t][e] over the s-th slice
// of d for the experts e = 8 z + w of its warps w; lanes read float4 pieces of the weight row and
// of x (coalesced), multiply in fp32, fold each 16 products into a compensated lane sum, and the
// 32 lane sums are added compensated (a fixed tree).
constexpr int kSmallT = kSmallRouterT;
constexpr int kSmallSlice = 512;


// Four consecutive elements of x: their bits (copied as they are) and their fp32 values.
struct X4f {
  float4 bits;
  __device__ __forceinline__ float4 val() const { return bits; }
};
struct X4b {
  uint2 bits;
  __device__ __forceinline__ float4 val() const {
    const float2 fa = __bfloat1622float2(*(const __nv_bfloat162*)&bits.x);
    const float2 fb = __bfloat1622float2(*(const __nv_bfloat162*)&bits.y);
    return make_float4(fa.x, fa.y, fb.x, fb.y);
  }
};
__device__ __forceinline__ X4f load_x4(const float* p) { return X4f{*(const float4*)p}; }
__device__ __forceinline__ X4b load_x4(const __nv_bfloat16* p) { return X4b{*(const uint2*)p}; }
__device__ __forceinline__ void store_x4(float* p, const X4f& v) { *(float4*)p = v.bits; }
__device__ __forceinline__ void store_x4(__nv_bfloat16* p, const X4b& v) { *(uint2*)p = v.bits; }

// xcopy (or null): x is read from memory the caller keeps on the host (a host-buffer call) and
// warp 0 of the blocks of the first expert group also writes what it reads to xcopy, the device
// copy every later kernel of the call reads.
// (bf16 x: at most 32 registers, so eight blocks share an SM and a 32-token decode call of a
// 64-expert layer, 1024 blocks, runs in one wave)
template <typename TX>
__global__ void __launch_bounds__(kLogitThreads, sizeof(TX) == 2 ? 8 : 1)
router_logits_small_kernel(const TX* __restrict__ x, const float* __restrict__ wr, int T, int d,
                           int E, int d_per_split, float2* __restrict__ part,
                           TX* __restrict__ xcopy) {
  pdl_wait();
  pdl_launch_dependents();
  const int t = blockIdx.x, s = blockIdx.y;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int beg = s * d_per_split;
  const int end = min(d, beg + d_per_split);
  const TX* xr = x + (size_t)t * d;
  TX* xc = xcopy && blockIdx.z == 0 && warp == 0 ? xcopy + (size_t)t * d : nullptr;
  // one expert per warp: blockIdx.z picks the group of kLogitThreads / 32 experts
  {
    const int e = blockIdx.z * (kLogitThreads / 32) + warp;
    if (e >= E) return;
    const float* wrow = wr + (size_t)e * d;
    float hi = 0.f, lo = 0.f;
    float acc = 0.f;
    int cnt = 0;
    for (int c = beg + lane * 4; c < end; c += 128) {
      const float4 wv = *(const float4*)(wrow + c);
      const auto xb = load_x4(xr + c);
      if (xc) store_x4(xc + c, xb);
      const float4 xv = xb.val();
      acc = fmaf(xv.x, wv.x, acc);
      acc = fmaf(xv.y, wv.y, acc);
      acc = fmaf(xv.z, wv.z, acc);
      acc = fmaf(xv.w, wv.w, acc);
      if (++cnt == 4) {
        df_add(hi, lo, acc);
        acc = 0.f;
        cnt = 0;
      }
    }
    df_add(hi, lo, acc);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float ohi = __shfl_xor_sync(0xffffffffu, hi, o);
      const float olo = __shfl_xor_sync(0xffffffffu, lo, o);
      df_add(hi, lo, ohi, olo);
    }
    if (lane == 0) part[((size_t)s * T + t) * E + e] = make_float2(hi, lo);
  }
}

// Router scores for large T with bf16 x (d a multiple of 32, 16-byte aligned x and W_r).  The
// work is the units (64-token x 64-expert tile, 32-column chunk of d), numbered tile-major, and a
// persistent grid of G CTAs (as many as fit on the SMs, each at least kSKMinUnits units) takes
// contiguous, equal runs of them (stream-K): no tail wave, and a CTA's run may start or end inside
// a tile.  Each thread keeps TM tokens x 4 experts (experts tx, tx + 16, tx + 32, tx + 48, so a
// warp's weight reads cover 16 consecutive rows and hit distinct bank groups) and adds each
// chunk's 32 fp32 FMAs into a Kahan-compensated fp32 sum, as the other router-score kernels do.
// Where its run leaves a tile, a CTA writes the tile's compensated sums to split slice
// seg = (its index) - (index of the CTA that starts the tile); the CTA that ends a tile also
// writes zero pairs to the slices after its own, up to n_split, so the selection kernel adds a
// fixed number of slices for every tile.  x and W_r go through a three-stage shared-memory ring
// as fp32 (row stride 36 floats): W_r by cp.async, x through registers (converted when stored),
// two units ahead; one block barrier per unit.
constexpr int kSKT = 64, kSKE = 64, kSKS = kChunkK + 4, kSKStages = 3;
constexpr int kSKTM = 4;        // tokens per thread: 256 threads, two CTAs per SM
constexpr int kSKMinUnits = 8;  // 256 columns of d per CTA at least
constexpr size_t kSKSmem = (size_t)kSKStages * (kSKT + kSKE) * kSKS * sizeof(float);
template <int TM>
struct SkCfg {
  static constexpr int kThreads = kSKT * kSKE / (4 * TM);
  static constexpr int kWPieces = kSKE * kChunkK / 4 / kThreads;  // 16-byte pieces per thread
  static constexpr int kXPieces = kSKT * kChunkK / 8 / kThreads;
};

// the CTA whose run [g U / G, (g + 1) U / G) holds unit u
__host__ __device__ __forceinline__ int sk_owner(long long u, long long U, int G) {
  return (int)(((u + 1) * (long long)G - 1) / U);
}

__device__ __forceinline__ void bf16x8_to_f32(const uint4& u, float (&v)[8]) {
  const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const float2 f = __bfloat1622float2(*(const __nv_bfloat162*)&w[q]);
    v[2 * q] = f.x;
    v[2 * q + 1] = f.y;
  }
}

// A unit's place: token tile, expert tile and chunk, advanced one unit at a time (no division in
// the loop).
struct SkCursor {
  int tt, et, ch;
  __device__ __forceinline__ void next(int etiles, int nc) {
    if (++ch == nc) {
      ch = 0;
      if (++et == etiles) {
        et = 0;
        ++tt;
      }
    }
  }
};

template <int TM>
__global__ void __launch_bounds__(SkCfg<TM>::kThreads, 2)
router_logits_sk_kernel(const __nv_bfloat16* __restrict__ x, const float* __restrict__ wr, int T,
                        int d, int E, int n_split, float2* __restrict__ part,
                        __nv_bfloat16* __restrict__ xcopy) {
  using C = SkCfg<TM>;
  extern __shared__ __align__(16) float sk_smem[];
  float* xs = sk_smem;                              // [stage][64 tokens][kSKS]
  float* ws = sk_smem + kSKStages * kSKT * kSKS;    // [stage][64 experts][kSKS]
  pdl_wait();
  pdl_launch_dependents();
  const int nc = d / kChunkK;
  const int etiles = (E + kSKE - 1) / kSKE;
  const int U = ((T + kSKT - 1) / kSKT) * etiles * nc;
  const int G = gridDim.x, g = blockIdx.x;
  const int u0 = (int)((long long)g * U / G), u1 = (int)((long long)(g + 1) * U / G);
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  SkCursor ld, cu;  // the next unit to load, the unit being computed
  {
    const int tile = u0 / nc;
    ld.tt = tile / etiles;
    ld.et = tile - ld.tt * etiles;
    ld.ch = u0 - tile * nc;
    cu = ld;
  }

  // W_r: 64 rows x 32 floats in 16-byte pieces q = tid + kThreads r: row q / 8, columns (q % 8) * 4
  // x: 64 rows x 32 bf16 in 16-byte pieces q = tid + kThreads r: row q / 4, columns (q % 4) * 8
  uint4 xr[C::kXPieces];
  int x_t0 = 0, x_k0 = 0;  // where the pieces in xr came from
  bool x_keep = false;     // and whether they go to xcopy (units of the first expert tile)
  // the next unit's W_r pieces (cp.async) and x pieces (registers), then advance the cursor
  auto issue = [&](bool live, int stage) {
    if (live) {
      const int t0 = ld.tt * kSKT, e0 = ld.et * kSKE, k0 = ld.ch * kChunkK;
      x_t0 = t0;
      x_k0 = k0;
      x_keep = xcopy != nullptr && ld.et == 0;
      float* wsb = ws + stage * kSKE * kSKS;
#pragma unroll
      for (int r = 0; r < C::kWPieces; ++r) {
        const int q = tid + r * C::kThreads, row = q >> 3, c4 = (q & 7) * 4;
        if (e0 + row < E)
          cp_async16((uint32_t)__cvta_generic_to_shared(&wsb[row * kSKS + c4]),
                     wr + (size_t)(e0 + row) * d + k0 + c4);
        else
          *(float4*)&wsb[row * kSKS + c4] = make_float4(0.f, 0.f, 0.f, 0.f);
      }
#pragma unroll
      for (int r = 0; r < C::kXPieces; ++r) {
        const int q = tid + r * C::kThreads, row = q >> 2, c8 = (q & 3) * 8;
        xr[r] = t0 + row < T ? *(const uint4*)(x + (size_t)(t0 + row) * d + k0 + c8)
                             : make_uint4(0u, 0u, 0u, 0u);
      }
      ld.next(etiles, nc);
    }
    cp_async_commit();  // (an empty group past the run keeps the group count uniform)
  };
  auto store_x = [&](bool live, int stage) {
    if (live) {
      float* xsb = xs + stage * kSKT * kSKS;
#pragma unroll
      for (int r = 0; r < C::kXPieces; ++r) {
        const int q = tid + r * C::kThreads, row = q >> 2, c8 = (q & 3) * 8;
        float v[8];
        bf16x8_to_f32(xr[r], v);
        *(float4*)&xsb[row * kSKS + c8] = make_float4(v[0], v[1], v[2], v[3]);
        *(float4*)&xsb[row * kSKS + c8 + 4] = make_float4(v[4], v[5], v[6], v[7]);
        if (x_keep && x_t0 + row < T) *(uint4*)(xcopy + (size_t)(x_t0 + row) * d + x_k0 + c8) = xr[r];
      }
    }
  };

  float sum[TM][4], comp[TM][4];
#pragma unroll
  for (int i = 0; i < TM; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) sum[i][j] = comp[i][j] = 0.f;

  issue(true, 0);
  store_x(true, 0);
  issue(u0 + 1 < u1, 1);
  store_x(u0 + 1 < u1, 1);
  int stage = 0;
  for (int u = u0; u < u1; ++u) {
    cp_async_wait<1>();  // this thread's W_r pieces of unit u have landed
    __syncthreads();     // everyone's pieces of unit u are visible; unit u - 1's stage is free
    const int ahead = stage == 0 ? kSKStages - 1 : stage - 1;  // the stage of unit u + 2
    const bool live2 = u + 2 < u1;
    issue(live2, ahead);
    const float* xsb = xs + stage * kSKT * kSKS;
    const float* wsb = ws + stage * kSKE * kSKS;
    float acc[TM][4];
#pragma unroll
    for (int i = 0; i < TM; ++i)
#pragma unroll
      for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
#pragma unroll
    for (int kk = 0; kk < kChunkK; kk += 4) {
      float4 b[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) b[j] = *(const float4*)&wsb[(tx + 16 * j) * kSKS + kk];
#pragma unroll
      for (int i = 0; i < TM; ++i) {
        const float4 a = *(const float4*)&xsb[(ty * TM + i) * kSKS + kk];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          acc[i][j] = fmaf(a.x, b[j].x, acc[i][j]);
          acc[i][j] = fmaf(a.y, b[j].y, acc[i][j]);
          acc[i][j] = fmaf(a.z, b[j].z, acc[i][j]);
          acc[i][j] = fmaf(a.w, b[j].w, acc[i][j]);
        }
      }
    }
#pragma unroll
    for (int i = 0; i < TM; ++i)
#pragma unroll
      for (int j = 0; j < 4; ++j) kahan_add(sum[i][j], comp[i][j], acc[i][j]);
    store_x(live2, ahead);
    const bool tile_end = cu.ch == nc - 1;
    if (tile_end || u + 1 == u1) {
      const long long tile = (long long)cu.tt * etiles + cu.et;
      const int seg = g - sk_owner(tile * nc, U, G);  // < n_split (the host's bound)
      const int t0 = cu.tt * kSKT, e0 = cu.et * kSKE;
      const int zend = tile_end ? n_split : seg + 1;
#pragma unroll
      for (int i = 0; i < TM; ++i) {
        const int t = t0 + ty * TM + i;
        if (t >= T) continue;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const int e = e0 + tx + 16 * j;
          if (e >= E || seg >= n_split) continue;
          part[((size_t)seg * T + t) * E + e] = make_float2(sum[i][j], -comp[i][j]);
          for (int z = seg + 1; z < zend; ++z)
            part[((size_t)z * T + t) * E + e] = make_float2(0.f, 0.f);
          sum[i][j] = comp[i][j] = 0.f;
        }
      }
    }
    cu.next(etiles, nc);
    stage = stage == kSKStages - 1 ? 0 : stage + 1;
  }
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

constexpr int kSelectThreads = 256;

// S_h (Eq. 1) for all experts into smem, readings: empty-history terms are 0; c_mode 0 uses
// C_i / sum C, c_mode 1 the raw C_i.  sum N is exact (int64), sum C a compensated fp32 sum of the
// fp32-rounded C_i; the three ratios are fp32 divisions (relative error ~3e-7, far inside the
// 1e-5 margin at which a token's selection counts as decided).  No fp64 arithmetic: it would run
// on GB300's narrow fp64 pipe in every block.  The selection kernel runs this before its
// dependency wait: the accounts are at least two launches old (the router-score kernel comes
// between), and every kernel lets its dependent start only after its own wait.  The loads bypass
// L1 (ld.global.cg), which may still hold an earlier call's lines before the wait.
__device__ void history_score_block(const int64_t* accN, const double* accP, const double* accC,
                                    int E, const RouteParams& rp, float* s_h) {
  __shared__ long long red_n[kSelectThreads / 32];
  __shared__ float red_c[2][kSelectThreads / 32];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  long long n_sum = 0;
  float c_hi = 0.f, c_lo = 0.f;
  for (int e = tid; e < E; e += blockDim.x) {
    n_sum += (long long)__ldcg(accN + e);
    df_add(c_hi, c_lo, (float)__ldcg(accC + e));
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    n_sum += __shfl_xor_sync(0xffffffffu, n_sum, o);
    const float oh = __shfl_xor_sync(0xffffffffu, c_hi, o);
    const float ol = __shfl_xor_sync(0xffffffffu, c_lo, o);
    df_add(c_hi, c_lo, oh, ol);
  }
  if (lane == 0) {
    red_n[warp] = n_sum;
    red_c[0][warp] = c_hi;
    red_c[1][warp] = c_lo;
  }
  __syncthreads();
  if (tid == 0) {
    long long a = 0;
    float bh = 0.f, bl = 0.f;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) {
      a += red_n[w];
      df_add(bh, bl, red_c[0][w], red_c[1][w]);
    }
    red_n[0] = a;
    red_c[0][0] = bh + bl;
  }
  __syncthreads();
  const float total_n = (float)red_n[0];
  const float total_c = red_c[0][0];
  for (int e = tid; e < E; e += blockDim.x) {
    const long long ni = __ldcg(accN + e);
    const float n = (float)ni;
    const float a = ni > 0 ? n / total_n : 0.f;
    const float b = ni > 0 ? (float)__ldcg(accP + e) / n : 0.f;
    const float ce = (float)__ldcg(accC + e);
    float c;
    if (rp.c_mode == EAT_C_RAW) c = ce;
    else c = total_c > 0.f ? ce / total_c : 0.f;
    s_h[e] = rp.w1 * a + rp.w2 * b + rp.w3 * c;
  }
  __syncthreads();
}

// Warp-wide bitonic sort of the 32 x EPL (key, index) pairs a warp holds (element j * 32 + lane
// in register j of that lane), ascending by key and, for equal keys, by index: the order the
// selection's rank rules use.  The network is fixed (no data-dependent branches on the warp's
// control flow); strides below 32 exchange across lanes, larger ones between a lane's registers.
template <int EPL>
__device__ __forceinline__ void warp_sort_pairs(float (&k)[EPL], int (&x)[EPL], int lane) {
  const unsigned full = 0xffffffffu;
#pragma unroll
  for (int size = 2; size <= 32 * EPL; size <<= 1) {
#pragma unroll
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      if (stride >= 32) {
        const int js = stride >> 5;
#pragma unroll
        for (int j = 0; j < EPL; ++j) {
          if ((j & js) == 0) {
            const int jp = j | js;
            const bool up = ((j * 32 + lane) & size) == 0;
            const bool gt = k[j] > k[jp] || (k[j] == k[jp] && x[j] > x[jp]);
            if (gt == up) {
              const float tk = k[j];
              k[j] = k[jp];
              k[jp] = tk;
              const int tx = x[j];
              x[j] = x[jp];
              x[jp] = tx;
            }
          }
        }
      } else {
#pragma unroll
        for (int j = 0; j < EPL; ++j) {
          const float ok = __shfl_xor_sync(full, k[j], stride);
          const int ox = __shfl_xor_sync(full, x[j], stride);
          const bool up = ((j * 32 + lane) & size) == 0;
          const bool keep_min = up == ((lane & stride) == 0);
          const bool other_less = ok < k[j] || (ok == k[j] && ox < x[j]);
          if (keep_min == other_less) {
            k[j] = ok;
            x[j] = ox;
          }
        }
      }
    }
  }
}
// Element r (0-based) of the sorted pairs, broadcast to the warp.
template <int EPL>
__device__ __forceinline__ void sorted_at(const float (&k)[EPL], const int (&x)[EPL], int r,
                                          float& kr, int& xr) {
  float kv = 0.f;
  int xv = 0;
#pragma unroll
  for (int j = 0; j < EPL; ++j)
    if (j == (r >> 5)) {
      kv = k[j];
      xv = x[j];
    }
  kr = __shfl_sync(0xffffffffu, kv, r & 31);
  xr = __shfl_sync(0xffffffffu, xv, r & 31);
}

template <int EPL>
__global__ void __launch_bounds__(kSelectThreads)
route_select_kernel(const float2* __restrict__ part, int n_split, const float* __restrict__ bias,
                    int T, int E, int K, const int64_t* __restrict__ accN,
                    const double* __restrict__ accP, const double* __restrict__ accC,
                    RouteParams rp, float inv_temp, int32_t* __restrict__ out_idx,
                    float* __restrict__ out_w, int32_t* __restrict__ out_k,
                    float* __restrict__ out_p) {
  __shared__ float s_h[kMaxExperts];
  history_score_block(accN, accP, accC, E, rp, s_h);
  pdl_wait();
  pdl_launch_dependents();

  const int lane = threadIdx.x & 31;
  const int warps = blockDim.x >> 5;
  const int t = blockIdx.x * warps + (threadIdx.x >> 5);
  if (t >= T) return;
  const unsigned full = 0xffffffffu;
  const float inv_e = 1.0f / (float)E;

  float p[EPL], I[EPL];
  bool valid[EPL];
  float hi[EPL], lo[EPL], bv[EPL];
#pragma unroll
  for (int i = 0; i < EPL; ++i) {
    const int e = lane + 32 * i;
    valid[i] = e < E;
    hi[i] = 0.f;
    lo[i] = 0.f;
    bv[i] = bias && valid[i] ? bias[e] : 0.f;
  }
  // the score partials in slice order, a chunk of slices' loads in flight before their sums
  constexpr int kChunk = EPL <= 1 ? 8 : (EPL <= 2 ? 4 : (EPL <= 4 ? 2 : 1));
  for (int sp0 = 0; sp0 < n_split; sp0 += kChunk) {
    float2 v[kChunk][EPL];
#pragma unroll
    for (int c = 0; c < kChunk; ++c)
#pragma unroll
      for (int i = 0; i < EPL; ++i)
        v[c][i] = sp0 + c < n_split && valid[i]
                      ? part[((size_t)(sp0 + c) * T + t) * E + lane + 32 * i]
                      : make_float2(0.f, 0.f);
#pragma unroll
    for (int c = 0; c < kChunk; ++c)
#pragma unroll
      for (int i = 0; i < EPL; ++i)
        if (sp0 + c < n_split && valid[i]) df_add(hi[i], lo[i], v[c][i].x, v[c][i].y);
  }
  float lmax = -INFINITY;
#pragma unroll
  for (int i = 0; i < EPL; ++i) {
    float z = -INFINITY;
    if (valid[i]) {
      if (bias) df_add(hi[i], lo[i], bv[i]);
      z = (hi[i] + lo[i]) * inv_temp;
    }
    p[i] = z;
    lmax = fmaxf(lmax, z);
  }
  // softmax (§3.2): p = exp(z - max) / sum
  const float m = warp_max(lmax);
  float ssum = 0.f;
#pragma unroll
  for (int i = 0; i < EPL; ++i) {
    p[i] = valid[i] ? expf(p[i] - m) : 0.f;
    ssum += p[i];
  }
  ssum = warp_sum(ssum);
  float psum = 0.f;
#pragma unroll
  for (int i = 0; i < EPL; ++i) {
    p[i] = valid[i] ? p[i] / ssum : 0.f;
    psum += p[i];
  }
  if (rp.opd_scale) {
    // §3.5 OPD reweighting: p'_i = s_i p_i / sum_j s_j p_j replaces p from here on
    float qs = 0.f;
#pragma unroll
    for (int i = 0; i < EPL; ++i) {
      p[i] = valid[i] ? p[i] * rp.opd_scale[lane + 32 * i] : 0.f;
      qs += p[i];
    }
    qs = warp_sum(qs);
    psum = 0.f;
#pragma unroll
    for (int i = 0; i < EPL; ++i) {
      p[i] = valid[i] ? p[i] / qs : 0.f;
      psum += p[i];
    }
  }
  // A NaN probability (non-finite hidden state or router weights) loses every comparison, which
  // would select every expert in the rank-based modes: such a token selects none (reading R15 of
  // the oracle), its output row is NaN and it adds nothing to the accounts.
  bool nan_p = false;
#pragma unroll
  for (int i = 0; i < EPL; ++i) nan_p |= valid[i] && isnan(p[i]);
  const bool bad = __any_sync(full, nan_p);
  // Eq. 3-4: mean and population standard deviation of g = p
  const float mu = warp_sum(psum) * inv_e;
  float dev = 0.f;
#pragma unroll
  for (int i = 0; i < EPL; ++i) {
    const float dlt = valid[i] ? p[i] - mu : 0.f;
    dev += dlt * dlt;
  }
  const float sigma = sqrtf(warp_sum(dev) * inv_e);
  // Eq. 5, PPL adjustment and smoothing (§3.3)
  const float tau = fmaxf(rp.alpha1 * mu, mu - rp.alpha2 * sigma);
  float second = tau;  // same-call blend, or the stream's previous tau_final (temporal reading)
  if (rp.smoothing == EAT_SMOOTH_TEMPORAL && rp.tau_in) {
    const float prev = rp.tau_in[t];
    if (!isnan(prev)) second = prev;
  }
  float ppl_f = rp.ppl_factor;
  if (rp.ppl_sign_dev) {  // the sign eat_ppl_update wrote on the device (read after the wait)
    const int sg = __ldcg(rp.ppl_sign_dev);
    ppl_f = sg > 0 ? rp.ppl_up : (sg < 0 ? rp.ppl_down : 1.0f);
  }
  float tau_f = rp.kappa1 * (ppl_f * tau) + rp.kappa2 * second;

  if (rp.clamp) {
    // order statistics of p (ascending, ties by index; padding lanes sort last)
    float sk[EPL];
    int sx[EPL];
#pragma unroll
    for (int i = 0; i < EPL; ++i) {
      sk[i] = valid[i] ? p[i] : INFINITY;
      sx[i] = lane + 32 * i;
    }
    warp_sort_pairs<EPL>(sk, sx, lane);
    const float h_lo = (float)(E - 1) * rp.q_lo;
    const float h_hi = (float)(E - 1) * rp.q_hi;
    const int lo0 = (int)floorf(h_lo), hi0 = (int)floorf(h_hi);
    const int lo1 = min(lo0 + 1, E - 1), hi1 = min(hi0 + 1, E - 1);
    float v_lo0, v_lo1, v_hi0, v_hi1;
    int unused;
    sorted_at<EPL>(sk, sx, lo0, v_lo0, unused);
    sorted_at<EPL>(sk, sx, lo1, v_lo1, unused);
    sorted_at<EPL>(sk, sx, hi0, v_hi0, unused);
    sorted_at<EPL>(sk, sx, hi1, v_hi1, unused);
    const float q_lo = v_lo0 + (h_lo - (float)lo0) * (v_lo1 - v_lo0);
    const float q_hi = v_hi0 + (h_hi - (float)hi0) * (v_hi1 - v_hi0);
    tau_f = fminf(fmaxf(tau_f, q_lo), q_hi);
  }

  if (rp.tau_out && lane == 0) rp.tau_out[t] = tau_f;

  // Eq. 2 importance and Eq. 6 candidate set
  bool cand[EPL];
  int ncand = 0;
#pragma unroll
  for (int i = 0; i < EPL; ++i) {
    const int e = lane + 32 * i;
    I[i] = valid[i] ? (1.f - rp.beta) * p[i] + rp.beta * s_h[e] : -INFINITY;
    cand[i] = valid[i] && I[i] > tau_f;
    ncand += __popc(__ballot_sync(full, cand[i]));
  }
  bool sel[EPL];
  if (rp.mode != EAT_ROUTER_EAT) {
    // §4.1 baselines: rank by (p desc, index asc); Top-K keeps ranks < K, Top-P keeps the
    // smallest prefix whose cumulative probability reaches top_p (at most K)
    int r[EPL];
    float cum[EPL];
#pragma unroll
    for (int i = 0; i < EPL; ++i) {
      r[i] = 0;
      cum[i] = 0.f;
    }
#pragma unroll
    for (int jb = 0; jb < EPL; ++jb) {
      for (int jl = 0; jl < 32; ++jl) {
        const int ej = jb * 32 + jl;
        const float pj = __shfl_sync(full, p[jb], jl);
        if (ej < E) {
#pragma unroll
          for (int i = 0; i < EPL; ++i) {
            const int ei = lane + 32 * i;
            if (pj > p[i] || (pj == p[i] && ej < ei)) {
              r[i] += 1;
              cum[i] += pj;
            }
          }
        }
      }
    }
#pragma unroll
    for (int i = 0; i < EPL; ++i)
      sel[i] = valid[i] && r[i] < K && (rp.mode == EAT_ROUTER_TOPK || cum[i] < rp.top_p);
  } else if (ncand == 0) {
    // argmax I, lowest index on ties
    float bv = -INFINITY;
    int be = 0x7fffffff;
#pragma unroll
    for (int i = 0; i < EPL; ++i) {
      const int e = lane + 32 * i;
      if (valid[i] && (I[i] > bv || (I[i] == bv && e < be))) { bv = I[i]; be = e; }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float ov = __shfl_xor_sync(full, bv, o);
      const int oe = __shfl_xor_sync(full, be, o);
      if (ov > bv || (ov == bv && oe < be)) { bv = ov; be = oe; }
    }
#pragma unroll
    for (int i = 0; i < EPL; ++i) sel[i] = (lane + 32 * i) == be;
  } else if (ncand <= K) {
#pragma unroll
    for (int i = 0; i < EPL; ++i) sel[i] = cand[i];
  } else {
    // keep the K largest candidates by (I desc, index asc): sort (-I, index) ascending with the
    // non-candidates last and keep what does not come after the K-th pair
    float sk[EPL];
    int sx[EPL];
#pragma unroll
    for (int i = 0; i < EPL; ++i) {
      sk[i] = cand[i] ? -I[i] : INFINITY;
      sx[i] = lane + 32 * i;
    }
    warp_sort_pairs<EPL>(sk, sx, lane);
    float kk;
    int kx;
    sorted_at<EPL>(sk, sx, K - 1, kk, kx);
#pragma unroll
    for (int i = 0; i < EPL; ++i) {
      const float key = -I[i];
      const int ei = lane + 32 * i;
      sel[i] = cand[i] && (key < kk || (key == kk && ei <= kx));
    }
  }

  if (bad) {
#pragma unroll
    for (int i = 0; i < EPL; ++i) sel[i] = false;
  }
  // Eq. 7-8: renormalised gates over the selected experts, g = p
  float gs = 0.f;
#pragma unroll
  for (int i = 0; i < EPL; ++i) gs += sel[i] ? p[i] : 0.f;
  const float denom = warp_sum(gs) + rp.eps;
  const unsigned lt = (1u << lane) - 1u;
  int base = 0;
  const size_t row = (size_t)t * K;
#pragma unroll
  for (int i = 0; i < EPL; ++i) {
    const unsigned b = __ballot_sync(full, sel[i]);
    if (sel[i]) {
      const int pos = base + __popc(b & lt);
      out_idx[row + pos] = lane + 32 * i;
      out_w[row + pos] = p[i] / denom;
      if (out_p) out_p[row + pos] = p[i];
    }
    base += __popc(b);
  }
  if (lane >= base && lane < K) {
    out_idx[row + lane] = -1;
    out_w[row + lane] = 0.f;
    if (out_p) out_p[row + lane] = 0.f;
  }
  if (lane == 0) out_k[t] = base;
}

}  // namespace

namespace {

// CTAs of router_logits_sk_kernel resident per SM, and the SM count, of the current device (both
// queried once per device; concurrent first calls compute the same values)
struct SkDevice {
  std::atomic<int> ready{0};
  int sms = 0, per_sm = 0;
};
SkDevice g_sk_dev[64];

bool sk_device(int& sms, int& per_sm) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return false;
  SkDevice& D = g_sk_dev[dev];
  if (!D.ready.load(std::memory_order_acquire)) {
    int n = 0, b = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
        cudaFuncSetAttribute(router_logits_sk_kernel<kSKTM>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSKSmem) != cudaSuccess ||
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&b, router_logits_sk_kernel<kSKTM>,
                                                      SkCfg<kSKTM>::kThreads, kSKSmem) != cudaSuccess ||
        n < 1 || b < 1)
      return false;
    D.sms = n;
    D.per_sm = b;
    D.ready.store(1, std::memory_order_release);
  }
  sms = D.sms;
  per_sm = D.per_sm;
  return true;
}

// Grid and split slices of the stream-K router for a call; cap > 0 bounds the slices (a caller
// with fixed scratch).  A tile of nc units meets at most 1 + ceil((nc - 1) / m) CTA runs when every
// run holds at least m units; n_split is that bound (slices a tile does not use are zero pairs).
struct SkPlan {
  int grid = 0, n_split = 0;
};
bool sk_plan(int T, int d, int E, int cap, SkPlan& out) {
  int sms = 0, per_sm = 0;
  if (!sk_device(sms, per_sm)) return false;
  const long long nc = d / kChunkK;
  const long long tiles = (long long)((T + kSKT - 1) / kSKT) * ((E + kSKE - 1) / kSKE);
  const long long U = tiles * nc;
  long long G = std::min<long long>((long long)sms * per_sm, U / kSKMinUnits);
  G = std::max<long long>(1, std::min(G, U));
  auto bound = [&](long long g) {
    const long long m = U / g;
    return g == tiles && U % g == 0 ? 1LL : std::min(nc, 1 + (nc - 1 + m - 1) / m);
  };
  long long n = bound(G);
  if (cap > 0 && n > cap) {
    if (cap == 1) {
      G = tiles;  // every CTA one whole tile
    } else {
      const long long m_req = (nc - 1 + cap - 2) / (cap - 1);
      G = std::max<long long>(1, U / m_req);
    }
    n = bound(G);
  }
  out.grid = (int)G;
  out.n_split = (int)n;
  return true;
}

bool sk_eligible(int T, int d) { return T > kSmallT && d % kChunkK == 0; }

}  // namespace

int router_split(int T, int d, int E) {
  if (T <= kSmallT) return (d + kSmallSlice - 1) / kSmallSlice;
  if (sk_eligible(T, d)) {
    SkPlan pl;
    if (sk_plan(T, d, E, 0, pl)) return pl.n_split;
  }
  // enough CTAs for two waves, each slice at least 256 columns of d
  const long long tiles = (long long)((T + kTileT - 1) / kTileT) * ((E + kTileE - 1) / kTileE);
  int split = 1;
  while (tiles * split < 2 * 152 && d / (split * 2) >= 256 && split < 64) split *= 2;
  return split;
}

bool router_copies_x(const void* x, int x_bf16, const float* w_router, int T, int d) {
  const bool vec_ok = d % 4 == 0 && ((uintptr_t)x & 15) == 0 && ((uintptr_t)w_router & 15) == 0;
  return vec_ok && (T <= kSmallT || (x_bf16 && sk_eligible(T, d)));
}

cudaError_t launch_router_logits(const void* x, int x_bf16, const float* w_router, int T, int d,
                                 int E, int n_split, float2* part, cudaStream_t st, void* xcopy) {
  const bool vec_ok = d % 4 == 0 && ((uintptr_t)x & 15) == 0 && ((uintptr_t)w_router & 15) == 0;
  if (xcopy && (!router_copies_x(x, x_bf16, w_router, T, d) || ((uintptr_t)xcopy & 15) != 0))
    return cudaErrorInvalidValue;
  if (T <= kSmallT && vec_ok) {
    int per = (d + n_split - 1) / n_split;
    per = (per + 127) / 128 * 128;
    dim3 grid(T, n_split, (E + kLogitThreads / 32 - 1) / (kLogitThreads / 32));
    if (x_bf16)
      return launch_pdl(router_logits_small_kernel<__nv_bfloat16>, grid, dim3(kLogitThreads), 0,
                        st, (const __nv_bfloat16*)x, w_router, T, d, E, per, part,
                        (__nv_bfloat16*)xcopy);
    return launch_pdl(router_logits_small_kernel<float>, grid, dim3(kLogitThreads), 0, st,
                      (const float*)x, w_router, T, d, E, per, part, (float*)xcopy);
  }
  if (x_bf16 && sk_eligible(T, d) && vec_ok) {
    SkPlan pl;
    if (!sk_plan(T, d, E, n_split, pl)) return cudaErrorInvalidDevice;
    if (pl.n_split > n_split) return cudaErrorInvalidValue;
    return launch_pdl(router_logits_sk_kernel<kSKTM>, dim3(pl.grid), dim3(SkCfg<kSKTM>::kThreads),
                      kSKSmem, st, (const __nv_bfloat16*)x, w_router, T, d, E, n_split, part,
                      (__nv_bfloat16*)xcopy);
  }
  int per = (d + n_split - 1) / n_split;
  per = (per + kChunkK - 1) / kChunkK * kChunkK;
  dim3 grid((T + kTileT - 1) / kTileT, (E + kTileE - 1) / kTileE, n_split);
  if (x_bf16)
    return launch_pdl(router_logits_kernel<__nv_bfloat16>, grid, dim3(kLogitThreads), 0, st,
                      (const __nv_bfloat16*)x, w_router, T, d, E, per, part);
  return launch_pdl(router_logits_kernel<float>, grid, dim3(kLogitThreads), 0, st,
                    (const float*)x, w_router, T, d, E, per, part);
}

cudaError_t launch_route_select(const float2* part, int n_split, const float* b_router, int T,
                                int E, int K, const int64_t* accN, const double* accP,
                                const double* accC, RouteParams rp, int32_t* idx, float* w,
                                int32_t* k, float* psel, cudaStream_t st) {
  const int warps = kSelectThreads / 32;
  dim3 grid((T + warps - 1) / warps);
  const float inv_temp = (float)(1.0 / (double)rp.temperature);
#define EAT_SELECT(EPL)                                                                    \
  launch_pdl(route_select_kernel<EPL>, grid, dim3(kSelectThreads), 0, st, part, n_split,    \
             b_router, T, E, K, accN, accP, accC, rp, inv_temp, idx, w, k, psel)
  if (E <= 32) return EAT_SELECT(1);
  if (E <= 64) return EAT_SELECT(2);
  if (E <= 128) return EAT_SELECT(4);
  return EAT_SELECT(8);
#undef EAT_SELECT
}

}  // namespace eat
