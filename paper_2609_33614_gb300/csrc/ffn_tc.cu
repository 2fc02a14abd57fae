// Tensor-core expert FFN kernels for bf16 and e4m3-weight layers (the dominant cost of the EAT MoE
// layer): grouped SwiGLU expert GEMMs over the activated experts only (§3.4: an expert runs only
// on the tokens that selected it), written for sm_103a with tcgen05.mma (accumulators in TMEM),
// TMA tile loads into 128B-swizzled shared memory and mbarrier pipelines.
//
// Orientation ("swap AB"): a tile is 128 weight rows (output features of one expert) x BN tokens
// (16..128 rows of that expert's slot list), so decode calls with a handful of tokens still issue
// full M = 128 MMAs and simply stream the activated experts' weights.  Calls of 1024 tokens or more
// run on SM pairs instead (tc_pair_kernel below: M = 256 weight rows x 256 tokens per MMA).
//   gate/up kernel: D_gate = Wg[e, f0:f0+128, :] . Xperm[slots]^T and D_up likewise, both in TMEM;
//       the epilogue writes act[slot, f] = silu(D_gate) * D_up in bf16 (fp32 accumulation).
//   down kernel:    D = Wd[e, c0:c0+128, :] . act[slots]^T over a K slice: with split-K (decode)
//       fp32 partials opart[split][slot][c], summed in fixed order by the combine kernel; without
//       it, bf16 rows O[slot][c].
// Persistent CTAs (one per SM) walk the work units (token tile, feature tile, K slice) of all
// groups; the group sizes live on the device (written by the permute kernel), so no host sync.
// Warp roles: warp 0 lane 0 issues TMA; warp 1 owns TMEM and lane 0 issues MMAs; warps 2-5 (and
// 6-9 for e4m3 tiles of 64 or more tokens, each warp half of the tile's columns) drain TMEM
// (double-buffered accumulators, so the epilogue of tile i overlaps the MMAs of tile i + 1).
// Every mbarrier wait is bounded (2 s); on expiry the kernel records an error in the device status
// word, lets in-flight copies and MMAs finish, frees its TMEM and returns.
#include "ffn_tc.cuh"

#include <cuda.h>
#include <cudaTypedefs.h>

#include <cstring>
#include <mutex>
#include <vector>

namespace eat {

namespace {

constexpr int kBM = 128;                  // weight rows per tile (MMA M)
constexpr int kBK = 64;                   // 64 bf16 = 128 B: one 128B-swizzle row
constexpr int kBK8 = 128;                 // 128 e4m3 = 128 B: the same row for fp8 layers
constexpr int kNumBN = 4;
constexpr int kBNs[kNumBN] = {16, 32, 64, 128};  // single-SM token tiles; SM pairs load 128 per CTA
constexpr unsigned long long kWaitLimitNs = 2000000000ull;
constexpr int kSmemBudget = 220 * 1024;

// -------------------------------------------------------------------------------- PTX wrappers
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ unsigned long long globaltimer() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count));
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Bounded wait on the phase with the given parity.  Returns false when it gave up: because another
// role raised the CTA's abort flag (check_abort), or after kWaitLimitNs (then it raises the flag and
// records `code` in the device status word).
__device__ __noinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag,
                                       unsigned int* err, unsigned int code, bool check_abort,
                                       unsigned long long limit_ns = kWaitLimitNs) {
  if (mbar_try_wait(bar, parity)) return true;
  const unsigned long long t0 = globaltimer();
  for (;;) {
    if (mbar_try_wait(bar, parity)) return true;
    if (check_abort && *abort_flag) return false;
    if (globaltimer() - t0 > limit_ns) {
      *abort_flag = 1;
      atomicOr(err, code);
      return false;
    }
  }
}

// The bounded wait by all lanes of a warp, with one outcome for the whole warp (a lane that gave
// up makes every lane give up), so warp-synchronous code after it never sees diverged lanes.
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag,
                                          unsigned int* err, unsigned int code) {
  const bool ok = mbar_wait(bar, parity, abort_flag, err, code, true);
  return __all_sync(0xffffffffu, ok);
}

__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, uint64_t* bar,
                                            int c0, int c1) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4}], [%2];" ::"r"(smem_u32(dst)),
      "l"(map), "r"(smem_u32(bar)), "r"(c0), "r"(c1)
      : "memory");
}
// The proxy fence that orders bytes copied by cp.async (generic proxy) before the tensor core
// reads them (async proxy).
__device__ __forceinline__ void fence_proxy_async() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tmem_alloc(uint32_t* slot, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_u32(slot)),
               "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}
// D[tmem] (+)= A[smem desc] . B[smem desc]^T, both K-major, kind::f16 (bf16 in, fp32 accumulate)
__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc,
                                         uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// Arrive on `bar` once every MMA this thread issued so far has completed.
__device__ __forceinline__ void mma_commit(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          smem_u32(bar))
      : "memory");
}
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, "
      "%12, %13, %14, %15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
}
// D[tmem] (+)= A[smem desc] . B[smem desc]^T, both K-major, kind::f8f6f4 (e4m3 in, fp32
// accumulate; K = 32 per instruction, 32 bytes of each 128-byte row like the bf16 form).
__device__ __forceinline__ void mma_e4m3(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc,
                                         uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n}\n" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void tmem_wait_ld() {
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// Shared-memory matrix descriptor: K-major operand, 128B swizzle, rows of 128 B, 8-row groups
// 1024 B apart (SBO); LBO unused for swizzled K-major layouts; version field 1 (bit 46).
__device__ __forceinline__ uint64_t sdesc_k128(uint32_t saddr) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFF) >> 4);
  d |= (uint64_t)1 << 16;
  d |= (uint64_t)(1024 >> 4) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
}
// Instruction descriptor, kind::f16: D fp32, A and B bf16, both K-major, M = 128, N = n.
__host__ __device__ constexpr uint32_t idesc_bf16(int n) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(n >> 3) << 17) |
         ((uint32_t)(kBM >> 4) << 24);
}
// Instruction descriptor, kind::f8f6f4: D fp32, A and B e4m3 (format code 0), both K-major,
// M = 128, N = n.
__host__ __device__ constexpr uint32_t idesc_e4m3(int n) {
  return (1u << 4) | ((uint32_t)(n >> 3) << 17) | ((uint32_t)(kBM >> 4) << 24);
}

__host__ __device__ constexpr int tmem_cols_for(int c) {
  return c <= 32 ? 32 : c <= 64 ? 64 : c <= 128 ? 128 : c <= 256 ? 256 : 512;
}

// Kernel modes: the down projection (one A tile, plain epilogue); gate/up with two accumulators
// (gate and up A tiles of 128 rows against one B tile, single-SM kernel); gate/up interleaved (one
// A tile of 64 gate rows over the 64 up rows of the same features, one accumulator: an MMA covers
// both projections of 64 features, and the epilogue pairs the gate and up warps of each feature;
// SM-pair kernel).
enum : int { kModeDown = 0, kModeGateUp = 1, kModeGateUpIL = 2 };

template <int BN, int MODE, bool W8 = false>
struct Cfg {
  static_assert(MODE == kModeDown || MODE == kModeGateUp, "single-SM kernel modes");
  static constexpr bool kGateUp = MODE == kModeGateUp;
  static constexpr int kNA = kGateUp ? 2 : 1;
  static constexpr int kNB = W8 ? 2 : 1;         // fp8: the B tile's e4m3 hi and lo parts
  static constexpr int kKB = W8 ? kBK8 : kBK;    // K elements of a k-block (128 B per row)
  static constexpr int kABytes = kBM * 128;
  static constexpr int kBBytes = BN * 128;
  static constexpr int kSubBytes = kNA * kABytes + kNB * kBBytes;  // one k-block's tiles
  // k-blocks per pipeline stage: a stage completes on one barrier phase, which costs ~0.6 µs
  // however few bytes it carries, so a stage carries two k-blocks wherever three such stages fit
  static constexpr int kKPS = 6 * kSubBytes <= kSmemBudget - 2048 ? 2 : 1;
  // e4m3 tiles of 64 or more tokens are drained by two warps per TMEM lane quarter (one per half
  // of the tile's columns), so an accumulator buffer returns to the MMA issuer sooner (e4m3
  // prefill +20 %; the bf16 gathering gate/up at 128-token tiles was slower with eight)
  static constexpr int kEpiWarps = (W8 && BN >= 64) ? 8 : 4;
  static constexpr int kThreads = 64 + 32 * kEpiWarps;
  static constexpr int kStageBytes = kKPS * kSubBytes;
  // fp8: the hi and lo B tiles sit back to back in the stage, so one MMA of N = BN + n covers both
  // (hi in accumulator columns [0, BN), lo in [BN, BN + n)) and reads its A slice once, where the
  // double-buffered accumulators fit in TMEM (gate/up up to 64 tokens, down up to 128)
  static constexpr bool kFuse = W8 && 4 * kNA * BN <= 512;
  static constexpr int kProjCols = kFuse ? 2 * BN : BN;  // accumulator columns per projection
  static constexpr int kAccCols = kNA * kProjCols;
  static constexpr int kStagesRaw = (kSmemBudget - 2048) / kStageBytes;
  static constexpr int kStages = kStagesRaw > 12 ? 12 : kStagesRaw;
  static constexpr int kTmemCols = tmem_cols_for(2 * kAccCols);
  static constexpr int kSmemBytes = 1024 + kStages * kStageBytes + 512;
  static_assert(kSmemBytes <= 227 * 1024, "shared memory of one CTA");
};

struct TcArgs {
  int n_groups;
  const int32_t* row_offs;   // [G+1] slot ranges per group, or nullptr: uniform_rows each
  const int32_t* tile_offs;  // [G+1] prefix of token tiles, or nullptr: uniform
  int uniform_rows;
  int b_shift_per_group;     // B row = slot - g * b_shift_per_group
  int a_rows_per_group;      // A row = g * a_rows_per_group + m0
  int M;                     // output features per group
  int m_tile;                // output features per unit (128, or 64 for interleaved gate/up)
  int m_tiles;
  int kblocks;
  int n_split;
  int kb_per_split;
  void* out;
  long long split_stride;    // elements between split slices of the fp32 output
  int out_bf16;              // down kernel without split-K: write bf16 rows instead of fp32
  const int32_t* b_rows;     // gather mode: slot -> token; B rows are copied from bx by the warp
  const __nv_bfloat16* bx;   // gather mode: token rows [T, row stride kblocks * 64] (16-bit)
  const float* scale0;       // fp8 weights: per-row scales of the A matrix (gate, or down)
  const float* scale1;       // fp8 weights: per-row scales of the up matrix
  const float* bscale;       // fp8: per-row scales of the B operand, indexed like its rows
  int b_lo_rows;             // fp8: row offset of the B operand's lo plane in its tensor map
  int prefetch_a;            // the group layout was written two or more launches back: issue the
                             // first stages' weight loads before waiting for the previous kernel
  int gate_first;            // 16-row interleaved gate/up A tile: the gate rows come first
  unsigned int* err;
};

struct Unit {
  int g, slot0, nrows, m0, kb0, kb1, split;
};

// The call's group offsets (row_offs, tile_offs), from global memory or a CTA's shared copy.
struct Offs {
  const int32_t* row;   // nullptr: uniform groups
  const int32_t* tile;  // nullptr: uniform groups
};
constexpr int kMaxGroups = 256;  // n_experts is at most 256

// All threads of the CTA: the group offsets into shared memory (one round trip instead of the
// dependent loads of a binary search per unit decode); the caller synchronises before use.  The
// loads bypass L1 (ld.global.cg): before the CTA's dependency wait, this SM's L1 may still hold
// the lines of an earlier call's offsets, while L2 holds the permute's completed writes.
__device__ __forceinline__ Offs stage_offsets(const TcArgs& a, int32_t* s_row, int32_t* s_tile) {
  for (int i = threadIdx.x; i <= a.n_groups; i += blockDim.x) {
    if (a.row_offs) s_row[i] = __ldcg(a.row_offs + i);
    if (a.tile_offs) s_tile[i] = __ldcg(a.tile_offs + i);
  }
  return {a.row_offs ? s_row : nullptr, a.tile_offs ? s_tile : nullptr};
}

template <int BN>
__device__ __forceinline__ Unit decode_unit(const TcArgs& a, int u, Offs o) {
  Unit w;
  w.split = u % a.n_split;
  const int r = u / a.n_split;
  const int mi = r % a.m_tiles;
  const int tl = r / a.m_tiles;
  int g, j;
  if (o.tile) {
    int lo = 0, hi = a.n_groups - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (o.tile[mid] <= tl) lo = mid;
      else hi = mid - 1;
    }
    g = lo;
    j = tl - o.tile[lo];
  } else {
    const int tpg = (a.uniform_rows + BN - 1) / BN;
    g = tl / tpg;
    j = tl % tpg;
  }
  const int beg = o.row ? o.row[g] : g * a.uniform_rows;
  const int end = o.row ? o.row[g + 1] : (g + 1) * a.uniform_rows;
  w.g = g;
  w.slot0 = beg + j * BN;
  w.nrows = min(BN, end - w.slot0);
  w.m0 = mi * a.m_tile;
  w.kb0 = w.split * a.kb_per_split;
  w.kb1 = min(a.kblocks, w.kb0 + a.kb_per_split);
  return w;
}

// A CTA's share of the work: units blockIdx.x, + gridDim.x, ...  (Units are handed out in rounds;
// an even split of all units' k-blocks over the CTAs, with the split units finished through fp32
// partials, measured within 1 % on decode calls: the SMs' streaming rates differ by about 10 %,
// and the CTA finishing a split unit would wait on another CTA of the grid.)
template <int BN>
struct UnitIter {
  int units, u;
  Offs o;
  __device__ UnitIter(int units_, Offs o_) : units(units_), u(blockIdx.x), o(o_) {}
  __device__ bool next(const TcArgs& a, Unit& w) {
    if (u >= units) return false;
    w = decode_unit<BN>(a, u, o);
    u += gridDim.x;
    return true;
  }
};

// silu(g) = g / (1 + e^-g) with the hardware exponential and an approximate division: relative
// error about 1e-6, far below the bf16 rounding of the activation it feeds (4e-3).  For g below
// about -88 the denominator overflows to infinity and the quotient is 0, the function's limit.
__device__ __forceinline__ float silu_f(float g) { return __fdividef(g, 1.0f + __expf(-g)); }

// W8 (fp8 layers): the weights stay e4m3 all the way to the tensor core.  The B operand arrives
// as two e4m3 planes per row (hi and lo, with hi + lo the row divided by its power-of-two scale,
// written by split_e4m3_kernel); a k-block holds the e4m3 A tiles of 128 elements and the hi and
// lo B tiles, every k-step issues W . hi and W . lo into the same fp32 accumulator
// (kind::f8f6f4), and the epilogue multiplies by the weight row's scale and the B row's scale.
template <int BN, int MODE, bool W8>
__global__ void __launch_bounds__(Cfg<BN, MODE, W8>::kThreads, 1)
tc_ffn_kernel(const __grid_constant__ CUtensorMap mapA0, const __grid_constant__ CUtensorMap mapA1,
              const __grid_constant__ CUtensorMap mapB, const TcArgs args) {
  using C = Cfg<BN, MODE, W8>;
  constexpr bool GATEUP = C::kGateUp;
  constexpr int S = C::kStages;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint64_t* full = (uint64_t*)(smem + S * C::kStageBytes);
  uint64_t* empty = full + S;
  uint64_t* tfull = empty + S;
  uint64_t* tempty = tfull + 2;
  uint64_t* mma_done = tempty + 2;
  uint32_t* tmem_slot = (uint32_t*)(mma_done + 1);
  volatile int* abort_flag = (volatile int*)(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], args.b_rows ? 2 : 1);  // + the gathered rows' arrival
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tfull[b], 1);
      mbar_init(&tempty[b], C::kEpiWarps);
    }
    mbar_init(mma_done, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) tmem_alloc(tmem_slot, C::kTmemCols);
  if (threadIdx.x == 32) {
    asm volatile("prefetch.tensormap [%0];" ::"l"(&mapA0) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(&mapB) : "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  // A tiles of one k-block: one 128-row box, or the gate and up boxes of the two accumulators
  auto load_a = [&](uint8_t* st, uint64_t* bar, int kb, int a_row) {
    tma_load_2d(st, &mapA0, bar, kb * C::kKB, a_row);
    if (GATEUP) tma_load_2d(st + C::kABytes, &mapA1, bar, kb * C::kKB, a_row);
  };
  __shared__ int32_t s_row[kMaxGroups + 1], s_tile[kMaxGroups + 1];
  Offs go{nullptr, nullptr};
  auto count_units = [&]() {
    const int total_tiles = go.tile ? go.tile[args.n_groups]
                                    : args.n_groups * ((args.uniform_rows + BN - 1) / BN);
    return total_tiles * args.m_tiles * args.n_split;
  };

  // The weights do not depend on the previous kernel, and the group layout (permute output) is at
  // least two launches old when the host sets prefetch_a (every launch only lets its dependent
  // start after its own wait): the producer fills the first stages' A tiles while the previous
  // kernel finishes; the B tiles of those stages follow after the wait.
  int pre = 0;  // stages whose A tiles are in flight
  const bool early = args.prefetch_a && !args.b_rows;  // (gathering launches follow the permute)
  if (early) {
    go = stage_offsets(args, s_row, s_tile);
    __syncthreads();
  }
  if (early && warp == 0 && lane == 0) {
    UnitIter<BN> it_p(count_units(), go);
    for (Unit w; pre < S && it_p.next(args, w);) {
      const int a_row = w.g * args.a_rows_per_group + w.m0;
      for (int kb = w.kb0; kb < w.kb1 && pre < S; kb += C::kKPS, ++pre) {
        const int nk = min(C::kKPS, w.kb1 - kb);  // k-blocks of this stage
        mbar_expect_tx(&full[pre], nk * C::kSubBytes);
        for (int j = 0; j < nk; ++j)
          load_a(smem + pre * C::kStageBytes + j * C::kSubBytes, &full[pre], kb + j, a_row);
      }
    }
  }
  // from here on the CTA reads what the previous kernel wrote
  pdl_wait();
  pdl_launch_dependents();
  if (!early) {
    go = stage_offsets(args, s_row, s_tile);
    __syncthreads();
  }
  const int units = count_units();

  if (GATEUP && !W8 && warp == 0 && args.b_rows) {
    // ------------------------------------------------------------ producer, gathered tokens:
    // lane 0 issues the weight TMA; all lanes copy the tile's token rows from x with 16-byte
    // cp.async into the 128B-swizzled B tile of each k-block of the stage (lane l: column chunk
    // l % 8 of rows l / 8 + 4 i).  A stage's rows are released LAG stages later: wait for the
    // lane's own copies, fence the async proxy, and one arrive per warp on the stage's full
    // barrier.
    constexpr int PER = BN / 4;
    constexpr int LAG = S > 2 ? S - 2 : 1;
    const unsigned fullmask = 0xffffffffu;
    const int cc = lane & 7, r0 = lane >> 3;
    const size_t ld = (size_t)args.kblocks * kBK;
    int stage = 0;
    uint32_t phase = 0;
    long long it = 0, released = 0;
    bool ok = true;
    UnitIter<BN> it_u(units, go);
    for (Unit w; ok && it_u.next(args, w);) {
      const int a_row = w.g * args.a_rows_per_group + w.m0;
      int tok[PER];
#pragma unroll
      for (int i = 0; i < PER; ++i) {
        const int r = r0 + 4 * i;
        tok[i] = r < w.nrows ? args.b_rows[w.slot0 + r] : -1;
      }
      for (int kb = w.kb0; kb < w.kb1; kb += C::kKPS) {
        const int nk = C::kKPS == 1 ? 1 : min(C::kKPS, w.kb1 - kb);  // k-blocks of this stage
        bool okw = true;
        if (lane == 0) okw = mbar_wait(&empty[stage], phase ^ 1u, abort_flag, args.err, 1u, true);
        okw = __shfl_sync(fullmask, okw ? 1 : 0, 0) != 0;
        if (!okw) {
          ok = false;
          break;
        }
        uint8_t* st = smem + stage * C::kStageBytes;
        if (lane == 0) {
          mbar_expect_tx(&full[stage], nk * C::kNA * C::kABytes);
#pragma unroll
          for (int j = 0; j < C::kKPS; ++j)
            if (j < nk) load_a(st + j * C::kSubBytes, &full[stage], kb + j, a_row);
        }
#pragma unroll
        for (int j = 0; j < C::kKPS; ++j) {
          if (j >= nk) break;
          const uint32_t sb = smem_u32(st + j * C::kSubBytes + C::kNA * C::kABytes);
#pragma unroll
          for (int i = 0; i < PER; ++i) {
            if (tok[i] >= 0) {
              const int r = r0 + 4 * i;
              cp_async16(sb + r * 128 + ((cc ^ (r & 7)) << 4),
                         args.bx + (size_t)tok[i] * ld + (kb + j) * kBK + cc * 8);
            }
          }
        }
        cp_async_commit();
        ++it;
        if (it - released > LAG) {
          cp_async_wait<LAG>();
          fence_proxy_async();
          __syncwarp();
          if (lane == 0) mbar_arrive(&full[released % S]);
          ++released;
        }
        if (++stage == S) {
          stage = 0;
          phase ^= 1u;
        }
      }
    }
    // release the stages still held (also on abort, so their barriers can complete), then let the
    // weight copies in flight land before the CTA may exit
    cp_async_wait<0>();
    fence_proxy_async();
    __syncwarp();
    if (lane == 0) {
      for (; released < it; ++released) mbar_arrive(&full[released % S]);
      const long long first = it > S ? it - S : 0;
      for (long long i = first; i < it; ++i)
        mbar_wait(&full[i % S], (uint32_t)((i / S) & 1), abort_flag, args.err, 2u, false);
    }
  } else if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------------------ TMA producer
      int stage = 0;
      uint32_t phase = 0;
      long long issued = 0;
      bool ok = true;
      UnitIter<BN> it_u(units, go);
      for (Unit w; ok && it_u.next(args, w);) {
        const int a_row = w.g * args.a_rows_per_group + w.m0;
        const int b_row = w.slot0 - w.g * args.b_shift_per_group;
        for (int kb = w.kb0; kb < w.kb1; kb += C::kKPS) {
          const int nk = min(C::kKPS, w.kb1 - kb);
          uint8_t* st = smem + stage * C::kStageBytes;
          if (issued >= pre) {  // (the first `pre` stages: A already in flight, stage unused)
            if (!mbar_wait(&empty[stage], phase ^ 1u, abort_flag, args.err, 1u, true)) {
              ok = false;
              break;
            }
            mbar_expect_tx(&full[stage], nk * C::kSubBytes);
            for (int j = 0; j < nk; ++j) load_a(st + j * C::kSubBytes, &full[stage], kb + j, a_row);
          }
          for (int j = 0; j < nk; ++j) {
            uint8_t* sbt = st + j * C::kSubBytes + C::kNA * C::kABytes;
            const int kx = (kb + j) * C::kKB;
            tma_load_2d(sbt, &mapB, &full[stage], kx, b_row);
            if (W8) tma_load_2d(sbt + C::kBBytes, &mapB, &full[stage], kx, b_row + args.b_lo_rows);
          }
          ++issued;
          if (++stage == S) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      // let the copies still in flight land before the CTA may exit
      const long long first = issued > S ? issued - S : 0;
      for (long long i = first; i < issued; ++i)
        mbar_wait(&full[i % S], (uint32_t)((i / S) & 1), abort_flag, args.err, 2u, false);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ------------------------------------------------------------ MMA issuer
      int stage = 0;
      uint32_t phase = 0;
      int local = 0;
      bool ok = true;
      UnitIter<BN> it_u(units, go);
      for (Unit w; ok && it_u.next(args, w); ++local) {
        const int buf = local & 1;
        const uint32_t tph = (uint32_t)((local >> 1) & 1);
        if (!mbar_wait(&tempty[buf], tph ^ 1u, abort_flag, args.err, 4u, true)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d0 = tmem_base + (uint32_t)(buf * C::kAccCols);
        const uint32_t d1 = d0 + C::kProjCols;
        // MMA width: the tile's rows rounded up to 16 (a partial tile computes no padding; the
        // fused fp8 MMA spans the hi tile's BN rows and the lo tile's first n)
        const int n_mma = min(BN, (w.nrows + 15) & ~15);
        const uint32_t idesc = !W8       ? idesc_bf16(n_mma)
                               : C::kFuse ? idesc_e4m3(BN + n_mma)
                                          : idesc_e4m3(n_mma);
        for (int kb = w.kb0; kb < w.kb1; kb += C::kKPS) {
          const int nk = min(C::kKPS, w.kb1 - kb);
          if (!mbar_wait(&full[stage], phase, abort_flag, args.err, 8u, true)) {
            ok = false;
            break;
          }
          tc_fence_after();
#pragma unroll
          for (int j = 0; j < C::kKPS; ++j) {
            if (j >= nk) break;
            const uint32_t sa0 = smem_u32(smem + stage * C::kStageBytes + j * C::kSubBytes);
            const uint32_t sa1 = sa0 + C::kABytes;
            const uint32_t sb = sa0 + C::kNA * C::kABytes;
            // four k-steps of 32 bytes per 128-byte row: 16 bf16 or 32 e4m3 elements each
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              const uint64_t da0 = sdesc_k128(sa0 + k * 32), db = sdesc_k128(sb + k * 32);
              const uint32_t acc = (kb > w.kb0 || j > 0 || k > 0) ? 1u : 0u;
              if constexpr (C::kFuse) {
                mma_e4m3(d0, da0, db, idesc, acc);
                if (C::kNA == 2) mma_e4m3(d1, sdesc_k128(sa1 + k * 32), db, idesc, acc);
              } else if constexpr (W8) {
                const uint64_t dl = sdesc_k128(sb + C::kBBytes + k * 32);
                mma_e4m3(d0, da0, db, idesc, acc);
                mma_e4m3(d0, da0, dl, idesc, 1u);
                if (C::kNA == 2) {
                  const uint64_t da1 = sdesc_k128(sa1 + k * 32);
                  mma_e4m3(d1, da1, db, idesc, acc);
                  mma_e4m3(d1, da1, dl, idesc, 1u);
                }
              } else {
                mma_bf16(d0, da0, db, idesc, acc);
                if (C::kNA == 2) mma_bf16(d1, sdesc_k128(sa1 + k * 32), db, idesc, acc);
              }
            }
          }
          mma_commit(&empty[stage]);
          if (++stage == S) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        mma_commit(&tfull[buf]);
      }
      // no MMA may still be running when TMEM is freed
      mma_commit(mma_done);
      mbar_wait(mma_done, 0u, abort_flag, args.err, 16u, false);
    }
  } else {
    // ------------------------------------------------- epilogue (warps 2 .. 2 + kEpiWarps - 1)
    const int q = warp & 3;  // TMEM lane quarter this warp may access
    const int row = 32 * q + lane;
    constexpr int kCols = BN / (C::kEpiWarps / 4);  // the tile columns of one warp
    const int cbeg = ((warp - 2) >> 2) * kCols;
    int local = 0;
    UnitIter<BN> it_u(units, go);
    for (Unit w; it_u.next(args, w); ++local) {
      const int buf = local & 1;
      const uint32_t tph = (uint32_t)((local >> 1) & 1);
      if (!warp_wait(&tfull[buf], tph, abort_flag, args.err, 32u)) break;
      tc_fence_after();
      const uint32_t tbase = tmem_base + ((uint32_t)(32 * q) << 16) + (uint32_t)(buf * C::kAccCols);
      const int f = w.m0 + row;
      const bool fok = f < args.M;
      float s0 = 1.0f, s1 = 1.0f;  // fp8 weights: the row scales of the A matrices
      if (W8 && fok) {
        const size_t ar = (size_t)w.g * args.a_rows_per_group + f;
        s0 = args.scale0[ar];
        if (GATEUP) s1 = args.scale1[ar];
      }
      const float* bsc = W8 ? args.bscale + (w.slot0 - w.g * args.b_shift_per_group) : nullptr;
      const int cend = min(cbeg + kCols, w.nrows);
      for (int c0 = cbeg; c0 < cend; c0 += 16) {
        uint32_t g[16], up[16];
        tmem_ld16(tbase + c0, g);
        if (GATEUP) tmem_ld16(tbase + C::kProjCols + c0, up);
        if constexpr (C::kFuse) {  // + the lo parts' columns
          uint32_t g2[16], up2[16];
          tmem_ld16(tbase + BN + c0, g2);
          if (GATEUP) tmem_ld16(tbase + C::kProjCols + BN + c0, up2);
          tmem_wait_ld();
#pragma unroll
          for (int c = 0; c < 16; ++c) {
            g[c] = __float_as_uint(__uint_as_float(g[c]) + __uint_as_float(g2[c]));
            if (GATEUP) up[c] = __float_as_uint(__uint_as_float(up[c]) + __uint_as_float(up2[c]));
          }
        }
        tmem_wait_ld();
        if (fok) {
#pragma unroll
          for (int c = 0; c < 16; ++c) {
            if (c0 + c < w.nrows) {
              const size_t slot = (size_t)(w.slot0 + c0 + c);
              const float sc = W8 ? bsc[c0 + c] : 1.0f;
              const float gv = W8 ? __uint_as_float(g[c]) * (s0 * sc) : __uint_as_float(g[c]);
              if (GATEUP) {
                const float uv = W8 ? __uint_as_float(up[c]) * (s1 * sc) : __uint_as_float(up[c]);
                ((__nv_bfloat16*)args.out)[slot * args.M + f] = __float2bfloat16_rn(silu_f(gv) * uv);
              } else if (args.out_bf16) {
                ((__nv_bfloat16*)args.out)[slot * args.M + f] = __float2bfloat16_rn(gv);
              } else {
                ((float*)args.out)[(size_t)w.split * args.split_stride + slot * args.M + f] = gv;
              }
            }
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty[buf]);
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem_base, C::kTmemCols);
}

// ------------------------------------------------------------ SM-pair kernels (cta_group::2)
// Large calls run on pairs of SMs (2-CTA clusters).  The pair issues M = 256 x N = 256 MMAs: each
// CTA holds 128 rows of A (weight rows) and 128 of the tile's 256 token rows of B, so a k-block is
// 32 KB per SM for the flops the single-SM kernel stages in 48 KB; a pipeline stage holds two
// k-blocks and three stages are in flight.  Rank 0 of the pair
// issues the MMAs (tcgen05.mma.cta_group::2) and commits them to the barriers of both CTAs; both
// CTAs load their halves with TMA completing on rank 0's full barrier (rank 0 expects the bytes
// of both); each CTA drains its own TMEM rows, and rank 0 reuses an accumulator buffer once the
// epilogues of both CTAs released it.  Modes: the down projection (256 output features per unit)
// and the interleaved gate/up (each CTA the gate and up rows of 64 features, 128 features per
// unit: alternating in groups of 16 rows, or 64 gate rows over the 64 up rows; see IL4 below).
// The MMA width is the unit's token rows rounded up to 32 (each CTA loads half of it), so a
// partial tile computes no padding beyond that.
constexpr int kPairBN = 256;
constexpr int kPairRows = kPairBN / 2;

template <int MODE, bool IL4 = false>
struct PairCfg {
  static constexpr bool kIL = MODE == kModeGateUpIL;
  static constexpr int kABytes = kBM * kBK * 2;
  static constexpr int kBBytes = kPairRows * kBK * 2;
  // k-blocks per pipeline stage: each stage completes on one barrier phase, and a phase costs
  // ~0.6 µs however few bytes it carries, so a stage carries two k-blocks' A and B tiles (64 KB
  // per CTA)
  static constexpr int kKPS = 2;
  static constexpr int kSubBytes = kABytes + kBBytes;  // one k-block's A and B tiles
  static constexpr int kStageBytes = kKPS * kSubBytes;
  // TMEM is drained by two warps per lane quarter, one per half of the 256 token columns: the
  // accumulator buffer goes back to the MMA issuer in half the time (10 warps in all)
  static constexpr int kEpiWarps = 8;
  static constexpr int kThreads = 64 + 32 * kEpiWarps;
  // exchange buffers of the 4 (feature half, column half) warp pairs: 2 buffers x gate and up x
  // 16 columns x 32 lanes (not with the 16-row interleave, whose warps pair gate and up by shuffles)
  static constexpr int kXchgFloats = (kIL && !IL4) ? 4 * 2 * 2 * 16 * 32 : 0;
  // the whole 227 KB a CTA may hold: 1 KB of alignment slack and 256 B of barriers besides the
  // stages (three, beside the gate/up exchange buffers too)
  static constexpr int kStagesRaw = (227 * 1024 - 1024 - 256 - kXchgFloats * 4) / kStageBytes;
  static constexpr int kStages = kStagesRaw > 8 ? 8 : kStagesRaw;
  static constexpr int kAccCols = kPairBN;
  static constexpr int kTmemCols = 512;
  static constexpr int kSmemBytes = 1024 + kStages * kStageBytes + kXchgFloats * 4 + 256;
  static constexpr int kFeat = kIL ? 64 : 128;  // output features of one CTA in a unit
  static_assert(kSmemBytes <= 227 * 1024, "shared memory of one CTA");
};

__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
// Address of the same shared variable in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t map_rank(uint32_t saddr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(saddr), "r"(rank));
  return r;
}
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;"
               ::: "memory");
}
// TMA load into this CTA's shared memory, completing on an mbarrier of either CTA of the pair.
__device__ __forceinline__ void tma_load_2d_pair(void* dst, const CUtensorMap* map,
                                                 uint32_t bar_cluster, int c0, int c1) {
  asm volatile(
      "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4}], [%2];" ::"r"(smem_u32(dst)),
      "l"(map), "r"(bar_cluster), "r"(c0), "r"(c1)
      : "memory");
}
// The same for a 4D tensor map (coordinates innermost first).
__device__ __forceinline__ void tma_load_4d_pair(void* dst, const CUtensorMap* map,
                                                 uint32_t bar_cluster, int c0, int c1, int c2,
                                                 int c3) {
  asm volatile(
      "cp.async.bulk.tensor.4d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4, %5, %6}], [%2];" ::"r"(smem_u32(dst)),
      "l"(map), "r"(bar_cluster), "r"(c0), "r"(c1), "r"(c2), "r"(c3)
      : "memory");
}
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t bar_cluster) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(bar_cluster)
               : "memory");
}
__device__ __forceinline__ void tmem_alloc_pair(uint32_t* slot, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_u32(slot)),
               "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void mma_bf16_pair(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc,
                                              uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// Arrive on `bar` of both CTAs of the pair once the MMAs issued so far completed.
__device__ __forceinline__ void mma_commit_pair(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64"
      " [%0], %1;" ::"r"(smem_u32(bar)),
      "h"((uint16_t)3)
      : "memory");
}
__host__ __device__ constexpr uint32_t idesc_bf16_pair(int n) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(n >> 3) << 17) | ((uint32_t)(256 >> 4) << 24);
}
// MMA width of a pair unit: token rows rounded up to 32 (16 per CTA), at most 256.
__device__ __forceinline__ int pair_n(int nrows) { return min(kPairBN, (nrows + 31) & ~31); }

// With FOLD a launch carries two unit sets: the routed experts (args, mapA0/A1/B) and, after them,
// the always-on shared experts of the same call (args_s, mapA0s/A1s/Bs), so a large call's
// projection pays one ramp and one tail for both.  Without FOLD the second set is ignored.
//
// IL4 (interleaved gate/up only): the A tile comes from one 4D view of the gate and up weights
// that alternates 16 gate rows and 16 up rows (mapA0; see encode_gu4), so each TMEM lane quarter
// holds the gate and up rows of the same 16 features and the epilogue pairs them with shuffles
// instead of the shared-memory exchange.
template <int MODE, bool FOLD, bool IL4>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(PairCfg<MODE, IL4>::kThreads, 1)
tc_pair_kernel(const __grid_constant__ CUtensorMap mapA0, const __grid_constant__ CUtensorMap mapA1,
               const __grid_constant__ CUtensorMap mapB, const TcArgs args,
               const __grid_constant__ CUtensorMap mapA0s, const __grid_constant__ CUtensorMap mapA1s,
               const __grid_constant__ CUtensorMap mapBs, const TcArgs args_s) {
  using C = PairCfg<MODE, IL4>;
  constexpr bool IL = C::kIL;
  static_assert(!IL4 || IL, "the 16-row interleave is a gate/up layout");
  constexpr int S = C::kStages;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  float* xchg = (float*)(smem + S * C::kStageBytes);
  uint64_t* full = (uint64_t*)(xchg + C::kXchgFloats);
  uint64_t* empty = full + S;
  uint64_t* tfull = empty + S;
  uint64_t* tempty = tfull + 2;
  uint64_t* mma_done = tempty + 2;
  uint64_t* xbar = mma_done + 1;
  uint32_t* tmem_slot = (uint32_t*)(xbar + 8);
  volatile int* abort_flag = (volatile int*)(tmem_slot + 1);

  const uint32_t rank = cluster_rank();
  const bool leader = rank == 0;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tfull[b], 1);
      mbar_init(&tempty[b], 2 * C::kEpiWarps);  // the epilogue warps of both CTAs (rank 0's)
    }
    mbar_init(mma_done, 1);
    for (int i = 0; i < 8; ++i) mbar_init(&xbar[i], 2);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) tmem_alloc_pair(tmem_slot, C::kTmemCols);
  if (threadIdx.x == 32) {
    asm volatile("prefetch.tensormap [%0];" ::"l"(&mapA0) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(&mapB) : "memory");
    if (FOLD) {
      asm volatile("prefetch.tensormap [%0];" ::"l"(&mapA0s) : "memory");
      asm volatile("prefetch.tensormap [%0];" ::"l"(&mapBs) : "memory");
    }
  }
  tc_fence_before();
  cluster_sync_all();  // both CTAs' barriers exist before either signals the other
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  pdl_wait();
  pdl_launch_dependents();

  const int pair = blockIdx.x >> 1, n_pairs = gridDim.x >> 1;
  const int total_tiles = args.tile_offs
                              ? args.tile_offs[args.n_groups]
                              : args.n_groups * ((args.uniform_rows + kPairBN - 1) / kPairBN);
  const int units_r = total_tiles * args.m_tiles * args.n_split;
  const int units = units_r + (FOLD ? args_s.n_groups *
                                            ((args_s.uniform_rows + kPairBN - 1) / kPairBN) *
                                            args_s.m_tiles * args_s.n_split
                                      : 0);
  // unit u of the launch: the routed set first, then the shared one (true)
  auto unit_at = [&](int u, Unit& w) -> bool {
    if (!FOLD || u < units_r) {
      w = decode_unit<kPairBN>(args, u, Offs{args.row_offs, args.tile_offs});
      return false;
    }
    w = decode_unit<kPairBN>(args_s, u - units_r, Offs{nullptr, nullptr});
    return true;
  };
  const uint32_t full0 = map_rank(smem_u32(full), 0);      // rank 0's full[0]
  const uint32_t tempty0 = map_rank(smem_u32(tempty), 0);  // rank 0's tempty[0]

  if (warp == 0) {
    if (lane == 0) {
      // ---------------------------------------------------------- TMA producer (both CTAs)
      int stage = 0;
      uint32_t phase = 0;
      long long issued = 0;
      bool ok = true;
      for (int u = pair; u < units && ok; u += n_pairs) {
        Unit w;
        const bool sh = unit_at(u, w);
        const CUtensorMap* mA0 = sh ? &mapA0s : &mapA0;
        const CUtensorMap* mA1 = sh ? &mapA1s : &mapA1;
        const CUtensorMap* mB = sh ? &mapBs : &mapB;
        const int n = pair_n(w.nrows);
        const int a_rows = sh ? args_s.a_rows_per_group : args.a_rows_per_group;
        const int b_shift = sh ? args_s.b_shift_per_group : args.b_shift_per_group;
        const int a_row = w.g * a_rows + w.m0 + (int)rank * C::kFeat;
        const int b_row = w.slot0 - w.g * b_shift + (int)rank * (n / 2);
        for (int kb = w.kb0; kb < w.kb1; kb += C::kKPS) {
          const int nk = min(C::kKPS, w.kb1 - kb);  // k-blocks of this stage
          if (!mbar_wait(&empty[stage], phase ^ 1u, abort_flag, args.err, 1u, true)) {
            ok = false;
            break;
          }
          uint8_t* st = smem + stage * C::kStageBytes;
          const uint32_t fb = full0 + 8u * (uint32_t)stage;
          if (leader) mbar_expect_tx(&full[stage], 2 * nk * C::kSubBytes);
#pragma unroll
          for (int j = 0; j < C::kKPS; ++j) {
            if (j < nk) {
              uint8_t* sj = st + j * C::kSubBytes;
              const int kx = (kb + j) * kBK;
              if (IL4) {
                tma_load_4d_pair(sj, mA0, fb, kx, 0, 0, a_row / 16);
              } else if (IL) {
                tma_load_2d_pair(sj, mA0, fb, kx, a_row);
                tma_load_2d_pair(sj + C::kABytes / 2, mA1, fb, kx, a_row);
              } else {
                tma_load_2d_pair(sj, mA0, fb, kx, a_row);
              }
              tma_load_2d_pair(sj + C::kABytes, mB, fb, kx, b_row);
            }
          }
          ++issued;
          if (++stage == S) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      // rank 0: let the copies of both CTAs still in flight land before the pair may exit
      if (leader) {
        const long long first = issued > S ? issued - S : 0;
        for (long long i = first; i < issued; ++i)
          mbar_wait(&full[i % S], (uint32_t)((i / S) & 1), abort_flag, args.err, 2u, false);
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && leader) {
      // ---------------------------------------------------------- MMA issuer (rank 0)
      int stage = 0;
      uint32_t phase = 0;
      int local = 0;
      bool ok = true;
      for (int u = pair; u < units && ok; u += n_pairs, ++local) {
        Unit w;
        unit_at(u, w);
        const int buf = local & 1;
        const uint32_t tph = (uint32_t)((local >> 1) & 1);
        if (!mbar_wait(&tempty[buf], tph ^ 1u, abort_flag, args.err, 4u, true)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d0 = tmem_base + (uint32_t)(buf * C::kAccCols);
        const uint32_t idesc = idesc_bf16_pair(pair_n(w.nrows));
        for (int kb = w.kb0; kb < w.kb1; kb += C::kKPS) {
          const int nk = min(C::kKPS, w.kb1 - kb);
          if (!mbar_wait(&full[stage], phase, abort_flag, args.err, 8u, true)) {
            ok = false;
            break;
          }
          tc_fence_after();
#pragma unroll
          for (int j = 0; j < C::kKPS; ++j) {
            if (j < nk) {
              const uint32_t sa = smem_u32(smem + stage * C::kStageBytes + j * C::kSubBytes);
              const uint32_t sb = sa + C::kABytes;
#pragma unroll
              for (int k = 0; k < kBK / 16; ++k)
                mma_bf16_pair(d0, sdesc_k128(sa + k * 32), sdesc_k128(sb + k * 32), idesc,
                              (kb > w.kb0 || j > 0 || k > 0) ? 1u : 0u);
            }
          }
          mma_commit_pair(&empty[stage]);
          if (++stage == S) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        mma_commit_pair(&tfull[buf]);
      }
      // no MMA may still be running when either CTA frees its TMEM
      mma_commit_pair(mma_done);
    }
    if (lane == 0) mbar_wait(mma_done, 0u, abort_flag, args.err, 16u, false);
  } else if (IL4) {
    // ------------------------------ epilogue, gate/up interleaved in 16-row groups (warps 2..9)
    // Warp w drains TMEM lane quarter q = w % 4 for the token columns [128 ch, 128 ch + 128),
    // ch = (w - 2) / 4.  Lanes i and i + 16 hold the two rows (gate and up, in the order of the
    // view) of feature 16 q + i.  Per 32 columns lanes 0-15 finish the first 16 and lanes 16-31
    // the second 16; each takes the other row's value for its columns from its partner lane.
    const int q = warp & 3;
    const int ch = (warp - 2) >> 2;
    const bool lo = lane < 16;
    int local = 0;
    for (int u = pair; u < units; u += n_pairs, ++local) {
      Unit w;
      const bool sh = unit_at(u, w);  // (scalars, as in the exchange epilogue below)
      __nv_bfloat16* const out = (__nv_bfloat16*)(sh ? args_s.out : args.out);
      const int M = sh ? args_s.M : args.M;
      const bool gate_first = (sh ? args_s.gate_first : args.gate_first) != 0;
      const bool mine_is_gate = lo == gate_first;
      const int buf = local & 1;
      const uint32_t tph = (uint32_t)((local >> 1) & 1);
      if (!warp_wait(&tfull[buf], tph, abort_flag, args.err, 32u)) break;
      tc_fence_after();
      const uint32_t tbase =
          tmem_base + ((uint32_t)(32 * q) << 16) + (uint32_t)(buf * C::kAccCols);
      const int f = w.m0 + (int)rank * C::kFeat + 16 * q + (lane & 15);
      const bool fok = f < M;
      const int c_end = min(128 * ch + 128, w.nrows);
      for (int c0 = 128 * ch; c0 < c_end; c0 += 32) {
        uint32_t v0[16], v1[16];
        tmem_ld16(tbase + c0, v0);
        tmem_ld16(tbase + c0 + 16, v1);
        tmem_wait_ld();
        const int cb = c0 + (lo ? 0 : 16);
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          const float mine = __uint_as_float(lo ? v0[j] : v1[j]);
          const float other =
              __shfl_xor_sync(0xffffffffu, __uint_as_float(lo ? v1[j] : v0[j]), 16);
          const float g = mine_is_gate ? mine : other;
          const float up = mine_is_gate ? other : mine;
          if (fok && cb + j < w.nrows)
            out[(size_t)(w.slot0 + cb + j) * M + f] = __float2bfloat16_rn(silu_f(g) * up);
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        if (leader) mbar_arrive(&tempty[buf]);
        else mbar_arrive_cluster(tempty0 + 8u * (uint32_t)buf);
      }
    }
  } else if (IL) {
    // ---------------------------------------- epilogue, interleaved gate/up (warps 2..9)
    // Warp w drains TMEM lane quarter w % 4 (gate rows in quarters 0-1, up rows in 2-3) for the
    // token columns [128 ch, 128 ch + 128), ch = (w - 2) / 4; a gate warp and the up warp of the
    // same features and columns exchange halves through shared memory, 32 columns at a time.
    const int q = warp & 3;
    const int half = q & 1;
    const bool is_gate = q < 2;
    const int ch = (warp - 2) >> 2;
    const int xp = half * 2 + ch;  // the warp pair's exchange buffers and barriers
    float* xh = xchg + xp * (2 * 2 * 16 * 32);
    uint64_t* xb = xbar + xp * 2;
    int local = 0;
    long long chunk = 0;
    bool ok = true;
    for (int u = pair; u < units && ok; u += n_pairs, ++local) {
      Unit w;
      // the unit set's output and width as scalars (a reference to either parameter struct
      // would let the stores below alias it and reload its fields every element)
      const bool sh = unit_at(u, w);
      __nv_bfloat16* const out = (__nv_bfloat16*)(sh ? args_s.out : args.out);
      const int M = sh ? args_s.M : args.M;
      const int buf = local & 1;
      const uint32_t tph = (uint32_t)((local >> 1) & 1);
      if (!warp_wait(&tfull[buf], tph, abort_flag, args.err, 32u)) break;
      tc_fence_after();
      const uint32_t tbase =
          tmem_base + ((uint32_t)(32 * q) << 16) + (uint32_t)(buf * C::kAccCols);
      const int f = w.m0 + (int)rank * C::kFeat + 32 * half + lane;
      const bool fok = f < M;
      const int keep = is_gate ? 0 : 16;
      const int c_end = min(128 * ch + 128, w.nrows);
      for (int c0 = 128 * ch; c0 < c_end; c0 += 32, ++chunk) {
        uint32_t v0[16], v1[16];
        tmem_ld16(tbase + c0, v0);
        tmem_ld16(tbase + c0 + 16, v1);
        tmem_wait_ld();
        const int b = (int)(chunk & 1);
        float* mine_out = xh + (b * 2 + (is_gate ? 0 : 1)) * 512;
        const float* theirs = xh + (b * 2 + (is_gate ? 1 : 0)) * 512;
#pragma unroll
        for (int j = 0; j < 16; ++j)
          mine_out[j * 32 + lane] = __uint_as_float(is_gate ? v1[j] : v0[j]);
        __syncwarp();
        if (lane == 0) mbar_arrive(&xb[b]);
        if (!warp_wait(&xb[b], (uint32_t)((chunk >> 1) & 1), abort_flag, args.err, 128u)) {
          ok = false;
          break;
        }
        if (fok) {
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            const int col = c0 + keep + j;
            if (col < w.nrows) {
              const float o = theirs[j * 32 + lane];
              const float m = __uint_as_float(is_gate ? v0[j] : v1[j]);
              const float h = is_gate ? silu_f(m) * o : silu_f(o) * m;
              out[(size_t)(w.slot0 + col) * M + f] = __float2bfloat16_rn(h);
            }
          }
        }
      }
      if (!ok) break;
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        if (leader) mbar_arrive(&tempty[buf]);
        else mbar_arrive_cluster(tempty0 + 8u * (uint32_t)buf);
      }
    }
  } else {
    // ------------------------------------------- epilogue, down projection (warps 2..9)
    // warp w drains TMEM lane quarter w % 4 for the token columns [128 ch, 128 ch + 128)
    const int q = warp & 3;
    const int ch = (warp - 2) >> 2;
    int local = 0;
    for (int u = pair; u < units; u += n_pairs, ++local) {
      Unit w;
      const bool sh = unit_at(u, w);  // (scalars, as in the gate/up epilogue)
      void* const out = sh ? args_s.out : args.out;
      const int M = sh ? args_s.M : args.M;
      const int out_bf16 = sh ? args_s.out_bf16 : args.out_bf16;
      const long long sstride = sh ? args_s.split_stride : args.split_stride;
      const int buf = local & 1;
      const uint32_t tph = (uint32_t)((local >> 1) & 1);
      if (!warp_wait(&tfull[buf], tph, abort_flag, args.err, 32u)) break;
      tc_fence_after();
      const uint32_t tbase =
          tmem_base + ((uint32_t)(32 * q) << 16) + (uint32_t)(buf * C::kAccCols);
      const int f = w.m0 + (int)rank * C::kFeat + 32 * q + lane;
      const bool fok = f < M;
      const int c_end = min(128 * ch + 128, w.nrows);
      for (int c0 = 128 * ch; c0 < c_end; c0 += 16) {
        uint32_t g[16];
        tmem_ld16(tbase + c0, g);
        tmem_wait_ld();
        if (fok) {
#pragma unroll
          for (int c = 0; c < 16; ++c) {
            if (c0 + c < w.nrows) {
              const size_t slot = (size_t)(w.slot0 + c0 + c);
              if (out_bf16)
                ((__nv_bfloat16*)out)[slot * M + f] = __float2bfloat16_rn(__uint_as_float(g[c]));
              else
                ((float*)out)[(size_t)w.split * sstride + slot * M + f] = __uint_as_float(g[c]);
            }
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        if (leader) mbar_arrive(&tempty[buf]);
        else mbar_arrive_cluster(tempty0 + 8u * (uint32_t)buf);
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // neither CTA leaves while the other may still signal it
  tc_fence_after();
  if (warp == 1) tmem_dealloc_pair(tmem_base, C::kTmemCols);
}

// Xperm[slot] = x[perm_tok[slot]] for every slot of the call (16-byte copies).
__global__ void __launch_bounds__(256)
gather_rows_kernel(const uint4* __restrict__ x, const int32_t* __restrict__ perm_tok,
                   const int32_t* __restrict__ n_rows, int row_vecs, uint4* __restrict__ xperm) {
  pdl_wait();
  pdl_launch_dependents();
  // one warp per row; each lane moves up to 8 16-byte pieces per pass, all loads before the stores
  const int lane = threadIdx.x & 31;
  const int slot = blockIdx.x * 8 + (threadIdx.x >> 5);
  if (slot >= *n_rows) return;
  const size_t src = (size_t)perm_tok[slot] * row_vecs;
  const size_t dst = (size_t)slot * row_vecs;
  for (int i0 = 0; i0 < row_vecs; i0 += 256) {
    uint4 v[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const int i = i0 + u * 32 + lane;
      if (i < row_vecs) v[u] = x[src + i];
    }
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const int i = i0 + u * 32 + lane;
      if (i < row_vecs) xperm[dst + i] = v[u];
    }
  }
}

// Self-test of the bounded wait: one thread waits on an mbarrier that nothing arrives on; after
// limit_ns the wait gives up, records bit 64 in the status word and the kernel returns normally.
__global__ void bounded_wait_selftest_kernel(unsigned long long limit_ns, unsigned int* err) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x != 0) return;
  abort_flag = 0;
  mbar_init(&bar, 1);
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  mbar_wait(&bar, 0u, &abort_flag, err, 64u, false, limit_ns);
}

// -------------------------------------------------------------------------------- host side
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = (PFN_cuTensorMapEncodeTiled_v12000)p;
  });
  return fn;
}

// 2D bf16 tensor [rows, cols] (row-major), box {64 cols, box_rows}, 128B swizzle, OOB -> 0.
bool encode_2d(CUtensorMap* m, const void* ptr, long long rows, long long cols, int box_rows) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
  cuuint32_t box[2] = {(cuuint32_t)kBK, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// 2D e4m3 tensor [rows, cols] (one byte per element), box {128 bytes, box_rows}, 128B swizzle,
// OOB -> 0: the fp8 weights and the e4m3 planes of the B operands.
bool encode_2d_u8(CUtensorMap* m, const void* ptr, long long rows, long long cols, int box_rows) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)cols};
  cuuint32_t box[2] = {(cuuint32_t)kBK8, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void*>(ptr), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// The gate and up weights of one expert set ([rows, cols] bf16 each, rows a multiple of 16) as one
// 4D view that alternates 16 rows of each: element (k, r, h, g) is row 16 g + r, column k of the
// lower (h = 0) or higher (h = 1) of the two allocations, so the box {64, 16, 2, 4} holds 128 rows
// [16 of one, 16 of the other, ...] of 64 columns, in the 128B-swizzled layout of a 2D box of 128
// rows.  The two allocations need not be adjacent: the h stride is their distance.  false when
// the view cannot be encoded (the caller then keeps the two 64-row boxes).
bool encode_gu4(CUtensorMap* m, const void* gate, const void* up, long long rows, long long cols,
                bool* gate_first) {
  auto fn = encode_fn();
  if (!fn || rows % 16 != 0 || gate == up) return false;
  const bool gf = (uintptr_t)gate < (uintptr_t)up;
  const char* lo = (const char*)(gf ? gate : up);
  const char* hi = (const char*)(gf ? up : gate);
  const unsigned long long dist = (unsigned long long)(hi - lo);
  if (dist % 16 != 0 || dist >= (1ULL << 40)) return false;
  cuuint64_t dims[4] = {(cuuint64_t)cols, 16, 2, (cuuint64_t)(rows / 16)};
  cuuint64_t strides[3] = {(cuuint64_t)cols * 2, (cuuint64_t)dist, (cuuint64_t)cols * 2 * 16};
  cuuint32_t box[4] = {(cuuint32_t)kBK, 16, 2, 4};
  cuuint32_t estr[4] = {1, 1, 1, 1};
  const bool ok = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<char*>(lo), dims, strides,
                     box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
  *gate_first = gf;
  return ok;
}

struct Maps {
  CUtensorMap wg, wu, wd, wsg, wsu, wsd;   // bf16 weights, or e4m3 weights of an fp8 layer
  CUtensorMap wg64, wu64, wsg64, wsu64;  // 64-row boxes for the interleaved gate/up A tile
  // the 16-row interleave of gate and up (encode_gu4) for the SM-pair gate/up, when it encodes
  CUtensorMap wgu4, wsgu4;
  bool il4 = false, sil4 = false;                   // routed / shared view available
  bool gate_first = true, sgate_first = true;       // gate rows first in the view
  CUtensorMap xperm[kNumBN], act[kNumBN], sact[kNumBN];
  // fp8 layers: the e4m3 hi/lo planes of the B operands (slot rows of x, token rows of x, the
  // routed and the shared activations)
  CUtensorMap xq[kNumBN], xqt[kNumBN], aq[kNumBN], saq[kNumBN];
};

int bn_index(int bn) {
  for (int i = 0; i < kNumBN; ++i)
    if (kBNs[i] == bn) return i;
  return kNumBN - 1;
}

template <int BN, int MODE, bool W8>
cudaError_t launch_tc(const CUtensorMap& a0, const CUtensorMap& a1, const CUtensorMap& b,
                      const TcArgs& args, int grid, cudaStream_t st) {
  using C = Cfg<BN, MODE, W8>;
  static std::once_flag once;
  static cudaError_t attr_err = cudaSuccess;
  std::call_once(once, [] {
    attr_err = cudaFuncSetAttribute(tc_ffn_kernel<BN, MODE, W8>,
                                    cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemBytes);
  });
  if (attr_err != cudaSuccess) return attr_err;
  if (grid <= 0) return cudaSuccess;
  return launch_pdl(tc_ffn_kernel<BN, MODE, W8>, dim3(grid), dim3(C::kThreads), C::kSmemBytes,
                    st, a0, a1, b, args);
}

// SM-pair kernels: one 2-CTA cluster per pair of SMs, at most as many pairs as can be resident.
// The routed set (a0, a1, b, args) and, when sargs is given, the shared set of the same call in
// the same launch; units counts both.
template <int MODE, bool FOLD, bool IL4>
cudaError_t launch_pair_t(const CUtensorMap& a0, const CUtensorMap& a1, const CUtensorMap& b,
                          const TcArgs& args, long long units, int num_sms, cudaStream_t st,
                          const CUtensorMap* sa0, const CUtensorMap* sa1, const CUtensorMap* sb,
                          const TcArgs* sargs) {
  using C = PairCfg<MODE, IL4>;
  static std::once_flag once;
  static cudaError_t attr_err = cudaSuccess;
  static int max_pairs = 0;
  std::call_once(once, [num_sms] {
    attr_err = cudaFuncSetAttribute(tc_pair_kernel<MODE, FOLD, IL4>,
                                    cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemBytes);
    if (attr_err != cudaSuccess) return;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(num_sms & ~1);
    cfg.blockDim = dim3(C::kThreads);
    cfg.dynamicSmemBytes = C::kSmemBytes;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = 2;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, tc_pair_kernel<MODE, FOLD, IL4>, &cfg) != cudaSuccess ||
        n <= 0) {
      cudaGetLastError();
      n = num_sms / 2;
    }
    max_pairs = std::min(n, num_sms / 2);
  });
  if (attr_err != cudaSuccess) return attr_err;
  const long long pairs = std::min<long long>(max_pairs, units);
  if (pairs <= 0) return cudaSuccess;
  TcArgs none;
  std::memset(&none, 0, sizeof(none));
  return launch_pdl(tc_pair_kernel<MODE, FOLD, IL4>, dim3((unsigned)(2 * pairs)), dim3(C::kThreads),
                    C::kSmemBytes, st, a0, a1, b, args, sa0 ? *sa0 : a0, sa1 ? *sa1 : a1,
                    sb ? *sb : b, sargs ? *sargs : none);
}
template <int MODE, bool IL4 = false>
cudaError_t launch_pair(const CUtensorMap& a0, const CUtensorMap& a1, const CUtensorMap& b,
                        const TcArgs& args, long long units, int num_sms, cudaStream_t st,
                        const CUtensorMap* sa0 = nullptr, const CUtensorMap* sa1 = nullptr,
                        const CUtensorMap* sb = nullptr, const TcArgs* sargs = nullptr) {
  if (sargs)
    return launch_pair_t<MODE, true, IL4>(a0, a1, b, args, units, num_sms, st, sa0, sa1, sb,
                                          sargs);
  return launch_pair_t<MODE, false, IL4>(a0, a1, b, args, units, num_sms, st, nullptr, nullptr,
                                         nullptr, nullptr);
}

// Single-SM launches: token tiles of 16..128 rows (256-row tiles run on SM pairs); W8 for fp8
// weights (single-SM kernels only, at any call size).
template <bool W8>
cudaError_t launch_up_bn(int bn, const CUtensorMap& a0, const CUtensorMap& a1,
                         const CUtensorMap& b, const TcArgs& args, int grid, cudaStream_t st) {
  switch (bn) {
    case 16: return launch_tc<16, kModeGateUp, W8>(a0, a1, b, args, grid, st);
    case 32: return launch_tc<32, kModeGateUp, W8>(a0, a1, b, args, grid, st);
    case 64: return launch_tc<64, kModeGateUp, W8>(a0, a1, b, args, grid, st);
    default: return launch_tc<128, kModeGateUp, W8>(a0, a1, b, args, grid, st);
  }
}

template <bool W8>
cudaError_t launch_down_bn(int bn, const CUtensorMap& a0, const CUtensorMap& b,
                           const TcArgs& args, int grid, cudaStream_t st) {
  switch (bn) {
    case 16: return launch_tc<16, kModeDown, W8>(a0, a0, b, args, grid, st);
    case 32: return launch_tc<32, kModeDown, W8>(a0, a0, b, args, grid, st);
    case 64: return launch_tc<64, kModeDown, W8>(a0, a0, b, args, grid, st);
    default: return launch_tc<128, kModeDown, W8>(a0, a0, b, args, grid, st);
  }
}

}  // namespace

// The largest group of a call has at most T rows (each token picks an expert once).  Calls of at
// least kPairMinTokens run both expert GEMMs on SM pairs with 256-token tiles (interleaved gate/
// up, 256-feature down tiles); smaller calls use single-SM kernels with tiles of the smallest
// width that holds T, at most 128.  (On a single SM the interleaved 256-token gate/up moves the
// same shared-memory bytes per flop as two 128-token accumulators and measured slower: OLMoE
// prefill gate/up 294 -> 316 us.)
constexpr int kPairMinTokens = 1024;
int tc_tile_rows(const TcLayer& L, int T) {
  for (int i = 0; i < kNumBN - 1; ++i)
    if (T <= kBNs[i]) return kBNs[i];
  return T >= kPairMinTokens && !L.w8 ? kPairBN : 128;
}
// Small calls gather their token rows inside the gate/up kernel (one launch and one HBM round
// trip fewer); large calls copy them to Xperm first: there the shared-memory-bound gate/up kernel
// loses more to the warp's cp.async traffic than the separate gather costs.  fp8 layers always
// read their B operand from the e4m3 planes that split_e4m3_kernel writes.
bool tc_gathers_in_kernel(const TcLayer& L, int T) { return T <= 128 && !L.w8; }

bool tc_folds_shared(const TcLayer& L, int T) {
  return L.S > 0 && !L.w8 && tc_tile_rows(L, T) == kPairBN;
}

int tc_tile_rows_down(const TcLayer& L, int T) { return tc_tile_rows(L, T); }

// k-blocks of a reduction of length n: 64 bf16 or 128 e4m3 elements (128 bytes of each row) per
// k-block; a ragged last fp8 k-block reads zeros beyond the row (TMA fill).
static int kblocks_of(const TcLayer& L, int n) { return L.w8 ? (n + kBK8 - 1) / kBK8 : n / kBK; }

// Split-K of the routed down projection: enough work units for ~8 waves of the persistent grid
// (so the last, partial wave is a small fraction of a memory-bound launch), each K slice at least
// 8 k-blocks (128 KB of weights per tile).  Estimated units = (token tiles + groups) x feature
// tiles; prefill calls already have plenty and keep one slice.
static int split_for(const TcLayer& L, int T) {
  const int m_tiles = (L.d + kBM - 1) / kBM;
  const int kblocks = kblocks_of(L, L.F);
  const int bn = tc_tile_rows_down(L, T);
  const long long rows = (long long)T * L.K;
  const long long est = ((rows + bn - 1) / bn + std::min<long long>(L.E, rows)) * m_tiles;
  int split = 1;
  while (est * split < 8LL * L.num_sms && kblocks / (split * 2) >= 8 && split < 32) split *= 2;
  return split;
}

// Split count with no empty K slice: n slices of ceil(kblocks / split) k-blocks each.
int tc_down_split(const TcLayer& L, int T) {
  const int kblocks = kblocks_of(L, L.F);
  const int split = split_for(L, T);
  const int per = (kblocks + split - 1) / split;
  return (kblocks + per - 1) / per;
}

long long tc_opart_rows(const TcLayer& L) {
  long long best = (long long)L.Tmax * L.K;
  for (int T = 1; T <= L.Tmax; ++T) {
    const int s = split_for(L, T);
    if (s == 1 && T > 4096) break;  // split is 1 from here on
    best = std::max(best, (long long)s * T * L.K);
  }
  return best;
}

int tc_configure(TcLayer& L, const eat_layer_desc& D, int K, int Tmax, const char** msg) {
  L.E = D.n_experts;
  L.d = D.d_model;
  L.F = D.d_ff;
  L.S = D.n_shared;
  L.Fs = D.n_shared > 0 ? D.d_ff_shared : 0;
  L.w8 = D.wdtype == EAT_FP8_E4M3;
  if (L.w8) {
    L.sg = D.w_gate_scale;
    L.su = D.w_up_scale;
    L.sd = D.w_down_scale;
    L.ssg = D.ws_gate_scale;
    L.ssu = D.ws_up_scale;
    L.ssd = D.ws_down_scale;
  }
  L.K = K;
  L.Tmax = Tmax;
  int dev = 0;
  cudaGetDevice(&dev);
  cudaDeviceProp prop;
  if (cudaGetDeviceProperties(&prop, dev) != cudaSuccess) {
    if (msg) *msg = "cudaGetDeviceProperties failed";
    return 1;
  }
  if (prop.major != 10 || prop.minor != 3) {
    if (msg) *msg = "the tensor-core kernels are built for sm_103a (GB300)";
    return 1;
  }
  L.num_sms = prop.multiProcessorCount;
  if (!encode_fn()) {
    if (msg) *msg = "cuTensorMapEncodeTiled is unavailable";
    return 1;
  }
  return 0;
}

int tc_bind(TcLayer& L, const eat_layer_desc& D, void* xperm, void* act, void* sact,
            const TcWork& q, const char** msg) {
  Maps* m = new Maps();
  std::memset(m, 0, sizeof(Maps));
  const long long rows = (long long)L.Tmax * L.K;
  L.q = q;
  bool ok;
  if (L.w8) {
    ok = encode_2d_u8(&m->wg, D.w_gate, (long long)L.E * L.F, L.d, kBM) &&
         encode_2d_u8(&m->wu, D.w_up, (long long)L.E * L.F, L.d, kBM) &&
         encode_2d_u8(&m->wd, D.w_down, (long long)L.E * L.d, L.F, kBM);
    if (ok && L.S > 0)
      ok = encode_2d_u8(&m->wsg, D.ws_gate, (long long)L.S * L.Fs, L.d, kBM) &&
           encode_2d_u8(&m->wsu, D.ws_up, (long long)L.S * L.Fs, L.d, kBM) &&
           encode_2d_u8(&m->wsd, D.ws_down, (long long)L.S * L.d, L.Fs, kBM);
  } else {
    ok = encode_2d(&m->wg, D.w_gate, (long long)L.E * L.F, L.d, kBM) &&
         encode_2d(&m->wu, D.w_up, (long long)L.E * L.F, L.d, kBM) &&
         encode_2d(&m->wg64, D.w_gate, (long long)L.E * L.F, L.d, kBM / 2) &&
         encode_2d(&m->wu64, D.w_up, (long long)L.E * L.F, L.d, kBM / 2) &&
         encode_2d(&m->wd, D.w_down, (long long)L.E * L.d, L.F, kBM);
    if (ok)
      m->il4 = L.F % 16 == 0 &&
               encode_gu4(&m->wgu4, D.w_gate, D.w_up, (long long)L.E * L.F, L.d, &m->gate_first);
    if (ok && L.S > 0) {
      ok = encode_2d(&m->wsg, D.ws_gate, (long long)L.S * L.Fs, L.d, kBM) &&
           encode_2d(&m->wsu, D.ws_up, (long long)L.S * L.Fs, L.d, kBM) &&
           encode_2d(&m->wsg64, D.ws_gate, (long long)L.S * L.Fs, L.d, kBM / 2) &&
           encode_2d(&m->wsu64, D.ws_up, (long long)L.S * L.Fs, L.d, kBM / 2) &&
           encode_2d(&m->wsd, D.ws_down, (long long)L.S * L.d, L.Fs, kBM);
      if (ok)
        m->sil4 = L.Fs % 16 == 0 && encode_gu4(&m->wsgu4, D.ws_gate, D.ws_up,
                                                (long long)L.S * L.Fs, L.d, &m->sgate_first);
    }
  }
  for (int i = 0; i < kNumBN && ok; ++i) {
    if (L.w8) {
      // the hi and lo planes of each B operand, one map over both (lo at row offset R)
      ok = encode_2d_u8(&m->xq[i], q.xq, 2 * rows, L.d, kBNs[i]) &&
           encode_2d_u8(&m->aq[i], q.aq, 2 * rows, L.F, kBNs[i]);
      if (ok && L.S > 0)
        ok = encode_2d_u8(&m->xqt[i], q.xqt, 2LL * L.Tmax, L.d, kBNs[i]) &&
             encode_2d_u8(&m->saq[i], q.saq, 2LL * L.S * L.Tmax, L.Fs, kBNs[i]);
      continue;
    }
    ok = encode_2d(&m->xperm[i], xperm, rows, L.d, kBNs[i]) &&
         encode_2d(&m->act[i], act, rows, L.F, kBNs[i]);
    if (ok && L.S > 0) ok = encode_2d(&m->sact[i], sact, (long long)L.S * L.Tmax, L.Fs, kBNs[i]);
  }
  if (!ok) {
    delete m;
    if (msg) *msg = "cuTensorMapEncodeTiled rejected a weight or workspace tensor";
    return 1;
  }
  L.maps = m;
  L.ready = true;
  return 0;
}

void tc_destroy(TcLayer& L) {
  delete (Maps*)L.maps;
  L.maps = nullptr;
  L.ready = false;
}

cudaError_t tc_launch_gather(const TcLayer& L, const TcCall& c, cudaStream_t st) {
  const int rows = c.T * L.K;
  const int vecs = L.d / 8;
  return launch_pdl(gather_rows_kernel, dim3((rows + 7) / 8), dim3(256), 0, st,
                    (const uint4*)c.x, c.perm_tok, c.offs + L.E, vecs, (uint4*)c.xperm);
}

cudaError_t tc_launch_up(const TcLayer& L, const TcCall& c, bool shared, cudaStream_t st) {
  const Maps* m = (const Maps*)L.maps;
  TcArgs a;
  std::memset(&a, 0, sizeof(a));
  const int bn = c.tile_rows;
  const bool pair = bn == kPairBN;  // SM pairs, interleaved gate/up: 128 features per unit
  a.M = shared ? L.Fs : L.F;
  a.m_tile = kBM;
  a.m_tiles = (a.M + a.m_tile - 1) / a.m_tile;
  a.kblocks = kblocks_of(L, L.d);
  a.n_split = 1;
  a.kb_per_split = a.kblocks;
  a.a_rows_per_group = a.M;
  a.err = c.status;
  // the group layout is two or more launches old unless this kernel gathers the rows itself
  // (then the permute is the previous launch)
  a.prefetch_a = tc_gathers_in_kernel(L, c.T) && !shared ? 0 : 1;
  if (L.w8) {
    a.scale0 = shared ? L.ssg : L.sg;
    a.scale1 = shared ? L.ssu : L.su;
    a.bscale = shared ? L.q.xqt_s : L.q.xq_s;
    a.b_lo_rows = shared ? L.Tmax : L.Tmax * L.K;
  }
  auto up_bn = [&](const CUtensorMap& a0, const CUtensorMap& a1, const CUtensorMap& b, int grid) {
    return L.w8 ? launch_up_bn<true>(bn, a0, a1, b, a, grid, st)
                : launch_up_bn<false>(bn, a0, a1, b, a, grid, st);
  };
  long long max_tiles;
  // the shared experts' unit set: every token of the call in order, weight 1 (reading R9)
  auto shared_args = [&](TcArgs& s) {
    s = a;
    s.M = L.Fs;
    s.m_tiles = (s.M + s.m_tile - 1) / s.m_tile;
    s.a_rows_per_group = s.M;
    s.prefetch_a = 1;
    if (L.w8) {
      s.scale0 = L.ssg;
      s.scale1 = L.ssu;
      s.bscale = L.q.xqt_s;
      s.b_lo_rows = L.Tmax;
    }
    s.n_groups = L.S;
    s.row_offs = nullptr;
    s.tile_offs = nullptr;
    s.uniform_rows = c.T;
    s.b_shift_per_group = c.T;
    s.out = c.sact;
  };
  if (shared) {
    CUtensorMap xm;
    if (L.w8) xm = m->xqt[bn_index(bn)];
    else if (!encode_2d(&xm, c.x, c.T, L.d, pair ? kPairRows : bn)) return cudaErrorInvalidValue;
    shared_args(a);
    max_tiles = (long long)L.S * ((c.T + bn - 1) / bn);
    const long long units = max_tiles * a.m_tiles;
    if (pair && m->sil4) {
      a.gate_first = m->sgate_first ? 1 : 0;
      return launch_pair<kModeGateUpIL, true>(m->wsgu4, m->wsgu4, xm, a, units, L.num_sms, st);
    }
    if (pair)
      return launch_pair<kModeGateUpIL>(m->wsg64, m->wsu64, xm, a, units, L.num_sms, st);
    const int grid = (int)std::min<long long>(L.num_sms, units);
    return up_bn(m->wsg, m->wsu, xm, grid);
  }
  a.n_groups = L.E;
  a.row_offs = c.offs;
  a.tile_offs = c.tile_offs;
  a.out = c.act;
  max_tiles = (long long)(c.T * L.K + bn - 1) / bn + L.E;
  const long long units = max_tiles * a.m_tiles;
  const int grid = (int)std::min<long long>(L.num_sms, units);
  if (tc_gathers_in_kernel(L, c.T)) {
    // small call: the token rows are gathered from x inside the kernel
    a.b_rows = c.perm_tok;
    a.bx = (const __nv_bfloat16*)c.x;
    return up_bn(m->wg, m->wu, m->wg, grid);
  }
  if (pair && c.fold_shared && L.S > 0) {  // the shared experts in the same launch
    TcArgs sa;
    shared_args(sa);
    CUtensorMap xm;
    if (!encode_2d(&xm, c.x, c.T, L.d, kPairRows)) return cudaErrorInvalidValue;
    const long long s_units = (long long)L.S * ((c.T + bn - 1) / bn) * sa.m_tiles;
    if (m->il4 && m->sil4) {
      a.gate_first = m->gate_first ? 1 : 0;
      sa.gate_first = m->sgate_first ? 1 : 0;
      return launch_pair<kModeGateUpIL, true>(m->wgu4, m->wgu4, m->xperm[bn_index(kPairRows)], a,
                                              units + s_units, L.num_sms, st, &m->wsgu4,
                                              &m->wsgu4, &xm, &sa);
    }
    return launch_pair<kModeGateUpIL>(m->wg64, m->wu64, m->xperm[bn_index(kPairRows)], a,
                                      units + s_units, L.num_sms, st, &m->wsg64, &m->wsu64, &xm,
                                      &sa);
  }
  if (pair && m->il4) {
    a.gate_first = m->gate_first ? 1 : 0;
    return launch_pair<kModeGateUpIL, true>(m->wgu4, m->wgu4, m->xperm[bn_index(kPairRows)], a,
                                            units, L.num_sms, st);
  }
  if (pair)
    return launch_pair<kModeGateUpIL>(m->wg64, m->wu64, m->xperm[bn_index(kPairRows)], a, units,
                                      L.num_sms, st);
  return up_bn(m->wg, m->wu, L.w8 ? m->xq[bn_index(bn)] : m->xperm[bn_index(bn)], grid);
}

cudaError_t tc_launch_down(const TcLayer& L, const TcCall& c, bool shared, int n_split,
                           cudaStream_t st) {
  const Maps* m = (const Maps*)L.maps;
  TcArgs a;
  std::memset(&a, 0, sizeof(a));
  const int bn = c.tile_rows_down;
  const bool pair = bn == kPairBN;  // SM pairs: 256 output features per unit
  const int Kdim = shared ? L.Fs : L.F;
  a.M = L.d;
  a.m_tile = pair ? 2 * kBM : kBM;
  a.m_tiles = (L.d + a.m_tile - 1) / a.m_tile;
  a.kblocks = kblocks_of(L, Kdim);
  a.n_split = n_split;
  a.kb_per_split = (a.kblocks + n_split - 1) / n_split;
  a.a_rows_per_group = L.d;
  a.err = c.status;
  a.prefetch_a = 1;  // the group layout is the permute's, two or more launches back
  if (L.w8) {
    a.scale0 = shared ? L.ssd : L.sd;
    a.bscale = shared ? L.q.saq_s : L.q.aq_s;
    a.b_lo_rows = shared ? L.S * L.Tmax : L.Tmax * L.K;
  }
  auto down_bn = [&](const CUtensorMap& a0, const CUtensorMap& b, int grid) {
    return L.w8 ? launch_down_bn<true>(bn, a0, b, a, grid, st)
                : launch_down_bn<false>(bn, a0, b, a, grid, st);
  };
  long long max_tiles;
  auto shared_args = [&](TcArgs& s) {
    s = a;
    s.kblocks = kblocks_of(L, L.Fs);
    s.n_split = 1;
    s.kb_per_split = s.kblocks;
    if (L.w8) {
      s.scale0 = L.ssd;
      s.bscale = L.q.saq_s;
      s.b_lo_rows = L.S * L.Tmax;
    }
    s.n_groups = L.S;
    s.row_offs = nullptr;
    s.tile_offs = nullptr;
    s.uniform_rows = c.T;
    s.out = c.sout;
    s.out_bf16 = 1;
    s.split_stride = 0;
  };
  if (shared) {
    shared_args(a);
    a.n_split = n_split;
    a.kb_per_split = (a.kblocks + n_split - 1) / n_split;
    max_tiles = (long long)L.S * ((c.T + bn - 1) / bn);
    const long long units = max_tiles * a.m_tiles;
    if (pair)
      return launch_pair<kModeDown>(m->wsd, m->wsd, m->sact[bn_index(kPairRows)], a, units,
                                    L.num_sms, st);
    const int grid = (int)std::min<long long>(L.num_sms, units);
    return down_bn(m->wsd, L.w8 ? m->saq[bn_index(bn)] : m->sact[bn_index(bn)], grid);
  }
  a.n_groups = L.E;
  a.row_offs = c.offs;
  a.tile_offs = c.tile_offs_down;
  a.out = c.opart;
  a.out_bf16 = n_split == 1 ? 1 : 0;
  a.split_stride = (long long)c.T * L.K * L.d;
  max_tiles = (long long)(c.T * L.K + bn - 1) / bn + L.E;
  const long long units = max_tiles * a.m_tiles * n_split;
  if (pair && c.fold_shared && L.S > 0) {  // the shared experts in the same launch
    TcArgs sa;
    shared_args(sa);
    const long long s_units = (long long)L.S * ((c.T + bn - 1) / bn) * sa.m_tiles;
    return launch_pair<kModeDown>(m->wd, m->wd, m->act[bn_index(kPairRows)], a, units + s_units,
                                  L.num_sms, st, &m->wsd, &m->wsd,
                                  &m->sact[bn_index(kPairRows)], &sa);
  }
  if (pair)
    return launch_pair<kModeDown>(m->wd, m->wd, m->act[bn_index(kPairRows)], a, units, L.num_sms,
                                  st);
  const int grid = (int)std::min<long long>(L.num_sms, units);
  return down_bn(m->wd, L.w8 ? m->aq[bn_index(bn)] : m->act[bn_index(bn)], grid);
}

cudaError_t tc_selftest_bounded_wait(unsigned long long limit_ns, unsigned int* dev_status,
                                     cudaStream_t st) {
  bounded_wait_selftest_kernel<<<1, 32, 0, st>>>(limit_ns, dev_status);
  return cudaGetLastError();
}

}  // namespace eat
