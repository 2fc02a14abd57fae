// Permute by expert: groups the selected (token, expert) pairs of one call by expert so that the
// expert FFNs read contiguous row lists ("only activated experts participate", §3.4).
//
// One CTA of 1024 threads.  Pass 1 counts n_e with shared-memory atomics (integer, order-free)
// and scans them into slot offsets and row-tile offsets.  Pass 2 walks the tokens in chunks of
// 1024 and gives every pair a STABLE slot (tokens ascending inside each expert): each warp finds
// the experts present among its 32 tokens with ballots, counts them per warp, the counts are
// scanned across warps per expert, and the same ballots give each lane its rank.  Stable slots
// make every later per-expert sum (P_total, the EMA norm mean) run in a fixed order.
#include "eat_internal.cuh"

namespace eat {

namespace {

constexpr int kPermThreads = 1024;
constexpr int kPermWarps = kPermThreads / 32;

// For the calling lane's experts ex[0..K) (-1 = none), iterate over the distinct experts present
// in the warp; fn(e, mask_of_lanes_with_e, j_of_this_lane_or_-1).
template <typename Fn>
__device__ __forceinline__ void for_each_warp_expert(const int* ex, int K, Fn fn) {
  const unsigned full = 0xffffffffu;
  unsigned done = 0;  // bit j set: ex[j] handled
  for (;;) {
    int mine = -1;
    for (int j = 0; j < K; ++j)
      if (!(done & (1u << j)) && ex[j] >= 0) { mine = ex[j]; break; }
    const unsigned pending = __ballot_sync(full, mine >= 0);
    if (!pending) break;
    const int leader = __ffs(pending) - 1;
    const int e = __shfl_sync(full, mine, leader);
    int jj = -1;
    for (int j = 0; j < K; ++j)
      if (ex[j] == e) { jj = j; break; }
    const unsigned m = __ballot_sync(full, jj >= 0);
    if (jj >= 0) done |= 1u << jj;
    fn(e, m, jj);
  }
}

__global__ void __launch_bounds__(kPermThreads)
permute_kernel(const int32_t* __restrict__ idx, const int32_t* __restrict__ kk,
               const float* __restrict__ psel, int T, int K, int E, int tile_rows, PermuteOut o) {
  extern __shared__ int sm[];
  pdl_wait();
  pdl_launch_dependents();
  int* cnt = sm;                      // [E]
  int* cursor = cnt + E;              // [E]
  int* wcnt = cursor + E;             // [kPermWarps][E]
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const unsigned lt = (1u << lane) - 1u;

  for (int e = tid; e < E; e += kPermThreads) cnt[e] = 0;
  __syncthreads();
  for (int i = tid; i < T * K; i += kPermThreads) {
    const int e = idx[i];
    if (e >= 0) atomicAdd(&cnt[e], 1);
  }
  __syncthreads();
  if (tid == 0) {
    int s = 0, ts = 0, na = 0;
    for (int e = 0; e < E; ++e) {
      o.offs[e] = s;
      o.tile_offs[e] = ts;
      o.n_e[e] = cnt[e];
      cursor[e] = s;
      if (cnt[e] > 0) o.active[na++] = e;
      s += cnt[e];
      ts += (cnt[e] + tile_rows - 1) / tile_rows;
    }
    o.offs[E] = s;
    o.tile_offs[E] = ts;
    for (int e = na; e < E; ++e) o.active[e] = -1;
    o.active[E] = na;
  }
  __syncthreads();

  int ex[kMaxK];
  for (int c0 = 0; c0 < T; c0 += kPermThreads) {
    const int t = c0 + tid;
    const int kt = t < T ? kk[t] : 0;
    for (int j = 0; j < K; ++j) ex[j] = (j < kt) ? idx[(size_t)t * K + j] : -1;
    for (int e = lane; e < E; e += 32) wcnt[warp * E + e] = 0;
    __syncwarp();
    for_each_warp_expert(ex, K, [&](int e, unsigned m, int jj) {
      if (lane == 0) wcnt[warp * E + e] = __popc(m);
    });
    __syncthreads();
    for (int e = tid; e < E; e += kPermThreads) {
      int run = cursor[e];
      for (int w = 0; w < kPermWarps; ++w) {
        const int c = wcnt[w * E + e];
        wcnt[w * E + e] = run;
        run += c;
      }
      cursor[e] = run;
    }
    __syncthreads();
    for_each_warp_expert(ex, K, [&](int e, unsigned m, int jj) {
      if (jj >= 0) {
        const int slot = wcnt[warp * E + e] + __popc(m & lt);
        o.perm_tok[slot] = t;
        o.slot_of[(size_t)t * K + jj] = slot;
        o.perm_p[slot] = psel[(size_t)t * K + jj];
      }
    });
    if (t < T)
      for (int j = kt; j < K; ++j) o.slot_of[(size_t)t * K + j] = -1;
    __syncthreads();
  }
}

}  // namespace

cudaError_t launch_permute(const int32_t* idx, const int32_t* k, const float* psel, int T, int K,
                           int E, int tile_rows, PermuteOut o, cudaStream_t st) {
  const size_t smem = (size_t)(2 * E + kPermWarps * E) * sizeof(int);
  return launch_pdl(permute_kernel, dim3(1), dim3(kPermThreads), smem, st, idx, k, psel, T, K, E,
                    tile_rows, o);
}

}  // namespace eat
