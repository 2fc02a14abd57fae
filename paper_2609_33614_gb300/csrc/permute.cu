// Permute by expert: groups the selected (token, expert) pairs of one call by expert so that the
// expert FFNs read contiguous row lists ("only activated experts participate", §3.4).
//
// A call of at most 1024 tokens runs as a single 1024-thread CTA that also counts; larger calls
// are split in chunks of 256 tokens, one CTA each, after a counting pass.  Counts n_e come from shared-memory atomics (integers, order-free); each
// chunk's first slot per expert is the expert's offset plus the counts of the earlier chunks.
// Inside a chunk every pair gets a STABLE slot (tokens ascending inside each expert): each warp
// finds the experts present among its 32 tokens with ballots, counts them per warp, the counts are
// scanned across warps per expert, and the same ballots give each lane its rank.  Stable slots
// make every later per-expert sum (P_total, the EMA norm mean) run in a fixed order.
#include "eat_internal.cuh"

namespace eat {

namespace {

constexpr int kPermThreads = 1024;   // single-CTA calls (T <= 1024)
constexpr int kChunkThreads = 256;   // tokens (and threads) per CTA of a multi-CTA call

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

// Per-chunk expert counts (large calls): chunk_cnt[c][e] = activations of expert e among the
// chunk's tokens [c * 256, (c + 1) * 256).
__global__ void __launch_bounds__(kChunkThreads)
permute_count_kernel(const int32_t* __restrict__ idx, int T, int K, int E,
                     int32_t* __restrict__ chunk_cnt) {
  extern __shared__ int cnt[];
  pdl_wait();
  pdl_launch_dependents();
  const int tid = threadIdx.x, c = blockIdx.x, nt = blockDim.x;
  for (int e = tid; e < E; e += nt) cnt[e] = 0;
  __syncthreads();
  const int t0 = c * nt, t1 = min(T, t0 + nt);
  for (int i = t0 * K + tid; i < t1 * K; i += nt) {
    const int e = idx[i];
    if (e >= 0) atomicAdd(&cnt[e], 1);
  }
  __syncthreads();
  for (int e = tid; e < E; e += nt) chunk_cnt[(size_t)c * E + e] = cnt[e];
}

// Slot assignment of one chunk of blockDim.x tokens.  With chunk_cnt == nullptr the kernel runs
// as a single CTA over a call of at most 1024 tokens and counts in place.
__global__ void __launch_bounds__(1024)
permute_assign_kernel(const int32_t* __restrict__ idx, const int32_t* __restrict__ kk,
                      const float* __restrict__ psel, int T, int K, int E, int tile_rows,
                      int tile_rows2, const int32_t* __restrict__ chunk_cnt, int n_chunks,
                      PermuteOut o) {
  extern __shared__ int sm[];
  pdl_wait();
  pdl_launch_dependents();
  int* cnt = sm;                      // [E] activations of each expert in the whole call
  int* cursor = cnt + E;              // [E] first slot of each expert for this chunk
  int* wcnt = cursor + E;             // [warps][E]
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int nt = blockDim.x, n_warps = nt >> 5;
  const int c = blockIdx.x;
  const unsigned lt = (1u << lane) - 1u;

  if (chunk_cnt == nullptr) {
    for (int e = tid; e < E; e += nt) {
      cnt[e] = 0;
      cursor[e] = 0;
    }
    __syncthreads();
    for (int i = tid; i < T * K; i += nt) {
      const int e = idx[i];
      if (e >= 0) atomicAdd(&cnt[e], 1);
    }
  } else {
    for (int e = tid; e < E; e += nt) {
      int tot = 0, before = 0;
      for (int cc = 0; cc < n_chunks; ++cc) {
        const int v = chunk_cnt[(size_t)cc * E + e];
        tot += v;
        if (cc < c) before += v;
      }
      cnt[e] = tot;
      cursor[e] = before;
    }
  }
  __syncthreads();
  if (tid == 0) {
    int s = 0, ts = 0, ts2 = 0, na = 0;
    for (int e = 0; e < E; ++e) {
      if (c == 0) {
        o.offs[e] = s;
        o.tile_offs[e] = ts;
        if (o.tile_offs2) o.tile_offs2[e] = ts2;
        o.n_e[e] = cnt[e];
        if (cnt[e] > 0) o.active[na++] = e;
      }
      cursor[e] += s;
      s += cnt[e];
      ts += (cnt[e] + tile_rows - 1) / tile_rows;
      ts2 += (cnt[e] + tile_rows2 - 1) / tile_rows2;
    }
    if (c == 0) {
      o.offs[E] = s;
      o.tile_offs[E] = ts;
      if (o.tile_offs2) o.tile_offs2[E] = ts2;
      for (int e = na; e < E; ++e) o.active[e] = -1;
      o.active[E] = na;
    }
  }
  __syncthreads();

  int ex[kMaxK];
  const int c_end = chunk_cnt == nullptr ? T : min(T, (c + 1) * nt);
  for (int c0 = c * nt; c0 < c_end; c0 += nt) {
    const int t = c0 + tid;
    const int kt = t < c_end ? kk[t] : 0;
    for (int j = 0; j < K; ++j) ex[j] = (j < kt) ? idx[(size_t)t * K + j] : -1;
    for (int e = lane; e < E; e += 32) wcnt[warp * E + e] = 0;
    __syncwarp();
    for_each_warp_expert(ex, K, [&](int e, unsigned m, int jj) {
      if (lane == 0) wcnt[warp * E + e] = __popc(m);
    });
    __syncthreads();
    for (int e = tid; e < E; e += nt) {
      int run = cursor[e];
      for (int w = 0; w < n_warps; ++w) {
        const int v = wcnt[w * E + e];
        wcnt[w * E + e] = run;
        run += v;
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
    if (t < c_end)
      for (int j = kt; j < K; ++j) o.slot_of[(size_t)t * K + j] = -1;
    __syncthreads();
  }
}

}  // namespace

int permute_chunks(int T) {
  return T <= kPermThreads ? 1 : (T + kChunkThreads - 1) / kChunkThreads;
}

cudaError_t launch_permute(const int32_t* idx, const int32_t* k, const float* psel, int T, int K,
                           int E, int tile_rows, int tile_rows2, PermuteOut o, int32_t* chunk_cnt,
                           cudaStream_t st) {
  const int n_chunks = permute_chunks(T);
  if (n_chunks == 1) {
    const size_t smem = (size_t)(2 * E + (kPermThreads / 32) * E) * sizeof(int);
    return launch_pdl(permute_assign_kernel, dim3(1), dim3(kPermThreads), smem, st, idx, k, psel,
                      T, K, E, tile_rows, tile_rows2, (const int32_t*)nullptr, 1, o);
  }
  cudaError_t e = launch_pdl(permute_count_kernel, dim3(n_chunks), dim3(kChunkThreads),
                             (size_t)E * sizeof(int), st, idx, T, K, E, chunk_cnt);
  if (e != cudaSuccess) return e;
  const size_t smem = (size_t)(2 * E + (kChunkThreads / 32) * E) * sizeof(int);
  return launch_pdl(permute_assign_kernel, dim3(n_chunks), dim3(kChunkThreads), smem, st, idx, k,
                    psel, T, K, E, tile_rows, tile_rows2, (const int32_t*)chunk_cnt, n_chunks,
                    o);
}

}  // namespace eat
