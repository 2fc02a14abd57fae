// Permute by expert: groups the selected (token, expert) pairs of one call by expert so that the
// expert FFNs read contiguous row lists (§3.4: an expert runs only on the tokens that selected it).
//
// Every pair gets a STABLE slot (tokens ascending inside each expert), so every later per-expert
// sum (P_total, the EMA norm mean) runs in a fixed order.  Inside a CTA each warp builds, per
// expert, the 32-bit mask of its lanes (tokens) that chose the expert (shared-memory atomicOr:
// the result does not depend on the order of the ORs); a pair's rank among the warp's pairs of
// its expert is the popcount of the mask below its lane, and the warps' counts are scanned per
// expert.  The work per lane is O(K), whatever the number of distinct experts.
//
// A call of at most 512 tokens runs as one CTA that also counts and writes the offsets.  Larger
// calls are cut into 128-token chunks: a counting kernel writes per-chunk expert counts, and its
// last CTA to finish (a ticket counter that it resets) scans them across chunks and writes the
// offsets; the assignment kernel then places each chunk from its chunk base.
#include "eat_internal.cuh"

namespace eat {

namespace {

constexpr int kSingleMax = 512;  // tokens (and threads) of a single-CTA call at most
constexpr int kChunk = 128;      // tokens (and threads) per CTA of a multi-CTA call
constexpr int kTicketInts = 64;  // the ticket word, padded; the chunk counts follow

__device__ __forceinline__ int ceil_div(int a, int b) { return (a + b - 1) / b; }

// Offsets from the per-expert counts cnt[0..E), run by one full warp: offs, both tile prefixes,
// n_e and the ascending active list.  With base != nullptr, base[e] = offs[e] (may alias cnt).
__device__ void write_offsets(int* cnt, int E, int tile_rows, int tile_rows2, PermuteOut o,
                              int* base, int lane) {
  const unsigned full = 0xffffffffu, lt = (1u << lane) - 1u;
  int s = 0, ts = 0, ts2 = 0, na = 0;
  for (int b = 0; b < E; b += 32) {
    const int e = b + lane;
    const int c = e < E ? cnt[e] : 0;
    const int c1 = ceil_div(c, tile_rows), c2 = ceil_div(c, tile_rows2);
    int v0 = c, v1 = c1, v2 = c2;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int a0 = __shfl_up_sync(full, v0, off);
      const int a1 = __shfl_up_sync(full, v1, off);
      const int a2 = __shfl_up_sync(full, v2, off);
      if (lane >= off) {
        v0 += a0;
        v1 += a1;
        v2 += a2;
      }
    }
    const unsigned act = __ballot_sync(full, e < E && c > 0);
    if (e < E) {
      o.offs[e] = s + v0 - c;
      o.tile_offs[e] = ts + v1 - c1;
      if (o.tile_offs2) o.tile_offs2[e] = ts2 + v2 - c2;
      o.n_e[e] = c;
      if (c > 0) o.active[na + __popc(act & lt)] = e;
      if (base) base[e] = s + v0 - c;
    }
    s += __shfl_sync(full, v0, 31);
    ts += __shfl_sync(full, v1, 31);
    ts2 += __shfl_sync(full, v2, 31);
    na += __popc(act);
  }
  if (lane == 0) {
    o.offs[E] = s;
    o.tile_offs[E] = ts;
    if (o.tile_offs2) o.tile_offs2[E] = ts2;
    o.active[E] = na;
  }
  for (int e = na + lane; e < E; e += 32) o.active[e] = -1;
}

// Per-chunk expert counts of a multi-CTA call; the last CTA to finish turns chunk_cnt[c][e] into
// the exclusive prefix over chunks and writes the offsets.
template <int KM>
__global__ void __launch_bounds__(kChunk)
permute_count_kernel(const int32_t* __restrict__ idx, const int32_t* __restrict__ kk, int T,
                     int K, int E, int tile_rows, int tile_rows2, int32_t* chunk_cnt,
                     int n_chunks, unsigned* ticket, PermuteOut o) {
  extern __shared__ int cnt[];  // [E]
  __shared__ int is_last;
  pdl_wait();
  pdl_launch_dependents();
  const int tid = threadIdx.x, nt = blockDim.x;
  for (int e = tid; e < E; e += nt) cnt[e] = 0;
  __syncthreads();
  const int t = blockIdx.x * nt + tid;
  const int kt = t < T ? kk[t] : 0;
#pragma unroll
  for (int j = 0; j < KM; ++j)
    if (j < K && j < kt) atomicAdd(&cnt[idx[(size_t)t * K + j]], 1);
  __syncthreads();
  for (int e = tid; e < E; e += nt) chunk_cnt[(size_t)blockIdx.x * E + e] = cnt[e];
  __threadfence();
  __syncthreads();
  if (tid == 0) is_last = atomicAdd(ticket, 1u) == (unsigned)(n_chunks - 1);
  __syncthreads();
  if (!is_last) return;
  __threadfence();
  for (int e = tid; e < E; e += nt) {
    int pre = 0;
    int c = 0;
    for (; c + 8 <= n_chunks; c += 8) {
      int v[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) v[u] = __ldcg(&chunk_cnt[(size_t)(c + u) * E + e]);
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        chunk_cnt[(size_t)(c + u) * E + e] = pre;
        pre += v[u];
      }
    }
    for (; c < n_chunks; ++c) {
      const int v = __ldcg(&chunk_cnt[(size_t)c * E + e]);
      chunk_cnt[(size_t)c * E + e] = pre;
      pre += v;
    }
    cnt[e] = pre;
  }
  __syncthreads();
  if (tid < 32) write_offsets(cnt, E, tile_rows, tile_rows2, o, nullptr, tid);
  if (tid == 0) *ticket = 0u;
}

// Slot assignment of blockDim.x consecutive tokens.  chunk_base == nullptr: a single-CTA call
// (T <= blockDim.x) that counts and writes the offsets itself; otherwise CTA c starts expert e
// at offs[e] + chunk_base[c][e].
template <int KM>
__global__ void __launch_bounds__(kSingleMax)
permute_assign_kernel(const int32_t* __restrict__ idx, const int32_t* __restrict__ kk,
                      const float* __restrict__ psel, int T, int K, int E, int tile_rows,
                      int tile_rows2, const int32_t* __restrict__ chunk_base, PermuteOut o) {
  extern __shared__ unsigned sm[];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int nt = blockDim.x, nw = nt >> 5;
  unsigned* mask = sm;                    // [nw][E] lanes of each warp that chose e
  int* wbase = (int*)(mask + nw * E);     // [nw][E] first slot of each warp's pairs of e
  int* cnt = wbase + nw * E;              // [E] counts, then offsets (single CTA)
  const unsigned lt = (1u << lane) - 1u;
  pdl_wait();
  pdl_launch_dependents();
  for (int i = tid; i < nw * E; i += nt) mask[i] = 0u;
  __syncthreads();
  const int t = blockIdx.x * nt + tid;
  const int kt = t < T ? kk[t] : 0;
  int ex[KM];
#pragma unroll
  for (int j = 0; j < KM; ++j) ex[j] = (j < K && j < kt) ? idx[(size_t)t * K + j] : -1;
#pragma unroll
  for (int j = 0; j < KM; ++j)
    if (ex[j] >= 0) atomicOr(&mask[warp * E + ex[j]], 1u << lane);
  __syncthreads();
  if (chunk_base == nullptr) {
    for (int e = tid; e < E; e += nt) {
      int c = 0;
      for (int w = 0; w < nw; ++w) c += __popc(mask[w * E + e]);
      cnt[e] = c;
    }
    __syncthreads();
    if (warp == 0) write_offsets(cnt, E, tile_rows, tile_rows2, o, cnt, lane);
    __syncthreads();
  }
  for (int e = tid; e < E; e += nt) {
    int run = chunk_base ? o.offs[e] + chunk_base[(size_t)blockIdx.x * E + e] : cnt[e];
    for (int w = 0; w < nw; ++w) {
      wbase[w * E + e] = run;
      run += __popc(mask[w * E + e]);
    }
  }
  __syncthreads();
#pragma unroll
  for (int j = 0; j < KM; ++j) {
    const int e = ex[j];
    if (e >= 0) {
      const int slot = wbase[warp * E + e] + __popc(mask[warp * E + e] & lt);
      o.perm_tok[slot] = t;
      o.slot_of[(size_t)t * K + j] = slot;
      o.perm_p[slot] = psel[(size_t)t * K + j];
    } else if (j < K && t < T) {
      o.slot_of[(size_t)t * K + j] = -1;
    }
  }
}

template <int KM>
cudaError_t launch_permute_k(const int32_t* idx, const int32_t* k, const float* psel, int T,
                             int K, int E, int tile_rows, int tile_rows2, PermuteOut o,
                             int32_t* scratch, cudaStream_t st) {
  if (T <= kSingleMax) {
    const int nt = (T + 31) / 32 * 32;
    const size_t smem = (size_t)(2 * (nt / 32) * E + E) * sizeof(int);
    return launch_pdl(permute_assign_kernel<KM>, dim3(1), dim3(nt), smem, st, idx, k, psel, T,
                      K, E, tile_rows, tile_rows2, (const int32_t*)nullptr, o);
  }
  const int n_chunks = permute_chunks(T);
  unsigned* ticket = (unsigned*)scratch;
  int32_t* chunk_cnt = scratch + kTicketInts;
  cudaError_t e = launch_pdl(permute_count_kernel<KM>, dim3(n_chunks), dim3(kChunk),
                             (size_t)E * sizeof(int), st, idx, k, T, K, E, tile_rows, tile_rows2,
                             chunk_cnt, n_chunks, ticket, o);
  if (e != cudaSuccess) return e;
  const size_t smem = (size_t)(2 * (kChunk / 32) * E + E) * sizeof(int);
  return launch_pdl(permute_assign_kernel<KM>, dim3(n_chunks), dim3(kChunk), smem, st, idx, k,
                    psel, T, K, E, tile_rows, tile_rows2, (const int32_t*)chunk_cnt, o);
}

}  // namespace

int permute_chunks(int T) { return T <= kSingleMax ? 1 : (T + kChunk - 1) / kChunk; }

size_t permute_scratch_ints(int Tmax, int E) {
  return kTicketInts + (size_t)permute_chunks(Tmax) * E;
}

cudaError_t launch_permute(const int32_t* idx, const int32_t* k, const float* psel, int T, int K,
                           int E, int tile_rows, int tile_rows2, PermuteOut o, int32_t* scratch,
                           cudaStream_t st) {
  if (K <= 2)
    return launch_permute_k<2>(idx, k, psel, T, K, E, tile_rows, tile_rows2, o, scratch, st);
  if (K <= 4)
    return launch_permute_k<4>(idx, k, psel, T, K, E, tile_rows, tile_rows2, o, scratch, st);
  if (K <= 8)
    return launch_permute_k<8>(idx, k, psel, T, K, E, tile_rows, tile_rows2, o, scratch, st);
  return launch_permute_k<16>(idx, k, psel, T, K, E, tile_rows, tile_rows2, o, scratch, st);
}

}  // namespace eat
