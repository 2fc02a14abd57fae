// Internal declarations shared by the translation units of libeat.so.
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <stdint.h>

#include "../../include/eat.h"

namespace eat {

// Programmatic dependent launch: every kernel of the chain waits for its predecessor's results
// with griddepcontrol.wait before touching global data, and lets its successor be scheduled early
// (the successor's CTAs then only run their local prologue until the wait returns).
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

bool pdl_enabled();

// Compensated fp32 sums ("double-float": a value is the unevaluated sum hi + lo).  GB300's fp64
// pipe runs about two lanes per SM per clock, so one fp64 warp instruction occupies it for ~64
// cycles; sums that need more than fp32 precision use these error-free fp32 steps instead.
// two_sum (Knuth): s = fl(a + b) and s + e == a + b exactly.
__device__ __forceinline__ void two_sum(float a, float b, float& s, float& e) {
  s = a + b;
  const float bb = s - a;
  e = (a - (s - bb)) + (b - bb);
}
// (hi, lo) += v
__device__ __forceinline__ void df_add(float& hi, float& lo, float v) {
  float s, e;
  two_sum(hi, v, s, e);
  hi = s;
  lo += e;
}
// (hi, lo) += (vhi, vlo)
__device__ __forceinline__ void df_add(float& hi, float& lo, float vhi, float vlo) {
  float s, e;
  two_sum(hi, vhi, s, e);
  hi = s;
  lo += e + vlo;
}

// 16-byte global -> shared copy (cp.async, L2 only), its group commit and wait.
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;" ::: "memory");
}
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t st, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = pdl_enabled() ? 1 : 0;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, ((KArgs)args)...);
}

constexpr int kMaxExperts = 256;
constexpr int kMaxK = 16;

// ---------------------------------------------------------------------------------------------
// Router (§3.1-§3.4)
// ---------------------------------------------------------------------------------------------
struct RouteParams {
  float w1, w2, w3, beta, alpha1, alpha2, kappa1, kappa2, ppl_factor, q_lo, q_hi, eps,
      temperature, top_p;
  int clamp, c_mode, mode, smoothing;
  const float* opd_scale;  // [E] or nullptr
  const float* tau_in;     // [T] previous tau_final per token stream (temporal smoothing) or null
  float* tau_out;          // [T] tau_final written back (temporal smoothing, forward calls) or null
  // device-side PPL sign (eat_ppl_update's output) read by the selection kernel instead of the
  // host-side ppl_factor, or null; its factors
  const int32_t* ppl_sign_dev;
  float ppl_up, ppl_down;
};

// Partial router logits: part[s][t][e] = sum over the s-th slice of d of x[t,j] Wr[e,j], as an
// unevaluated fp32 pair (hi, lo) whose exact sum carries the slice's score (see df_add).
// xcopy (or null): the kernel also writes the x it reads there (16-byte aligned, [T, d]); x may
// then be host memory the device can address (a page-locked host buffer).  Only calls for which
// router_copies_x holds can copy.
cudaError_t launch_router_logits(const void* x, int x_bf16, const float* w_router, int T, int d,
                                 int E, int n_split, float2* part, cudaStream_t st,
                                 void* xcopy = nullptr);
bool router_copies_x(const void* x, int x_bf16, const float* w_router, int T, int d);
// Warp-per-token softmax + history score + threshold + selection + renormalisation; the router
// scores are the sum over the n_split slices of part ([split][T][E] fp32 pairs).
cudaError_t launch_route_select(const float2* part, int n_split, const float* b_router, int T,
                                int E, int K, const int64_t* accN, const double* accP,
                                const double* accC, RouteParams rp, int32_t* idx, float* w,
                                int32_t* k, float* psel, cudaStream_t st);
constexpr int kSmallRouterT = 128;  // calls up to this many tokens use the GEMV-style router
int router_split(int T, int d, int E);

// ---------------------------------------------------------------------------------------------
// Permute by expert
// ---------------------------------------------------------------------------------------------
struct PermuteOut {
  int32_t* n_e;        // [E]
  int32_t* offs;       // [E+1] slot offsets per expert
  int32_t* tile_offs;  // [E+1] prefix of ceil(n_e / tile_rows)
  int32_t* tile_offs2; // [E+1] prefix of ceil(n_e / tile_rows2) (a second tile size), or null
  int32_t* perm_tok;   // [T*K] token of each slot
  int32_t* slot_of;    // [T*K] slot of (t, j), -1 for j >= k_t
  float* perm_p;       // [T*K] p of each slot
  int32_t* active;     // [E+1] ascending active experts, active[E] = count
};
int permute_chunks(int T);  // CTAs of the permute of a T-token call
// int32 words of the permute's scratch (a ticket counter, zero between calls, and the per-chunk
// expert counts) for calls of up to Tmax tokens
size_t permute_scratch_ints(int Tmax, int E);
cudaError_t launch_permute(const int32_t* idx, const int32_t* k, const float* psel, int T, int K,
                           int E, int tile_rows, int tile_rows2, PermuteOut o, int32_t* scratch,
                           cudaStream_t st);

// ---------------------------------------------------------------------------------------------
// Expert FFNs
// ---------------------------------------------------------------------------------------------
// Rows ("slots") of group g are row_offs[g] .. row_offs[g+1]-1, or g*uniform_rows ..
// (g+1)*uniform_rows-1 when row_offs == nullptr.  Which input row feeds slot s:
//   kRowGather:   in[row_tok[s]]            (routed experts: gather the token's hidden state)
//   kRowSlot:     in[s]                     (down projection: act rows are in slot order)
//   kRowIdentity: in[s - g*uniform_rows]    (shared experts: every token in order)
enum RowMode { kRowGather = 0, kRowSlot = 1, kRowIdentity = 2 };
struct GroupMap {
  const int32_t* row_offs;   // [G+1] or nullptr (uniform)
  const int32_t* tile_offs;  // [G+1] prefix of row tiles, or nullptr (uniform)
  const int32_t* row_tok;    // [rows] gather index (kRowGather)
  int row_mode;
  int n_groups;
  int uniform_rows;          // rows per group when row_offs == nullptr
  int max_tiles;             // upper bound of the total number of row tiles (grid size)
};

// act[slot, f] = silu(sum_j in[row, j] Wg[g, f, j]) * (sum_j in[row, j] Wu[g, f, j])
cudaError_t launch_ffn_gateup_simt(int dtype_bf16, const void* in, const void* wg, const void* wu,
                                   int Fout, int Kdim, GroupMap gm, void* act, cudaStream_t st);
// out[slot, c] = sum_f act[slot, f] Wd[g, c, f]   (fp32 output)
cudaError_t launch_ffn_down_simt(int dtype_bf16, const void* act, const void* wd, int Dout,
                                 int Kdim, GroupMap gm, float* out, cudaStream_t st);
constexpr int kSimtTileRows = 32;

// ---------------------------------------------------------------------------------------------
// Combine / unpermute and account update
// ---------------------------------------------------------------------------------------------
int combine_col_blocks(int d);  // column segments per token row (norm partials per slot)
cudaError_t launch_combine(int y_bf16, const void* opart, int o_bf16, int n_split,
                           int split_stride_rows, const int32_t* slot_of, const float* w,
                           const void* sout, int s_bf16, int S, int T, int K, int d, void* y,
                           float* nrm_part, const unsigned int* status, cudaStream_t st);
// rows: the call's T * K selection slots (bounds the blocks per expert); chunk_sums:
// [E][account_chunks(rows)] scratch; tickets: [E] words, zero between calls (the kernel leaves
// them zero).  status: the device status word (nonzero: an expert kernel of the call gave up on a
// bounded wait; the update is then skipped); status_mirror: device address of a host-mapped copy
// of the word, written by the block that finishes expert 0, or null.
int account_chunks(long long rows);
cudaError_t launch_account(const int32_t* offs, const float* perm_p, const float* nrm_part, int nb,
                           int E, long long rows, double alpha, int64_t* N, double* P, double* C,
                           int32_t* st_n, double* st_p, double* st_norm, long long* counters,
                           float4* chunk_sums, unsigned int* tickets, const unsigned int* status,
                           unsigned int* status_mirror, cudaStream_t st);

// §3.3 perplexity of a window of token negative log-likelihoods and the sign of its change.
cudaError_t launch_ppl_update(const float* nll, int n, double* state, int32_t* sign,
                              cudaStream_t st);

// Records msg as the text eat_last_error(NULL) returns on this thread (entry points without a
// handle).
void set_thread_error(const char* msg);

}  // namespace eat
