// extern "C" boundary of libeat.so (declared in include/eat.h): handle, argument validation,
// workspace, and the stream-ordered launch sequence of one EAT MoE layer call.
#include "eat_internal.cuh"
#if __has_include(<nvtx3/nvToolsExt.h>)
#include <nvtx3/nvToolsExt.h>
#define EAT_HAVE_NVTX 1
#endif
#include "ffn_tc.cuh"

#include <algorithm>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <new>
#include <string>
#include <vector>

using namespace eat;

struct eat_handle {
  eat_layer_desc desc;
  eat_params prm;
  int E = 0, d = 0, F = 0, S = 0, Fs = 0, Tmax = 0, K = 0;
  bool bf16 = false;  // hidden states and outputs in bf16
  bool w8 = false;    // e4m3 expert weights (tensor-core kernels, kind::f8f6f4)
  int backend = 0;  // 0 CUDA-core kernels (fp32 layers), 1 tcgen05 kernels (bf16 / fp8 layers)
  size_t elt = 4;

  void* mem = nullptr;
  int64_t* N = nullptr;
  double* P = nullptr;
  double* C = nullptr;
  int32_t* st_n = nullptr;
  double* st_p = nullptr;
  double* st_norm = nullptr;
  long long* counters = nullptr;  // [4] on the device: calls, sum |union|, sum k, spare
  float2* logit_part = nullptr;   // [split][T][E] partial router scores (fp32 pairs)
  int32_t* idx = nullptr;
  float* w = nullptr;
  int32_t* k = nullptr;
  float* psel = nullptr;
  PermuteOut perm{};
  void* act = nullptr;    // [Tmax*K, F]
  float* opart = nullptr; // [splits][Tmax*K, d]
  float* nrm_part = nullptr; // [Tmax*K, segments] partial sums of squares of expert rows
  int nb = 1;                 // column segments per row in the combine kernel
  void* sact = nullptr;   // [S*Tmax, Fs]
  float* sout = nullptr;  // [S*Tmax, d] (fp32; bf16 on the tensor-core path)
  TcWork q;               // fp8 layers: B-operand planes and scales
  void* xstage = nullptr; // [2][Tmax, d] inputs of host-buffer calls, used in turn
  void* ystage = nullptr; // [Tmax, d]
  // host-buffer calls copy their input on their own stream, into the staging buffer the call
  // before last used, so the copy overlaps the previous call's kernels (created on first use)
  cudaStream_t copy_st = nullptr;
  // shared experts run on a stream of the handle, forked from the call's stream before routing
  cudaStream_t side_st = nullptr;
  cudaEvent_t ev_fork = nullptr, ev_join = nullptr;
  cudaEvent_t ev_copied[2] = {nullptr, nullptr};  // input copy i done (copy stream)
  cudaEvent_t ev_done[2] = {nullptr, nullptr};    // the call that read buffer i done (its stream)
  int stage_i = 0;
  void* xperm = nullptr;  // [Tmax*K, d] gathered token rows (tensor-core path)
  unsigned int* status = nullptr;  // device status word: bounded waits that expired
  // host-mapped copy of the status word, written by the account kernel of every forward call
  // (the host pointer is read by the entry points without a synchronisation)
  unsigned int* mirror_host = nullptr;
  unsigned int* mirror_dev = nullptr;
  bool failed = false;  // a call saw the status word set: calls fail until eat_reset_accounts
  int32_t* chunk_cnt = nullptr;    // permute scratch: ticket word, then [chunks][E] counts
  float4* acc_sums = nullptr;        // account scratch: [E][chunks] compensated chunk sums
  unsigned int* acc_tickets = nullptr;  // [E] account tickets (zero between calls)
  long long opart_rows = 0;
  float* tau_state = nullptr;  // caller-owned [Tmax] previous tau_final per stream, or null
  const int32_t* ppl_sign_src = nullptr;  // caller-owned device PPL sign (eat_ppl_update), or null

  TcLayer tc{};

  long long launches = 0;
  std::string err;

  bool prof = false;
  int prof_cap = 0;
  std::vector<cudaEvent_t> ev;  // 2 per recorded launch
  std::vector<int> ev_kind;
  int prof_n = 0;
};

namespace {

thread_local std::string g_err;

eat_status fail(eat_handle* h, eat_status s, const std::string& msg) {
  if (h) h->err = msg;
  else g_err = msg;
  return s;
}

eat_status cuda_fail(eat_handle* h, cudaError_t e, const char* what) {
  return fail(h, EAT_ERR_CUDA, std::string(what) + ": " + cudaGetErrorString(e));
}

enum Kind {
  kRoute = 0, kPermute, kUp, kDown, kSUp, kSDown, kCombine, kAccount, kSelect, kGather, kKinds
};

// Run one launch, optionally bracketed by CUDA events for the per-kernel profile.
inline void nvtx_push(const char* what) {
#ifdef EAT_HAVE_NVTX
  nvtxRangePushA(what);
#else
  (void)what;
#endif
}
inline void nvtx_pop() {
#ifdef EAT_HAVE_NVTX
  nvtxRangePop();
#endif
}

template <typename Fn>
eat_status launch(eat_handle* h, int kind, cudaStream_t st, const char* what, Fn&& fn) {
  const bool rec = h->prof && h->prof_n < h->prof_cap;
  if (rec) cudaEventRecord(h->ev[2 * h->prof_n], st);
  nvtx_push(what);  // a named range per launch for timeline tools (no-op without one attached)
  const cudaError_t e = fn();
  nvtx_pop();
  ++h->launches;
  if (rec) {
    cudaEventRecord(h->ev[2 * h->prof_n + 1], st);
    h->ev_kind[h->prof_n] = kind;
    ++h->prof_n;
  }
  if (e != cudaSuccess) return cuda_fail(h, e, what);
  return EAT_OK;
}

#define EAT_TRY(x)                    \
  do {                                \
    eat_status s__ = (x);             \
    if (s__ != EAT_OK) return s__;    \
  } while (0)

RouteParams route_params(const eat_params& p, int ppl_sign) {
  RouteParams r;
  r.w1 = (float)p.w1;
  r.w2 = (float)p.w2;
  r.w3 = (float)p.w3;
  r.beta = (float)p.beta;
  r.alpha1 = (float)p.alpha1;
  r.alpha2 = (float)p.alpha2;
  r.kappa1 = (float)p.kappa1;
  r.kappa2 = (float)p.kappa2;
  r.ppl_factor = ppl_sign > 0 ? (float)p.ppl_up : (ppl_sign < 0 ? (float)p.ppl_down : 1.0f);
  r.q_lo = (float)p.q_lo;
  r.q_hi = (float)p.q_hi;
  r.eps = (float)p.eps;
  r.temperature = (float)p.temperature;
  r.clamp = p.clamp_enabled;
  r.c_mode = p.c_mode;
  r.mode = p.router_mode;
  r.top_p = (float)p.top_p;
  r.smoothing = p.smoothing_mode;
  r.opd_scale = nullptr;
  r.tau_in = nullptr;
  r.tau_out = nullptr;
  r.ppl_sign_dev = nullptr;
  r.ppl_up = (float)p.ppl_up;
  r.ppl_down = (float)p.ppl_down;
  return r;
}

size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

// A kernel of an earlier call gave up on a bounded wait (the status word is set): that call's
// outputs were NaN and the accounts stayed as they were; the handle refuses further calls until
// eat_reset_accounts.
eat_status check_state(eat_handle* h) {
  const unsigned int sw = h->mirror_host ? *(volatile unsigned int*)h->mirror_host : 0u;
  if (!h->failed && sw == 0u) return EAT_OK;
  h->failed = true;
  char msg[200];
  snprintf(msg, sizeof msg,
           "a kernel of an earlier call gave up on a bounded wait (status word 0x%x): its outputs "
           "were NaN and the accounts were left unchanged; eat_reset_accounts clears the state",
           sw);
  return fail(h, EAT_ERR_STATE, msg);
}

eat_status check_call(eat_handle* h, const void* x, int32_t T, int32_t ppl_sign) {
  if (!h) return fail(nullptr, EAT_ERR_INVALID_ARG, "null handle");
  if (!x) return fail(h, EAT_ERR_INVALID_ARG, "x is NULL");
  if (T < 1 || T > h->Tmax)
    return fail(h, EAT_ERR_INVALID_ARG,
                "T=" + std::to_string(T) + " outside [1, max_tokens=" + std::to_string(h->Tmax) +
                    "]");
  if (ppl_sign < -1 || ppl_sign > 1)
    return fail(h, EAT_ERR_INVALID_ARG, "ppl_sign must be -1, 0 or +1");
  if (((uintptr_t)x & 15) != 0)
    return fail(h, EAT_ERR_INVALID_ARG, "x must be 16-byte aligned");
  return check_state(h);
}

// Router + selection into (idx, w, k, psel).  x_host (or null): the router kernel reads the
// tokens there (a page-locked host buffer) and writes them to x, which later kernels read.
eat_status run_route(eat_handle* h, const void* x, int T, int ppl_sign, int32_t* idx, float* w,
                     int32_t* k, float* psel, bool write_tau, cudaStream_t st,
                     const void* x_host = nullptr) {
  RouteParams rp = route_params(h->prm, ppl_sign);
  rp.opd_scale = h->desc.opd_scale;
  rp.ppl_sign_dev = h->ppl_sign_src;
  if (h->prm.smoothing_mode == EAT_SMOOTH_TEMPORAL && h->tau_state) {
    rp.tau_in = h->tau_state;
    rp.tau_out = write_tau ? h->tau_state : nullptr;
  }
  const int split = router_split(T, h->d, h->E);
  EAT_TRY(launch(h, kRoute, st, "router logits", [&] {
    if (x_host)
      return launch_router_logits(x_host, h->bf16, h->desc.w_router, T, h->d, h->E, split,
                                  h->logit_part, st, const_cast<void*>(x));
    return launch_router_logits(x, h->bf16, h->desc.w_router, T, h->d, h->E, split,
                                h->logit_part, st);
  }));
  EAT_TRY(launch(h, kSelect, st, "route select", [&] {
    return launch_route_select(h->logit_part, split, h->desc.b_router, T, h->E, h->K, h->N,
                               h->P, h->C, rp, idx, w, k, psel, st);
  }));
  return EAT_OK;
}

// The always-on shared experts of §3.1 (weight 1).  They read only x, so a small call runs them on
// the handle's side stream while the routing kernels, which leave most SMs idle, run on its own.
eat_status run_shared(eat_handle* h, const TcCall& c, const void* x, int T, cudaStream_t ss) {
  if (h->backend == 1) {
    auto split = [&](TcSplit which, const char* what) {
      return launch(h, kGather, ss, what, [&] { return tc_launch_split(h->tc, c, which, ss); });
    };
    if (h->w8) EAT_TRY(split(TcSplit::kTokenX, "split x (tokens)"));
    EAT_TRY(launch(h, kSUp, ss, "tc shared gate/up",
                   [&] { return tc_launch_up(h->tc, c, true, ss); }));
    if (h->w8) EAT_TRY(split(TcSplit::kSharedAct, "split shared activations"));
    return launch(h, kSDown, ss, "tc shared down",
                  [&] { return tc_launch_down(h->tc, c, true, 1, ss); });
  }
  const int tpg = (T + kSimtTileRows - 1) / kSimtTileRows;
  GroupMap gs{nullptr, nullptr, nullptr, kRowIdentity, h->S, T, tpg * h->S};
  EAT_TRY(launch(h, kSUp, ss, "shared gate/up", [&] {
    return launch_ffn_gateup_simt(h->bf16, x, h->desc.ws_gate, h->desc.ws_up, h->Fs, h->d, gs,
                                  h->sact, ss);
  }));
  return launch(h, kSDown, ss, "shared down", [&] {
    return launch_ffn_down_simt(h->bf16, h->sact, h->desc.ws_down, h->d, h->Fs, gs,
                                (float*)h->sout, ss);
  });
}

// Small calls, whose shared-expert GEMMs have fewer work units than the GPU has SMs, run those
// GEMMs on the side stream next to the routing kernels; larger calls fill the GPU with them alone
// and keep them in the call's stream after the routed experts.
bool shared_on_side_stream(const eat_handle* h, int T, int tile_rows) {
  if (h->S == 0 || h->backend != 1) return false;
  const long long units =
      (long long)h->S * ((h->Fs + 127) / 128) * ((T + tile_rows - 1) / tile_rows);
  return units < h->tc.num_sms;
}

// x_host (or null): see run_route; the caller has checked that the router copies x for this call
// and that no shared expert reads x before the router has run (side stream).
eat_status run_forward(eat_handle* h, const void* x, int T, int ppl_sign, void* y,
                       int32_t* idx_opt, float* w_opt, int32_t* k_opt, cudaStream_t st,
                       const void* x_host = nullptr) {
  const int tile_rows = h->backend == 1 ? tc_tile_rows(h->tc, T) : kSimtTileRows;
  const int tile_rows_down = h->backend == 1 ? tc_tile_rows_down(h->tc, T) : kSimtTileRows;
  TcCall c;
  c.x = x;
  c.T = T;
  c.tile_rows = tile_rows;
  c.tile_rows_down = tile_rows_down;
  c.offs = h->perm.offs;
  c.tile_offs = h->perm.tile_offs;
  c.tile_offs_down = h->perm.tile_offs2;
  c.perm_tok = h->perm.perm_tok;
  c.xperm = h->xperm;
  c.act = h->act;
  c.opart = h->opart;
  c.sact = h->sact;
  c.sout = h->sout;
  c.status = h->status;
  const bool side = shared_on_side_stream(h, T, tile_rows);
  // large calls on SM pairs: the shared experts' units follow the routed ones in the same launches
  c.fold_shared = !side && h->backend == 1 && tc_folds_shared(h->tc, T);
  if (side) {
    // fork: the side stream starts after everything enqueued on st so far (x written, the
    // previous call's combine done with the shared outputs)
    cudaError_t e = cudaEventRecord(h->ev_fork, st);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(h->side_st, h->ev_fork, 0);
    if (e != cudaSuccess) return cuda_fail(h, e, "shared-expert stream fork");
    EAT_TRY(run_shared(h, c, x, T, h->side_st));
    e = cudaEventRecord(h->ev_join, h->side_st);
    if (e != cudaSuccess) return cuda_fail(h, e, "shared-expert stream join");
  }
  if (x_host && side) return fail(h, EAT_ERR_UNSUPPORTED, "host-read input with side-stream experts");
  EAT_TRY(run_route(h, x, T, ppl_sign, h->idx, h->w, h->k, h->psel, true, st, x_host));
  EAT_TRY(launch(h, kPermute, st, "permute", [&] {
    return launch_permute(h->idx, h->k, h->psel, T, h->K, h->E, tile_rows, tile_rows_down,
                          h->perm, h->chunk_cnt, st);
  }));
  const int rows = T * h->K;
  int n_split = 1;
  if (h->backend == 1) {
    n_split = tc_down_split(h->tc, T);
    // fp8 layers: each GEMM's B operand first becomes e4m3 hi/lo planes (the routed x rows are
    // gathered into slot order on the way)
    auto split = [&](TcSplit which, const char* what) {
      return launch(h, kGather, st, what, [&] { return tc_launch_split(h->tc, c, which, st); });
    };
    if (h->w8)
      EAT_TRY(split(TcSplit::kSlotX, "split x (slots)"));
    else if (!tc_gathers_in_kernel(h->tc, T))
      EAT_TRY(launch(h, kGather, st, "gather rows",
                     [&] { return tc_launch_gather(h->tc, c, st); }));
    EAT_TRY(launch(h, kUp, st, "tc gate/up", [&] { return tc_launch_up(h->tc, c, false, st); }));
    if (h->w8) EAT_TRY(split(TcSplit::kAct, "split activations"));
    EAT_TRY(launch(h, kDown, st, "tc down",
                   [&] { return tc_launch_down(h->tc, c, false, n_split, st); }));
  } else {
    GroupMap gm{h->perm.offs, h->perm.tile_offs, h->perm.perm_tok, kRowGather, h->E, 0,
                (rows + kSimtTileRows - 1) / kSimtTileRows + h->E};
    EAT_TRY(launch(h, kUp, st, "ffn gate/up", [&] {
      return launch_ffn_gateup_simt(h->bf16, x, h->desc.w_gate, h->desc.w_up, h->F, h->d, gm,
                                    h->act, st);
    }));
    EAT_TRY(launch(h, kDown, st, "ffn down", [&] {
      return launch_ffn_down_simt(h->bf16, h->act, h->desc.w_down, h->d, h->F, gm, h->opart, st);
    }));
  }
  if (side) {
    const cudaError_t e = cudaStreamWaitEvent(st, h->ev_join, 0);  // join before the combine
    if (e != cudaSuccess) return cuda_fail(h, e, "shared-expert stream join");
  } else if (h->S > 0 && !c.fold_shared) {
    EAT_TRY(run_shared(h, c, x, T, st));
  }
  EAT_TRY(launch(h, kCombine, st, "combine", [&] {
    const int tc = h->backend == 1;
    return launch_combine(h->bf16, h->opart, tc && n_split == 1, n_split, rows, h->perm.slot_of,
                          h->w, h->sout, tc, h->S, T, h->K, h->d, y, h->nrm_part, h->status, st);
  }));
  EAT_TRY(launch(h, kAccount, st, "account update", [&] {
    return launch_account(h->perm.offs, h->perm.perm_p, h->nrm_part, h->nb, h->E, rows,
                          h->prm.alpha, h->N, h->P, h->C, h->st_n, h->st_p, h->st_norm,
                          h->counters, h->acc_sums, h->acc_tickets, h->status, h->mirror_dev, st);
  }));
  if (idx_opt || w_opt || k_opt) {
    cudaError_t e = cudaSuccess;
    if (idx_opt && e == cudaSuccess)
      e = cudaMemcpyAsync(idx_opt, h->idx, sizeof(int32_t) * rows, cudaMemcpyDeviceToDevice, st);
    if (w_opt && e == cudaSuccess)
      e = cudaMemcpyAsync(w_opt, h->w, sizeof(float) * rows, cudaMemcpyDeviceToDevice, st);
    if (k_opt && e == cudaSuccess)
      e = cudaMemcpyAsync(k_opt, h->k, sizeof(int32_t) * T, cudaMemcpyDeviceToDevice, st);
    if (e != cudaSuccess) return cuda_fail(h, e, "routing copy-out");
  }
  return EAT_OK;
}

void free_handle(eat_handle* h) {
  if (!h) return;
  for (cudaEvent_t e : h->ev) cudaEventDestroy(e);
  for (int i = 0; i < 2; ++i) {
    if (h->ev_copied[i]) cudaEventDestroy(h->ev_copied[i]);
    if (h->ev_done[i]) cudaEventDestroy(h->ev_done[i]);
  }
  if (h->copy_st) cudaStreamDestroy(h->copy_st);
  if (h->ev_fork) cudaEventDestroy(h->ev_fork);
  if (h->ev_join) cudaEventDestroy(h->ev_join);
  if (h->side_st) cudaStreamDestroy(h->side_st);
  tc_destroy(h->tc);
  if (h->mirror_host) cudaFreeHost(h->mirror_host);
  if (h->mem) cudaFree(h->mem);
  delete h;
}

}  // namespace

extern "C" {

eat_status eat_default_params(eat_params* p) {
  if (!p) return fail(nullptr, EAT_ERR_INVALID_ARG, "params is NULL");
  p->alpha = 0.95;
  p->w1 = 0.3;
  p->w2 = 0.3;
  p->w3 = 0.4;
  p->beta = 0.6;
  p->alpha1 = 0.5;
  p->alpha2 = 1.0;
  p->kappa1 = 0.7;
  p->kappa2 = 0.3;
  p->ppl_up = 1.2;
  p->ppl_down = 0.9;
  p->q_lo = 0.10;
  p->q_hi = 0.90;
  p->eps = 1e-8;
  p->temperature = 1.0;
  p->max_k = 2;
  p->clamp_enabled = 1;
  p->c_mode = EAT_C_SUM;
  p->router_mode = EAT_ROUTER_EAT;
  p->top_p = 0.6;
  p->smoothing_mode = EAT_SMOOTH_CALL;
  return EAT_OK;
}

eat_status eat_create(const eat_layer_desc* desc, const eat_params* params, eat_handle** out) {
  if (!out) return fail(nullptr, EAT_ERR_INVALID_ARG, "out is NULL");
  *out = nullptr;
  if (!desc || !params) return fail(nullptr, EAT_ERR_INVALID_ARG, "desc or params is NULL");
  const eat_layer_desc& D = *desc;
  const eat_params& Pm = *params;
  if (D.n_experts < 1 || D.n_experts > kMaxExperts)
    return fail(nullptr, EAT_ERR_UNSUPPORTED, "n_experts must be in [1, 256]");
  if (D.d_model < 64 || D.d_model % 64 || D.d_ff < 64 || D.d_ff % 64)
    return fail(nullptr, EAT_ERR_UNSUPPORTED, "d_model and d_ff must be positive multiples of 64");
  if (D.n_shared < 0 || (D.n_shared > 0 && (D.d_ff_shared < 64 || D.d_ff_shared % 64)))
    return fail(nullptr, EAT_ERR_UNSUPPORTED, "d_ff_shared must be a positive multiple of 64");
  if (D.max_tokens < 1 || D.max_tokens > 65536)
    return fail(nullptr, EAT_ERR_INVALID_ARG, "max_tokens must be in [1, 65536]");
  if (!((D.wdtype == EAT_F32 && D.xdtype == EAT_F32) ||
        (D.wdtype == EAT_BF16 && D.xdtype == EAT_BF16) ||
        (D.wdtype == EAT_FP8_E4M3 && D.xdtype == EAT_BF16)))
    return fail(nullptr, EAT_ERR_UNSUPPORTED,
                "(wdtype, xdtype) must be (F32, F32), (BF16, BF16) or (FP8_E4M3, BF16)");
  if (D.wdtype == EAT_FP8_E4M3 &&
      (!D.w_gate_scale || !D.w_up_scale || !D.w_down_scale ||
       (D.n_shared > 0 && (!D.ws_gate_scale || !D.ws_up_scale || !D.ws_down_scale))))
    return fail(nullptr, EAT_ERR_INVALID_ARG, "fp8 weights need every per-row scale array");
  if (!D.w_router || !D.w_gate || !D.w_up || !D.w_down)
    return fail(nullptr, EAT_ERR_INVALID_ARG, "router or expert weight pointer is NULL");
  if (D.n_shared > 0 && (!D.ws_gate || !D.ws_up || !D.ws_down))
    return fail(nullptr, EAT_ERR_INVALID_ARG, "shared expert weight pointer is NULL");
  const uintptr_t al = (uintptr_t)D.w_gate | (uintptr_t)D.w_up | (uintptr_t)D.w_down |
                       (uintptr_t)(D.n_shared > 0 ? ((uintptr_t)D.ws_gate | (uintptr_t)D.ws_up |
                                                     (uintptr_t)D.ws_down)
                                                  : 0);
  if (al & 15) return fail(nullptr, EAT_ERR_INVALID_ARG, "weights must be 16-byte aligned");
  if (Pm.max_k < 1 || Pm.max_k > kMaxK || Pm.max_k > D.n_experts)
    return fail(nullptr, EAT_ERR_INVALID_ARG, "max_k must be in [1, min(E, 16)]");
  if (!(Pm.temperature > 0.0)) return fail(nullptr, EAT_ERR_INVALID_ARG, "temperature <= 0");
  if (!(Pm.alpha >= 0.0 && Pm.alpha <= 1.0))
    return fail(nullptr, EAT_ERR_INVALID_ARG, "alpha outside [0, 1]");
  if (!(Pm.q_lo >= 0.0 && Pm.q_lo <= Pm.q_hi && Pm.q_hi <= 1.0))
    return fail(nullptr, EAT_ERR_INVALID_ARG, "need 0 <= q_lo <= q_hi <= 1");
  if (Pm.c_mode != EAT_C_SUM && Pm.c_mode != EAT_C_RAW)
    return fail(nullptr, EAT_ERR_INVALID_ARG, "bad c_mode");
  if (Pm.smoothing_mode != EAT_SMOOTH_CALL && Pm.smoothing_mode != EAT_SMOOTH_TEMPORAL)
    return fail(nullptr, EAT_ERR_INVALID_ARG, "bad smoothing_mode");
  if (Pm.router_mode < EAT_ROUTER_EAT || Pm.router_mode > EAT_ROUTER_TOPP)
    return fail(nullptr, EAT_ERR_INVALID_ARG, "bad router_mode");
  if (Pm.router_mode == EAT_ROUTER_TOPP && !(Pm.top_p > 0.0 && Pm.top_p <= 1.0))
    return fail(nullptr, EAT_ERR_INVALID_ARG, "top_p must be in (0, 1]");

  eat_handle* h = new (std::nothrow) eat_handle();
  if (!h) return fail(nullptr, EAT_ERR_OOM, "host allocation failed");
  h->desc = D;
  h->prm = Pm;
  h->E = D.n_experts;
  h->d = D.d_model;
  h->F = D.d_ff;
  h->S = D.n_shared;
  h->Fs = D.n_shared > 0 ? D.d_ff_shared : 0;
  h->Tmax = D.max_tokens;
  h->K = Pm.max_k;
  h->bf16 = D.xdtype == EAT_BF16;  // hidden states (and y) in bf16
  h->w8 = D.wdtype == EAT_FP8_E4M3;
  h->elt = h->bf16 ? 2 : 4;
  h->backend = h->bf16 ? 1 : 0;
  h->opart_rows = (long long)h->Tmax * h->K;

  if (h->backend == 1) {
    const char* msg = nullptr;
    if (tc_configure(h->tc, D, h->K, h->Tmax, &msg) != 0) {
      std::string m = msg ? msg : "tensor-core setup failed";
      free_handle(h);
      return fail(nullptr, EAT_ERR_UNSUPPORTED, m);
    }
    h->opart_rows = tc_opart_rows(h->tc);
  }

  int max_lsplit = 0;
  for (int T = 1; T <= h->Tmax; ++T)
    max_lsplit = std::max(max_lsplit, router_split(T, h->d, h->E) * T);

  const size_t rows = (size_t)h->Tmax * h->K;
  struct Part { void** p; size_t bytes; };
  std::vector<Part> parts;
  auto add = [&](void* pp, size_t bytes) { parts.push_back({(void**)pp, bytes}); };
  add(&h->N, sizeof(int64_t) * h->E);
  add(&h->P, sizeof(double) * h->E);
  add(&h->C, sizeof(double) * h->E);
  add(&h->st_n, sizeof(int32_t) * h->E);
  add(&h->st_p, sizeof(double) * h->E);
  add(&h->st_norm, sizeof(double) * h->E);
  add(&h->counters, sizeof(long long) * 4);
  add(&h->status, sizeof(unsigned int) * 4);
  add(&h->logit_part, sizeof(float2) * (size_t)max_lsplit * h->E);
  add(&h->idx, sizeof(int32_t) * rows);
  add(&h->w, sizeof(float) * rows);
  add(&h->k, sizeof(int32_t) * h->Tmax);
  add(&h->psel, sizeof(float) * rows);
  add(&h->perm.n_e, sizeof(int32_t) * h->E);
  add(&h->perm.offs, sizeof(int32_t) * (h->E + 1));
  add(&h->perm.tile_offs, sizeof(int32_t) * (h->E + 1));
  add(&h->perm.tile_offs2, sizeof(int32_t) * (h->E + 1));
  add(&h->perm.perm_tok, sizeof(int32_t) * rows);
  add(&h->perm.slot_of, sizeof(int32_t) * rows);
  add(&h->perm.perm_p, sizeof(float) * rows);
  add(&h->perm.active, sizeof(int32_t) * (h->E + 1));
  add(&h->act, h->elt * rows * h->F);
  add(&h->opart, sizeof(float) * (size_t)h->opart_rows * h->d);
  h->nb = combine_col_blocks(h->d);
  add(&h->nrm_part, sizeof(float) * rows * h->nb);
  if (h->S > 0) {
    add(&h->sact, h->elt * (size_t)h->S * h->Tmax * h->Fs);
    add(&h->sout, sizeof(float) * (size_t)h->S * h->Tmax * h->d);
  }
  if (h->backend == 1 && !h->w8) {
    add(&h->xperm, h->elt * rows * h->d);
  }
  add(&h->chunk_cnt, sizeof(int32_t) * permute_scratch_ints(h->Tmax, h->E));
  add(&h->acc_sums, sizeof(float4) * (size_t)h->E * account_chunks((long long)rows));
  add(&h->acc_tickets, sizeof(unsigned int) * h->E);
  if (h->w8) {
    add(&h->q.xq, 2 * rows * h->d);
    add(&h->q.xq_s, sizeof(float) * rows);
    add(&h->q.aq, 2 * rows * h->F);
    add(&h->q.aq_s, sizeof(float) * rows);
    if (h->S > 0) {
      add(&h->q.xqt, 2 * (size_t)h->Tmax * h->d);
      add(&h->q.xqt_s, sizeof(float) * h->Tmax);
      add(&h->q.saq, 2 * (size_t)h->S * h->Tmax * h->Fs);
      add(&h->q.saq_s, sizeof(float) * (size_t)h->S * h->Tmax);
    }
  }
  add(&h->xstage, 2 * h->elt * (size_t)h->Tmax * h->d);
  add(&h->ystage, h->elt * (size_t)h->Tmax * h->d);
  size_t total = 0;
  for (auto& p : parts) total = align_up(total, 256) + align_up(p.bytes, 256);
  cudaError_t e = cudaMalloc(&h->mem, total);
  if (e != cudaSuccess) {
    cudaGetLastError();  // a failed allocation leaves the context usable: clear its error
    free_handle(h);
    return fail(nullptr, EAT_ERR_OOM,
                "cudaMalloc of " + std::to_string(total) + " bytes failed: " +
                    cudaGetErrorString(e));
  }
  size_t off = 0;
  for (auto& p : parts) {
    off = align_up(off, 256);
    *p.p = (char*)h->mem + off;
    off += align_up(p.bytes, 256);
  }
  e = cudaMemset(h->mem, 0, total);
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  if (e != cudaSuccess) {
    free_handle(h);
    return fail(nullptr, EAT_ERR_CUDA, std::string("workspace init: ") + cudaGetErrorString(e));
  }
  if (h->backend == 1) {
    const char* msg = nullptr;
    if (tc_bind(h->tc, D, h->xperm, h->act, h->sact, h->q, &msg) != 0) {
      std::string m = msg ? msg : "tensor map setup failed";
      free_handle(h);
      return fail(nullptr, EAT_ERR_CUDA, m);
    }
  }
  e = cudaHostAlloc((void**)&h->mirror_host, 16, cudaHostAllocMapped);
  if (e == cudaSuccess) {
    std::memset(h->mirror_host, 0, 16);
    e = cudaHostGetDevicePointer((void**)&h->mirror_dev, h->mirror_host, 0);
  }
  if (e != cudaSuccess) {
    cudaGetLastError();
    free_handle(h);
    return fail(nullptr, EAT_ERR_OOM,
                std::string("mapped host status word: ") + cudaGetErrorString(e));
  }
  if (h->S > 0) {  // created here, not on first use, so that a call may be stream-captured
    e = cudaStreamCreateWithFlags(&h->side_st, cudaStreamNonBlocking);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&h->ev_fork, cudaEventDisableTiming);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&h->ev_join, cudaEventDisableTiming);
    if (e != cudaSuccess) {
      free_handle(h);
      return fail(nullptr, EAT_ERR_CUDA, std::string("side stream: ") + cudaGetErrorString(e));
    }
  }
  *out = h;
  return EAT_OK;
}

eat_status eat_reset_accounts(eat_handle* h, void* stream) {
  if (!h) return fail(nullptr, EAT_ERR_INVALID_ARG, "null handle");
  cudaStream_t st = (cudaStream_t)stream;
  cudaError_t e = cudaMemsetAsync(h->N, 0, sizeof(int64_t) * h->E, st);
  if (e == cudaSuccess) e = cudaMemsetAsync(h->P, 0, sizeof(double) * h->E, st);
  if (e == cudaSuccess) e = cudaMemsetAsync(h->C, 0, sizeof(double) * h->E, st);
  if (e == cudaSuccess) e = cudaMemsetAsync(h->counters, 0, sizeof(long long) * 4, st);
  if (e == cudaSuccess) e = cudaMemsetAsync(h->status, 0, sizeof(unsigned int) * 4, st);
  // every earlier call has written its copy of the status word before the copy is cleared
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) return cuda_fail(h, e, "reset accounts");
  *(volatile unsigned int*)h->mirror_host = 0u;
  h->failed = false;
  h->launches = 0;
  return EAT_OK;
}

eat_status eat_route(eat_handle* h, const void* x, int32_t T, int32_t ppl_sign, int32_t* idx,
                     float* w, int32_t* k, void* stream) {
  EAT_TRY(check_call(h, x, T, ppl_sign));
  if (!idx || !w || !k) return fail(h, EAT_ERR_INVALID_ARG, "idx, w and k must be non-NULL");
  return run_route(h, x, T, ppl_sign, idx, w, k, nullptr, false, (cudaStream_t)stream);
}

eat_status eat_moe_forward(eat_handle* h, const void* x, int32_t T, int32_t ppl_sign, void* y,
                           int32_t* idx_opt, float* w_opt, int32_t* k_opt, void* stream) {
  EAT_TRY(check_call(h, x, T, ppl_sign));
  if (!y) return fail(h, EAT_ERR_INVALID_ARG, "y is NULL");
  if (y == x) return fail(h, EAT_ERR_INVALID_ARG, "y must not alias x");
  if (((uintptr_t)y & 15) != 0) return fail(h, EAT_ERR_INVALID_ARG, "y must be 16-byte aligned");
  return run_forward(h, x, T, ppl_sign, y, idx_opt, w_opt, k_opt, (cudaStream_t)stream);
}

// The device address of a page-locked host buffer (cudaHostAlloc / cudaHostRegister), or null for
// any other memory.
static void* mapped_host(const void* p) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  return a.type == cudaMemoryTypeHost ? a.devicePointer : nullptr;
}

static eat_status forward_host(eat_handle* h, const void* x_host, int32_t T, int32_t ppl_sign,
                               void* y_host, void* stream, bool sync) {
  EAT_TRY(check_call(h, x_host, T, ppl_sign));
  if (!y_host) return fail(h, EAT_ERR_INVALID_ARG, "y_host is NULL");
  cudaStream_t st = (cudaStream_t)stream;
  const size_t bytes = h->elt * (size_t)T * h->d;
  cudaError_t e = cudaSuccess;
  if (!h->copy_st) {
    e = cudaStreamCreateWithFlags(&h->copy_st, cudaStreamNonBlocking);
    for (int i = 0; i < 2 && e == cudaSuccess; ++i) {
      e = cudaEventCreateWithFlags(&h->ev_copied[i], cudaEventDisableTiming);
      if (e == cudaSuccess) e = cudaEventCreateWithFlags(&h->ev_done[i], cudaEventDisableTiming);
    }
    if (e != cudaSuccess) return cuda_fail(h, e, "copy stream setup");
  }
  const int i = h->stage_i;
  h->stage_i ^= 1;
  void* xs = (char*)h->xstage + (size_t)i * h->elt * h->Tmax * h->d;
  // Page-locked buffers on the tensor-core path: the router kernel reads x over the host link
  // while it computes and leaves the device copy in the staging buffer, and the combine kernel
  // writes y over the link, so no copy engine transfer and no extra launch sits on the call's
  // path.  Not when shared experts run beside the routing (they read x before the router has
  // run).
  void* xd = h->backend == 1 ? mapped_host(x_host) : nullptr;
  void* yd = xd ? mapped_host(y_host) : nullptr;
  if (xd && yd && ((uintptr_t)xd & 15) == 0 && ((uintptr_t)yd & 15) == 0 &&
      router_copies_x(xd, h->bf16, h->desc.w_router, T, h->d) &&
      !shared_on_side_stream(h, T, tc_tile_rows(h->tc, T))) {
    // a call on another stream may still read this staging buffer
    e = cudaStreamWaitEvent(st, h->ev_done[i], 0);
    if (e != cudaSuccess) return cuda_fail(h, e, "staging buffer wait");
    EAT_TRY(run_forward(h, xs, T, ppl_sign, yd, nullptr, nullptr, nullptr, st, xd));
    e = cudaEventRecord(h->ev_done[i], st);
    if (e == cudaSuccess && sync) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return cuda_fail(h, e, "host-buffer call");
    if (sync) return check_state(h);
    return EAT_OK;
  }
  // the copy waits for the call that last read this buffer (an event never recorded counts as
  // complete), and this call's kernels wait for the copy
  e = cudaStreamWaitEvent(h->copy_st, h->ev_done[i], 0);
  if (e == cudaSuccess) e = cudaMemcpyAsync(xs, x_host, bytes, cudaMemcpyHostToDevice, h->copy_st);
  if (e == cudaSuccess) e = cudaEventRecord(h->ev_copied[i], h->copy_st);
  if (e == cudaSuccess) e = cudaStreamWaitEvent(st, h->ev_copied[i], 0);
  if (e != cudaSuccess) return cuda_fail(h, e, "x host-to-device copy");
  EAT_TRY(run_forward(h, xs, T, ppl_sign, h->ystage, nullptr, nullptr, nullptr, st));
  e = cudaEventRecord(h->ev_done[i], st);
  if (e == cudaSuccess) e = cudaMemcpyAsync(y_host, h->ystage, bytes, cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess && sync) e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) return cuda_fail(h, e, "y device-to-host copy");
  if (sync) return check_state(h);  // this call's own kernels, now complete
  return EAT_OK;
}

eat_status eat_moe_forward_host(eat_handle* h, const void* x_host, int32_t T, int32_t ppl_sign,
                                void* y_host, void* stream) {
  return forward_host(h, x_host, T, ppl_sign, y_host, stream, true);
}

eat_status eat_moe_forward_host_async(eat_handle* h, const void* x_host, int32_t T,
                                      int32_t ppl_sign, void* y_host, void* stream) {
  return forward_host(h, x_host, T, ppl_sign, y_host, stream, false);
}

eat_status eat_set_tau_state(eat_handle* h, float* tau_state) {
  if (!h) return fail(nullptr, EAT_ERR_INVALID_ARG, "null handle");
  if (((uintptr_t)tau_state & 3) != 0)
    return fail(h, EAT_ERR_INVALID_ARG, "tau_state must be 4-byte aligned");
  h->tau_state = tau_state;
  return EAT_OK;
}

eat_status eat_set_ppl_sign_source(eat_handle* h, const int32_t* sign) {
  if (!h) return fail(nullptr, EAT_ERR_INVALID_ARG, "null handle");
  if (((uintptr_t)sign & 3) != 0)
    return fail(h, EAT_ERR_INVALID_ARG, "sign must be 4-byte aligned");
  h->ppl_sign_src = sign;
  return EAT_OK;
}

eat_status eat_destroy(eat_handle* h) {
  if (!h) return EAT_OK;
  cudaDeviceSynchronize();
  free_handle(h);
  return EAT_OK;
}

eat_status eat_get_accounts(eat_handle* h, int64_t* N, double* P, double* C, void* stream) {
  if (!h) return fail(nullptr, EAT_ERR_INVALID_ARG, "null handle");
  if (!N || !P || !C) return fail(h, EAT_ERR_INVALID_ARG, "N, P and C must be non-NULL");
  cudaStream_t st = (cudaStream_t)stream;
  cudaError_t e = cudaMemcpyAsync(N, h->N, sizeof(int64_t) * h->E, cudaMemcpyDeviceToDevice, st);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(P, h->P, sizeof(double) * h->E, cudaMemcpyDeviceToDevice, st);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(C, h->C, sizeof(double) * h->E, cudaMemcpyDeviceToDevice, st);
  if (e != cudaSuccess) return cuda_fail(h, e, "get accounts");
  return EAT_OK;
}

eat_status eat_set_accounts(eat_handle* h, const int64_t* N, const double* P, const double* C,
                            void* stream) {
  if (!h) return fail(nullptr, EAT_ERR_INVALID_ARG, "null handle");
  if (!N || !P || !C) return fail(h, EAT_ERR_INVALID_ARG, "N, P and C must be non-NULL");
  cudaStream_t st = (cudaStream_t)stream;
  cudaError_t e = cudaMemcpyAsync(h->N, N, sizeof(int64_t) * h->E, cudaMemcpyDeviceToDevice, st);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(h->P, P, sizeof(double) * h->E, cudaMemcpyDeviceToDevice, st);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(h->C, C, sizeof(double) * h->E, cudaMemcpyDeviceToDevice, st);
  if (e != cudaSuccess) return cuda_fail(h, e, "set accounts");
  return EAT_OK;
}

eat_status eat_get_call_stats(eat_handle* h, int32_t* n_e, double* sum_p, double* sum_norm,
                              void* stream) {
  if (!h) return fail(nullptr, EAT_ERR_INVALID_ARG, "null handle");
  cudaStream_t st = (cudaStream_t)stream;
  cudaError_t e = cudaSuccess;
  if (n_e) e = cudaMemcpyAsync(n_e, h->st_n, sizeof(int32_t) * h->E, cudaMemcpyDeviceToDevice, st);
  if (sum_p && e == cudaSuccess)
    e = cudaMemcpyAsync(sum_p, h->st_p, sizeof(double) * h->E, cudaMemcpyDeviceToDevice, st);
  if (sum_norm && e == cudaSuccess)
    e = cudaMemcpyAsync(sum_norm, h->st_norm, sizeof(double) * h->E, cudaMemcpyDeviceToDevice,
                        st);
  if (e != cudaSuccess) return cuda_fail(h, e, "get call stats");
  return EAT_OK;
}

eat_status eat_get_counters(eat_handle* h, int64_t* out, int32_t n) {
  if (!h) return fail(nullptr, EAT_ERR_INVALID_ARG, "null handle");
  if (!out || n < 0) return fail(h, EAT_ERR_INVALID_ARG, "out is NULL or n < 0");
  long long dev[4] = {0, 0, 0, 0};
  unsigned int stw = 0;
  cudaError_t e = cudaDeviceSynchronize();
  if (e == cudaSuccess) e = cudaMemcpy(dev, h->counters, sizeof(dev), cudaMemcpyDeviceToHost);
  if (e == cudaSuccess) e = cudaMemcpy(&stw, h->status, sizeof(stw), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(h, e, "get counters");
  const long long vals[5] = {dev[0], dev[1], dev[2], h->launches, (long long)stw};
  for (int i = 0; i < n && i < 5; ++i) out[i] = vals[i];
  return EAT_OK;
}

eat_status eat_profile_begin(eat_handle* h, int32_t capacity) {
  if (!h) return fail(nullptr, EAT_ERR_INVALID_ARG, "null handle");
  if (capacity < 1) return fail(h, EAT_ERR_INVALID_ARG, "capacity < 1");
  while ((int)h->ev.size() < 2 * capacity) {
    cudaEvent_t e;
    const cudaError_t r = cudaEventCreate(&e);
    if (r != cudaSuccess) return cuda_fail(h, r, "event create");
    h->ev.push_back(e);
  }
  h->ev_kind.assign(capacity, 0);
  h->prof_cap = capacity;
  h->prof_n = 0;
  h->prof = true;
  return EAT_OK;
}

eat_status eat_profile_end(eat_handle* h, double* ms, int64_t* launches, int32_t n) {
  if (!h) return fail(nullptr, EAT_ERR_INVALID_ARG, "null handle");
  if (!h->prof) return fail(h, EAT_ERR_STATE, "profiling was not started");
  h->prof = false;
  std::vector<double> acc(kKinds, 0.0);
  std::vector<long long> cnt(kKinds, 0);
  if (h->prof_n > 0) {
    const cudaError_t r = cudaEventSynchronize(h->ev[2 * h->prof_n - 1]);
    if (r != cudaSuccess) return cuda_fail(h, r, "event synchronize");
  }
  for (int i = 0; i < h->prof_n; ++i) {
    float m = 0.f;
    cudaEventElapsedTime(&m, h->ev[2 * i], h->ev[2 * i + 1]);
    acc[h->ev_kind[i]] += m;
    cnt[h->ev_kind[i]] += 1;
  }
  for (int i = 0; i < n && i < kKinds; ++i) {
    if (ms) ms[i] = acc[i];
    if (launches) launches[i] = cnt[i];
  }
  h->prof_n = 0;
  return EAT_OK;
}

int32_t eat_ffn_backend(const eat_handle* h) { return h ? h->backend : -1; }

eat_status eat_selftest_bounded_wait(int64_t limit_ns, uint32_t* status_out) {
  if (!status_out || limit_ns < 1000 || limit_ns > 1000000000LL)
    return fail(nullptr, EAT_ERR_INVALID_ARG, "need status_out and 1 us <= limit_ns <= 1 s");
  unsigned int* dev = nullptr;
  cudaError_t e = cudaMalloc(&dev, sizeof(unsigned int));
  if (e == cudaSuccess) e = cudaMemset(dev, 0, sizeof(unsigned int));
  if (e == cudaSuccess) e = tc_selftest_bounded_wait((unsigned long long)limit_ns, dev, nullptr);
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  unsigned int v = 0;
  if (e == cudaSuccess) e = cudaMemcpy(&v, dev, sizeof(v), cudaMemcpyDeviceToHost);
  if (dev) cudaFree(dev);
  if (e != cudaSuccess) return fail(nullptr, EAT_ERR_CUDA, std::string("self-test: ") +
                                                              cudaGetErrorString(e));
  *status_out = v;
  return EAT_OK;
}

eat_status eat_selftest_expire_wait(eat_handle* h, int64_t limit_ns, void* stream) {
  if (!h) return fail(nullptr, EAT_ERR_INVALID_ARG, "null handle");
  if (limit_ns < 1000 || limit_ns > 1000000000LL)
    return fail(h, EAT_ERR_INVALID_ARG, "need 1 us <= limit_ns <= 1 s");
  ++h->launches;
  const cudaError_t e =
      tc_selftest_bounded_wait((unsigned long long)limit_ns, h->status, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(h, e, "self-test launch");
  return EAT_OK;
}

const char* eat_last_error(const eat_handle* h) {
  if (!h) return g_err.empty() ? "no error recorded" : g_err.c_str();
  return h->err.empty() ? "no error recorded" : h->err.c_str();
}

const char* eat_status_string(eat_status s) {
  switch (s) {
    case EAT_OK: return "EAT_OK";
    case EAT_ERR_INVALID_ARG: return "EAT_ERR_INVALID_ARG";
    case EAT_ERR_UNSUPPORTED: return "EAT_ERR_UNSUPPORTED";
    case EAT_ERR_OOM: return "EAT_ERR_OOM";
    case EAT_ERR_CUDA: return "EAT_ERR_CUDA";
    case EAT_ERR_STATE: return "EAT_ERR_STATE";
  }
  return "EAT_UNKNOWN_STATUS";
}

}  // extern "C"

namespace eat {
void set_thread_error(const char* msg) { g_err = msg ? msg : ""; }
}  // namespace eat

namespace eat {
bool pdl_enabled() {
  static const bool on = [] {
    const char* v = getenv("EAT_PDL");
    return !(v && v[0] == '0');
  }();
  return on;
}
}  // namespace eat
