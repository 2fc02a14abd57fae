/*
 * eat.h -- C ABI of the GB300 (sm_103a) EAT MoE-layer hot path.
 *
 * EAT ("Expert Account Tracker", arxiv 2609.33614) replaces fixed Top-K routing in a
 * Mixture-of-Experts layer by a history-aware importance score and an adaptive per-token
 * threshold that activates a variable number of experts (§3.2-§3.4).  This library runs one MoE
 * layer forward pass under that rule on one GPU:
 *   router GEMM + softmax (§3.1-§3.2) -> history score S_h (Eq. 1) -> importance I (Eq. 2)
 *   -> threshold tau (Eq. 3-5, PPL adjustment, boundedness, smoothing; §3.3)
 *   -> variable-k selection and renormalisation (Eq. 6-8) -> permute by expert
 *   -> SwiGLU expert FFNs over the activated experts -> weighted combine / unpermute
 *   -> account update (N, P_total, C_s of §3.2).
 *
 * Conventions shared by every entry point:
 *  - Array pointers are DEVICE pointers unless the name ends in _host.  Row-major, no padding.
 *  - Weights are NOT owned: the caller keeps them alive and unchanged until eat_destroy.
 *  - The handle owns the expert accounts and a workspace sized for desc.max_tokens at
 *    eat_create; no entry point allocates afterwards.  One handle = one layer.
 *  - `stream` is a cudaStream_t passed as void* (NULL = legacy default stream).  Calls are
 *    asynchronous on that stream unless stated; arguments are validated on the host before any
 *    launch, and an invalid call returns an error without touching the device.
 *  - A handle is not thread-safe: calls on one handle must be serialised by the caller, and
 *    calls that may overlap on the GPU (different streams) must not share a handle.
 *  - Nothing throws across the ABI.  Every call returns an eat_status; eat_last_error gives a
 *    one-line description of the last failure on that handle.
 */
#ifndef EAT_H_
#define EAT_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum eat_status {
  EAT_OK = 0,
  EAT_ERR_INVALID_ARG = 1,  /* null pointer, size out of range, bad enum value */
  EAT_ERR_UNSUPPORTED = 2,  /* valid request outside what this build implements */
  EAT_ERR_OOM = 3,          /* device allocation failed in eat_create */
  EAT_ERR_CUDA = 4,         /* a CUDA runtime call or kernel launch failed */
  EAT_ERR_STATE = 5         /* handle not usable: a kernel of an earlier call gave up on a bounded
                               wait (device status word set); cleared by eat_reset_accounts */
} eat_status;

/* EAT_FP8_E4M3 is an expert-weight type only (wdtype, with xdtype EAT_BF16): OCP e4m3 bytes with
 * one fp32 scale per weight row (see eat_layer_desc).  Not from the paper: a storage format that
 * halves the weight bytes a decode call streams. */
typedef enum eat_dtype { EAT_F32 = 0, EAT_BF16 = 1, EAT_FP8_E4M3 = 2 } eat_dtype;

/* Expert selection rule.  EAT_ROUTER_EAT: the adaptive threshold of §3.3-§3.4 (Eq. 3-8).  The
 * baselines the paper compares with (§4.1), computed by the same kernels from the same
 * probabilities: EAT_ROUTER_TOPK, the K largest p (index ascending on ties); EAT_ROUTER_TOPP, the
 * smallest descending-p prefix whose cumulative probability reaches top_p, at most K experts.
 * Gates are always Eq. 7; the accounts are updated in every mode. */
typedef enum eat_router_mode {
  EAT_ROUTER_EAT = 0,
  EAT_ROUTER_TOPK = 1,
  EAT_ROUTER_TOPP = 2
} eat_router_mode;

/* Threshold smoothing of §3.3.  EAT_SMOOTH_CALL: the same-call blend kappa1 tau_PPL + kappa2 tau.
 * EAT_SMOOTH_TEMPORAL: an EMA over calls of one token stream, kappa1 tau_PPL + kappa2 tau_prev,
 * where tau_prev is that stream's tau_final of the previous call (see eat_set_tau_state). */
typedef enum eat_smoothing { EAT_SMOOTH_CALL = 0, EAT_SMOOTH_TEMPORAL = 1 } eat_smoothing;

/* How the EMA contribution C_s enters Eq. 1 (§3.2).  EAT_C_SUM: as the share C_i / sum_j C_j,
 * on the same [0, 1] scale as the other two terms (default).  EAT_C_RAW: the literal C_i. */
typedef enum eat_c_mode { EAT_C_SUM = 0, EAT_C_RAW = 1 } eat_c_mode;

/* Hyper-parameters of §3.2-§3.4; defaults (eat_default_params) are Table 1, the 1.2 / 0.9 factors
 * and 10% / 90% bounds of §3.3, and eps of Eq. 7. */
typedef struct eat_params {
  double alpha;        /* EMA factor of C_s (0.95): C <- (1 - alpha) C + alpha ||o||_2 */
  double w1, w2, w3;   /* Eq. 1 weights (0.3, 0.3, 0.4) */
  double beta;         /* Eq. 2 balance (0.6): I = (1 - beta) p + beta S_h */
  double alpha1;       /* Eq. 5 (0.5): tau = max(alpha1 mu, mu - alpha2 sigma) */
  double alpha2;       /* Eq. 5 (1.0) */
  double kappa1;       /* smoothing (0.7): tau_final = kappa1 tau_PPL + kappa2 tau */
  double kappa2;       /* smoothing (0.3) */
  double ppl_up;       /* factor when PPL rose (1.2) */
  double ppl_down;     /* factor otherwise (0.9) */
  double q_lo, q_hi;   /* boundedness: tau_final clamped to these quantiles of p (0.1, 0.9) */
  double eps;          /* Eq. 7 (1e-8) */
  double temperature;  /* router logits are divided by it before the softmax (1.0) */
  int32_t max_k;       /* K of Eq. 6: at most K experts per token, 1 <= K <= min(E, 16) */
  int32_t clamp_enabled; /* 1: apply the [q_lo, q_hi] bounds; 0: skip them */
  int32_t c_mode;      /* eat_c_mode */
  int32_t router_mode; /* eat_router_mode (EAT_ROUTER_EAT) */
  double top_p;        /* P of EAT_ROUTER_TOPP, in (0, 1] (0.6) */
  int32_t smoothing_mode; /* eat_smoothing (EAT_SMOOTH_CALL) */
} eat_params;

/* Fill *p with the defaults above, max_k = 2, router_mode EAT_ROUTER_EAT, top_p 0.6.  Returns
 * EAT_ERR_INVALID_ARG if p is NULL. */
eat_status eat_default_params(eat_params* p);

/* One MoE layer.  Shapes use nn.Linear layout (out_features x in_features), row-major:
 *   w_router [E, d] fp32, b_router [E] fp32 or NULL;
 *   w_gate, w_up [E, F, d], w_down [E, d, F] in wdtype;
 *   ws_gate, ws_up [S, Fs, d], ws_down [S, d, Fs] in wdtype, all NULL when n_shared == 0
 *   (always-on shared experts, added with weight 1, not routed, no account);
 *   opd_scale [E] fp32 or NULL: OPD inference reweighting (§3.5) -- the routing probabilities
 *   become p'_i = s_i p_i / sum_j s_j p_j before selection, and p' is used everywhere p is;
 *   w_gate_scale, w_up_scale [E, F], w_down_scale [E, d], ws_gate_scale, ws_up_scale [S, Fs],
 *   ws_down_scale [S, d] fp32: with wdtype EAT_FP8_E4M3, weight row r of each matrix is
 *   scale[r] * (its e4m3 bytes) (the shared ones NULL when n_shared == 0); ignored otherwise.
 * Supported: 1 <= E <= 256; d, F, Fs multiples of 64; (wdtype, xdtype) both EAT_F32, both
 * EAT_BF16, or EAT_FP8_E4M3 weights with EAT_BF16 hidden states; 1 <= max_tokens <= 65536.  All
 * weight pointers 16-byte aligned.  fp8 layers feed the e4m3 weights to the tensor cores
 * unconverted (e4m3 x e4m3 -> fp32 MMAs): each row of a GEMM's other operand (the hidden states,
 * then the bf16 SwiGLU activations) is scaled by a power of two and split into two e4m3 parts,
 * hi + lo, which hold a bf16 value exactly down to 2^-9 of its row's largest magnitude; both
 * parts are multiplied and accumulated in fp32.  fp8 layers always use the single-SM kernels. */
typedef struct eat_layer_desc {
  int32_t d_model, n_experts, d_ff, n_shared, d_ff_shared, max_tokens;
  int32_t wdtype, xdtype;
  const float* w_router;
  const float* b_router;
  const void* w_gate;
  const void* w_up;
  const void* w_down;
  const void* ws_gate;
  const void* ws_up;
  const void* ws_down;
  const float* opd_scale;
  const float* w_gate_scale;
  const float* w_up_scale;
  const float* w_down_scale;
  const float* ws_gate_scale;
  const float* ws_up_scale;
  const float* ws_down_scale;
} eat_layer_desc;

typedef struct eat_handle eat_handle;

/* Validate desc/params, allocate the accounts (zeroed: the empty history of §3.2) and the
 * workspace for max_tokens, and build the weight descriptors.  Synchronous.  On success *out
 * receives the handle; on failure *out is set to NULL and nothing stays allocated. */
eat_status eat_create(const eat_layer_desc* desc, const eat_params* params, eat_handle** out);

/* Zero the accounts N, P_total, C_s (§3.2: an expert with no history), the counters and the
 * device status word, and return the handle to service after EAT_ERR_STATE.  Synchronises
 * `stream` (every earlier call on it has finished when it returns). */
eat_status eat_reset_accounts(eat_handle* h, void* stream);

/* Routing only (§3.2-§3.4, Eq. 1-8) for T tokens x [T, d] (xdtype), 1 <= T <= max_tokens,
 * reading the current accounts and never changing them.  ppl_sign is the sign of
 * PPL_curr - PPL_prev (§3.3): +1 -> factor ppl_up, -1 -> ppl_down, 0 -> no signal (factor 1).
 * x must be 16-byte aligned.
 * Outputs: idx [T, K] int32 selected experts in ascending index order, -1 after the k-th;
 * w [T, K] fp32 renormalised gates g_norm (Eq. 7), 0 after the k-th; k [T] int32 count. */
eat_status eat_route(eat_handle* h, const void* x, int32_t T, int32_t ppl_sign,
                     int32_t* idx, float* w, int32_t* k, void* stream);

/* Failure state (every entry point that runs the layer or routes): the expert kernels never trap;
 * a wait that expires after its 2 s bound sets a bit in the handle's device status word and the
 * kernel returns early.  The combine kernel of that call then writes NaN rows to y and the account
 * update leaves N, P_total and C_s unchanged; the call's last kernel copies the word to host-mapped
 * memory.  The next eat_route / eat_moe_forward / eat_moe_forward_host(_async) on the handle that
 * finds the copy set returns EAT_ERR_STATE, and so does every later one until
 * eat_reset_accounts; eat_moe_forward_host, which synchronises, returns EAT_ERR_STATE for the
 * failing call itself. */

/* One layer call = one EMA timestep of §3.2 over T tokens, 1 <= T <= max_tokens (an empty call has
 * no batch mean to fold into the accounts and is rejected with EAT_ERR_INVALID_ARG): routing as
 * eat_route from the pre-call accounts,
 * y [T, d] (xdtype) = sum over selected e of g_norm,e * E_e(x_t) + sum of shared experts, then
 * the account update: N_e += n_e, P_total,e += sum of p over e's activations,
 * C_e <- (1 - alpha) C_e + alpha * mean ||E_e(x_t)||_2 when n_e > 0.
 * idx_opt / w_opt / k_opt may be NULL; when given they receive the routing as in eat_route.
 * y must not alias x; x and y must be 16-byte aligned.  A layer with shared experts may run them,
 * for a small call, on a stream of the handle that forks from `stream` at the start of the call
 * and joins it again before the outputs are combined (events recorded on `stream`), so the call
 * stays ordered on `stream` and can be stream-captured into a CUDA graph. */
eat_status eat_moe_forward(eat_handle* h, const void* x, int32_t T, int32_t ppl_sign, void* y,
                           int32_t* idx_opt, float* w_opt, int32_t* k_opt, void* stream);

/* eat_moe_forward with HOST buffers x_host [T, d] and y_host [T, d]: moves x to the device, runs
 * the layer, moves y back and synchronises the stream before returning.
 *  - Page-locked buffers (cudaHostAlloc / cudaHostRegister, 16-byte aligned) of a bf16 or fp8
 *    layer: the router kernel reads x_host over the host link while it computes and writes the
 *    device copy that the later kernels read, and the combine kernel writes y_host directly; no
 *    copy-engine transfer.  (Except for a call whose shared experts run beside the routing: those
 *    read x before the router has run, so such a call takes the copies below.)
 *  - Otherwise the input is copied on a stream of the handle (created on the first host-buffer
 *    call), and y is copied back on `stream`; pageable memory works but is staged by the driver.
 * Either way x lands in one of two staging buffers of the handle used in turn, so a call's input
 * never overwrites the input of the call before it while that call may still read it. */
eat_status eat_moe_forward_host(eat_handle* h, const void* x_host, int32_t T, int32_t ppl_sign,
                                void* y_host, void* stream);

/* eat_moe_forward_host without the final synchronisation: enqueues the layer and the movement of
 * x_host and y_host (as eat_moe_forward_host) on `stream`, and returns.  The caller
 * keeps both host buffers alive, and x_host unchanged, until the stream has passed this call
 * (cudaStreamSynchronize or an event) and reads y_host only after that.  With page-locked host
 * buffers (cudaHostAlloc / cudaHostRegister) the copies are asynchronous and consecutive calls
 * queue back to back on the GPU; with pageable buffers the runtime may block.  Calls on one handle
 * share its staging buffers, which stream order makes safe. */
eat_status eat_moe_forward_host_async(eat_handle* h, const void* x_host, int32_t T,
                                      int32_t ppl_sign, void* y_host, void* stream);

/* Size of the fixed device scratch eat_route_noalloc uses: 1 MiB = 131072 partial router scores,
 * each a compensated fp32 pair (hi, lo) of 8 bytes. */
#define EAT_NOALLOC_SCRATCH_BYTES (1u << 20)

/* Routing for callers that cannot allocate device memory.  The paper has no counterpart: this is a
 * deployment variant of eat_route.  Some callers cannot call cudaMalloc -- a serving process that
 * reserved nearly all HBM for its own pool, a decode loop that must not take cudaMalloc's implicit
 * device synchronisation, a framework that forbids allocations outside its own allocator -- and so
 * cannot create a handle.  This call computes exactly what eat_route computes (Eq. 1-8) from
 * caller-owned device buffers: x [T, d_model] (xdtype), w_router [E, d_model] fp32, b_router [E]
 * fp32 or NULL, accounts N [E] int64, P [E] fp64, C [E] fp64 (read only), and writes idx / w / k
 * as eat_route does.  It allocates nothing: its only scratch is a fixed 1 MiB array compiled into
 * the library, which every GPU that loads the library holds until the process exits.
 *  - T * n_experts must be <= 131072 (EAT_NOALLOC_SCRATCH_BYTES / 8), else EAT_ERR_INVALID_ARG;
 *    larger batches are routed in several calls.
 *  - The first call on each device looks up the scratch's device address (a one-time set-up per
 *    device, done with that device current), and so does the first call after the device's
 *    current context changed (e.g. after cudaDeviceReset); make that first call before any
 *    stream capture.
 *  - Calls share the scratch: two calls that may overlap on the GPU (different streams or host
 *    threads) race on it and must be serialised by the caller.
 *  - There is no per-stream threshold state without a handle: EAT_SMOOTH_TEMPORAL is routed as
 *    EAT_SMOOTH_CALL.
 * Errors are reported through eat_last_error(NULL). */
eat_status eat_route_noalloc(const void* x, int32_t T, int32_t d_model, int32_t n_experts,
                             int32_t xdtype, const float* w_router, const float* b_router,
                             const int64_t* N, const double* P, const double* C,
                             const eat_params* params, int32_t ppl_sign, int32_t* idx, float* w,
                             int32_t* k, void* stream);

/* Per-stream threshold state for EAT_SMOOTH_TEMPORAL: tau_state is a caller-owned device array
 * of max_tokens fp32 values; row t of every call is token stream t (e.g. sequence t of a decode
 * batch).  eat_route reads it; eat_moe_forward reads it and stores each token's tau_final back.
 * NaN entries mean "no previous call" (the same-call blend is used).  NULL detaches the state
 * (temporal mode then behaves as EAT_SMOOTH_CALL).  The array must stay alive while attached. */
eat_status eat_set_tau_state(eat_handle* h, float* tau_state);

/* The perplexity signal of §3.3's performance-based adjustment, for a model loop on the device.
 * nll: device [n] fp32 negative log-likelihoods of the n >= 1 tokens of the current window (e.g.
 * the tokens generated since the last call); ppl_state: a caller-owned device fp64 scalar holding
 * the previous window's perplexity (set it to NaN before the first window: no previous value);
 * sign: device int32 output.  One kernel on `stream` computes PPL_curr = exp(mean nll) (fp64 sum
 * in a fixed order), writes *sign = +1 when PPL_curr - PPL_prev > 0 (a drop in performance), -1
 * otherwise, 0 when there is no previous value or PPL_curr is NaN, and stores PPL_curr into
 * *ppl_state.  Errors through eat_last_error(NULL). */
eat_status eat_ppl_update(const float* nll, int32_t n, double* ppl_state, int32_t* sign,
                          void* stream);

/* Attach a device PPL sign (the `sign` of eat_ppl_update, caller-owned, alive while attached) to
 * the handle: eat_route / eat_moe_forward then read the sign from device memory when their
 * selection kernel runs, stream-ordered after the eat_ppl_update that wrote it, and ignore their
 * ppl_sign argument (which is still validated).  NULL detaches it. */
eat_status eat_set_ppl_sign_source(eat_handle* h, const int32_t* sign);

/* Layer-wise routing policy after §5.2 (experts in lower layers matter less than in higher ones:
 * the paper keeps 1.3-1.5 experts per token in layers 0-23 of a 32-layer stack and the full K
 * above).  Adjusts *p for layer `layer` of an n_layers stack: in the lower three quarters, max_k
 * becomes max(1, max_k / 3) and alpha1 (the threshold floor of Eq. 5) doubles; the upper quarter
 * keeps *p.  Call it on each layer's params before eat_create.  EAT_ERR_INVALID_ARG unless
 * 0 <= layer < n_layers and p is non-NULL. */
eat_status eat_layer_policy(int32_t layer, int32_t n_layers, eat_params* p);

/* Free everything the handle owns.  Synchronises the device first.  NULL is accepted. */
eat_status eat_destroy(eat_handle* h);

/* Snapshot / restore of the accounts (device pointers, [E] each): N int64, P_total fp64,
 * C_s fp64.  Stream-ordered copies. */
eat_status eat_get_accounts(eat_handle* h, int64_t* N, double* P, double* C, void* stream);
eat_status eat_set_accounts(eat_handle* h, const int64_t* N, const double* P, const double* C,
                            void* stream);

/* Per-expert statistics of the last eat_moe_forward (device pointers, [E] each): activation
 * count n_e, sum of p over the activations, sum of ||E_e(x_t)||_2 over the activations.  Any
 * pointer may be NULL.  Stream-ordered copies. */
eat_status eat_get_call_stats(eat_handle* h, int32_t* n_e, double* sum_p, double* sum_norm,
                              void* stream);

/* Counters since eat_create or the last eat_reset_accounts, into host array out[n]
 * (synchronises the device):
 *   out[0] forward calls, out[1] sum over calls of the number of distinct activated experts,
 *   out[2] sum over calls of the activations (sum_t k_t), out[3] kernel launches issued by this
 *   handle (all entry points), out[4] the device status word: 0, or the bits of kernel waits that
 *   expired (a kernel that gives up on a wait returns early and its outputs are invalid):
 *   1 the TMA producer waiting for a free pipeline stage, 2 copies still in flight at exit,
 *   4 the MMA issuer waiting for a free accumulator, 8 the MMA issuer waiting for a stage's data,
 *   16 MMAs still running before TMEM is freed, 32 the epilogue waiting for an accumulator,
 *   64 eat_selftest_bounded_wait / eat_selftest_expire_wait, 128 the gate/up epilogue's exchange
 *   between warps. */
eat_status eat_get_counters(eat_handle* h, int64_t* out, int32_t n);

/* Per-kernel device timing.  eat_profile_begin(h, capacity) makes every later launch of this
 * handle record a CUDA event pair (capacity = max launches recorded); eat_profile_end
 * synchronises, writes for each kernel kind i < n the summed milliseconds ms[i] and the launch
 * count launches[i], and stops recording.  Kernel kinds: 0 router scores, 1 permute, 2 routed
 * gate/up FFN, 3 routed down FFN, 4 shared gate/up, 5 shared down, 6 combine, 7 account,
 * 8 selection (softmax / threshold / Eq. 6-8), 9 token-row gather. */
eat_status eat_profile_begin(eat_handle* h, int32_t capacity);
eat_status eat_profile_end(eat_handle* h, double* ms, int64_t* launches, int32_t n);

/* Which expert-FFN kernels this handle uses: 0 = CUDA-core (fp32 layers), 1 = tcgen05/TMA
 * tensor-core kernels (bf16 layers).  -1 on a NULL handle. */
int32_t eat_ffn_backend(const eat_handle* h);

/* Diagnostic of the failure path: runs one kernel thread that waits, with the bounded wait the
 * tensor-core kernels use, on a barrier nothing arrives on.  After limit_ns (1 us .. 1 s) the wait
 * gives up, sets bit 64 in a device status word and the kernel returns; *status_out receives the
 * word (64 when the bound works) and the context stays usable.  Synchronous; allocates 4 bytes. */
eat_status eat_selftest_bounded_wait(int64_t limit_ns, uint32_t* status_out);

/* Diagnostic of the failure state: enqueues on `stream` the same bounded wait on a barrier nothing
 * arrives on, writing the handle's device status word.  After limit_ns (1 us .. 1 s) it gives up
 * and sets bit 64, exactly as an expert kernel whose wait expired would set its bit: the next
 * layer call on `stream` writes NaN outputs, leaves the accounts unchanged, and later calls return
 * EAT_ERR_STATE until eat_reset_accounts.  No fault, trap or hang is involved. */
eat_status eat_selftest_expire_wait(eat_handle* h, int64_t limit_ns, void* stream);

/* Last error on the handle (never NULL), or a generic text for a NULL handle. */
const char* eat_last_error(const eat_handle* h);
const char* eat_status_string(eat_status s);

#ifdef __cplusplus
}
#endif
#endif /* EAT_H_ */
