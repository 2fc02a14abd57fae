// Tensor-core (tcgen05 + TMEM + TMA) expert FFN kernels for bf16 and e4m3-weight layers:
// interface used by the host runtime.
#pragma once

#include "eat_internal.cuh"

namespace eat {

// fp8 layers: the workspace's e4m3 hi/lo planes of the GEMMs' B operands ([2][R][cols], the lo
// plane R rows after the hi plane) and their per-row power-of-two scales [R].
struct TcWork {
  uint8_t* xq = nullptr;   // x in slot order, R = Tmax * K, cols = d
  float* xq_s = nullptr;
  uint8_t* xqt = nullptr;  // x in token order (shared experts), R = Tmax, cols = d
  float* xqt_s = nullptr;
  uint8_t* aq = nullptr;   // routed activations, R = Tmax * K, cols = F
  float* aq_s = nullptr;
  uint8_t* saq = nullptr;  // shared activations, R = S * Tmax, cols = Fs
  float* saq_s = nullptr;
};

struct TcLayer {
  bool ready = false;
  int E = 0, d = 0, F = 0, S = 0, Fs = 0, K = 0, Tmax = 0;
  int num_sms = 0;
  bool w8 = false;  // e4m3 expert weights with per-row fp32 scales (kind::f8f6f4 MMAs)
  const float *sg = nullptr, *su = nullptr, *sd = nullptr;     // [E,F], [E,F], [E,d]
  const float *ssg = nullptr, *ssu = nullptr, *ssd = nullptr;  // shared experts
  TcWork q;
  void* maps = nullptr;  // host copy of the tensor maps (see ffn_tc.cu)
};

// The B operands an fp8 layer splits into e4m3 hi/lo planes before its GEMMs.
enum class TcSplit { kSlotX, kTokenX, kAct, kSharedAct };

struct TcCall {
  const void* x = nullptr;         // [T, d] bf16 hidden states of the call
  int T = 0;
  int tile_rows = 0;               // BN of the gate/up kernel (token rows per tile)
  int tile_rows_down = 0;          // BN of the down kernel
  const int32_t* offs = nullptr;   // [E+1] slot offsets
  const int32_t* tile_offs = nullptr;       // tile prefix for tile_rows
  const int32_t* tile_offs_down = nullptr;  // tile prefix for tile_rows_down
  const int32_t* perm_tok = nullptr;
  void* xperm = nullptr;           // [Tmax*K, d] gathered rows in slot order
  void* act = nullptr;             // [Tmax*K, F] bf16
  float* opart = nullptr;          // [split][T*K, d] fp32, or [T*K, d] bf16 without split-K
  void* sact = nullptr;            // [S*T, Fs] bf16
  void* sout = nullptr;            // [S*T, d] bf16
  unsigned int* status = nullptr;  // device status word (bounded-wait failures)
  bool fold_shared = false;        // the routed launches also run the shared experts (SM pairs)
};

// Device checks and the tensor-map encoder; 0 on success, *msg explains a failure.
int tc_configure(TcLayer& L, const eat_layer_desc& D, int K, int Tmax, const char** msg);
// Tensor maps over the weights and the handle's workspace buffers.
int tc_bind(TcLayer& L, const eat_layer_desc& D, void* xperm, void* act, void* sact,
            const TcWork& q, const char** msg);
void tc_destroy(TcLayer& L);
int tc_tile_rows(const TcLayer& L, int T);       // gate/up token rows per tile, call of T tokens
int tc_tile_rows_down(const TcLayer& L, int T);  // down-projection token rows per tile
bool tc_gathers_in_kernel(const TcLayer& L, int T);  // gate/up gathers x rows itself (no Xperm)
// A call of T tokens runs its shared experts inside the routed SM-pair launches (TcCall's
// fold_shared): one unit set after the other, one ramp and one tail per projection.
bool tc_folds_shared(const TcLayer& L, int T);
int tc_down_split(const TcLayer& L, int T);  // split-K slices of the routed down projection
long long tc_opart_rows(const TcLayer& L);   // rows of fp32 partials the workspace must hold
cudaError_t tc_launch_gather(const TcLayer& L, const TcCall& c, cudaStream_t st);
// fp8 layers: one B operand of the call as e4m3 hi/lo planes with per-row scales.
cudaError_t tc_launch_split(const TcLayer& L, const TcCall& c, TcSplit which, cudaStream_t st);
cudaError_t tc_launch_up(const TcLayer& L, const TcCall& c, bool shared, cudaStream_t st);
// Launches one thread waiting on an mbarrier nobody arrives on, bounded by limit_ns (the wait the
// tensor-core kernels use); the expiry sets bit 64 in *dev_status.
cudaError_t tc_selftest_bounded_wait(unsigned long long limit_ns, unsigned int* dev_status,
                                     cudaStream_t st);
cudaError_t tc_launch_down(const TcLayer& L, const TcCall& c, bool shared, int n_split,
                           cudaStream_t st);

}  // namespace eat
