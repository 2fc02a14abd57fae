// Tensor-core (tcgen05 + TMEM + TMA) expert FFN kernels for bf16 layers: interface used by the
// host runtime.
#pragma once

#include "eat_internal.cuh"

namespace eat {

struct TcLayer {
  bool ready = false;
  int E = 0, d = 0, F = 0, S = 0, Fs = 0, K = 0, Tmax = 0;
  void* maps = nullptr;  // host copy of the tensor maps (see ffn_tc.cu)
};

struct TcCall {
  const void* x = nullptr;
  int T = 0;
  int tile_rows = 0;
  const int32_t* offs = nullptr;
  const int32_t* tile_offs = nullptr;
  const int32_t* perm_tok = nullptr;
  void* act = nullptr;
  float* opart = nullptr;
  void* sact = nullptr;
  float* sout = nullptr;
  int max_split = 1;
};

// 0 on success; *msg explains a failure.
int tc_init(TcLayer& L, const eat_layer_desc& D, int K, int Tmax, const char** msg);
void tc_destroy(TcLayer& L);
int tc_tile_rows(const TcLayer& L, int T);   // token rows per tile for a call of T tokens
int tc_down_split(const TcLayer& L, int T);  // split-K slices of the routed down projection
int tc_max_split(const TcLayer& L);
cudaError_t tc_launch_up(const TcLayer& L, const TcCall& c, bool shared, cudaStream_t st);
cudaError_t tc_launch_down(const TcLayer& L, const TcCall& c, bool shared, int n_split,
                           cudaStream_t st);

}  // namespace eat
