// Placeholder until the tcgen05 kernels land: every entry reports "unsupported".
#include "ffn_tc.cuh"

namespace eat {

int tc_init(TcLayer& L, const eat_layer_desc&, int, int, const char** msg) {
  L.ready = false;
  if (msg) *msg = "tensor-core FFN kernels not built";
  return 1;
}
void tc_destroy(TcLayer&) {}
int tc_tile_rows(const TcLayer&, int) { return kSimtTileRows; }
int tc_down_split(const TcLayer&, int) { return 1; }
int tc_max_split(const TcLayer&) { return 1; }
cudaError_t tc_launch_up(const TcLayer&, const TcCall&, bool, cudaStream_t) {
  return cudaErrorNotSupported;
}
cudaError_t tc_launch_down(const TcLayer&, const TcCall&, bool, int, cudaStream_t) {
  return cudaErrorNotSupported;
}

}  // namespace eat
