// Tensor-core (tcgen05) kernel: placeholder until the kernel lands.
#include "kvx_internal.h"

namespace kvx {
bool tc_supported(const kvx_ctx*, std::string* why) {
  if (why) *why = "tensor-core kernel not built";
  return false;
}
kvx_status tc_prepare(kvx_ctx*, const void*) { return KVX_ERR_UNSUPPORTED; }
kvx_status launch_tc(const kvx_ctx*, const MapArgs&, cudaStream_t) {
  set_error("tensor-core kernel not built");
  return KVX_ERR_UNSUPPORTED;
}
}  // namespace kvx
