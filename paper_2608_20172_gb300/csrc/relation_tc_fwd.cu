// relation_tc_fwd.cu -- placeholder until the tcgen05 forward lands.
#include "kernels.h"

namespace rel {
namespace tc {
bool supports(relation_dtype, int) { return false; }
cudaError_t launch_fwd(const Problem&, cudaStream_t) { return cudaErrorNotSupported; }
cudaError_t launch_bwd(const Problem&, const BwdWorkspace&, cudaStream_t) {
  return cudaErrorNotSupported;
}
int bwd_launches() { return 2; }
}  // namespace tc
}  // namespace rel
