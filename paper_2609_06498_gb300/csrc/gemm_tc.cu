// tcgen05 GEMM (placeholder until the tensor-core kernel lands).
#include "gemm_tc.cuh"

namespace dflow {

void tc_layout(TcWorkspace &w, char *base, size_t &off, int sm_count, size_t rows_max) {
  (void)base; (void)off; (void)rows_max;
  w.sm_count = sm_count;
}
bool tc_supports(int, int, int, int, const EpArgs &) { return false; }
cudaError_t tc_init(const TcWorkspace &, cudaStream_t) { return cudaSuccess; }
cudaError_t gemm_tc(const TcWorkspace &, const void *, int, int, const void *, int, int, const EpArgs &,
                    int *, cudaStream_t) {
  return cudaErrorNotSupported;
}

}  // namespace dflow
