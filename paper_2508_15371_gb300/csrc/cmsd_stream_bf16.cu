// bfloat16 instantiations of the streaming and resample kernels.
#include "cmsd_stream_impl.cuh"

namespace cmsd {

cudaError_t launch_stream_bf16(int mode, bool sampled, const StreamArgs& a, int grid, size_t smem,
                               cudaStream_t s) {
  return launch_stream_t<uint16_t>(mode, sampled, a, grid, smem, s);
}
cudaError_t launch_resample_bf16(const StreamArgs& a, int grid, cudaStream_t s) {
  return launch_resample_t<uint16_t>(a, grid, s);
}

}  // namespace cmsd
