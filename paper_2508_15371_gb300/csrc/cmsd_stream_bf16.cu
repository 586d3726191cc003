// bfloat16 instantiations of the streaming and resample kernels.
#include "cmsd_stream_impl.cuh"

namespace cmsd {

cudaError_t launch_stream_bf16(int mode, bool sampled, bool second, const StreamArgs& a, int grid,
                               size_t smem, cudaStream_t s) {
  return launch_stream_t<uint16_t>(mode, sampled, second, a, grid, smem, s);
}

cudaError_t occupancy_stream_bf16(int mode, bool sampled, bool second, size_t smem, int* nb) {
  return occupancy_stream_t<uint16_t>(mode, sampled, second, smem, nb);
}

cudaError_t launch_resample_bf16(bool sampled, const StreamArgs& a, int grid, cudaStream_t s) {
  return launch_resample_t<uint16_t>(sampled, a, grid, s);
}

cudaError_t launch_resample_bound_bf16(const StreamArgs& a, int clusters, cudaStream_t s) {
  return launch_resample_bound_t<uint16_t>(a, clusters, s);
}

bool resample_bound_fits_bf16(int V) { return resample_bound_fits_t<uint16_t>(V); }

cudaError_t occupancy_resample_bf16(bool sampled, int* nb) { return occupancy_resample_t<uint16_t>(sampled, nb); }

}  // namespace cmsd
