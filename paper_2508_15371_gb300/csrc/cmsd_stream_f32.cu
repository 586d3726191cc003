// float32 instantiations of the streaming and resample kernels, the
// occupancy queries, and the device Philox fill used by the tests.
#include "cmsd_stream_impl.cuh"

namespace cmsd {

cudaError_t occupancy_stream_bf16(int mode, bool sampled, bool second, size_t smem, int* nb);
cudaError_t occupancy_resample_bf16(bool sampled, int* nb);

cudaError_t launch_resample_f32(bool sampled, const StreamArgs& a, int grid, cudaStream_t s) {
  return launch_resample_t<float>(sampled, a, grid, s);
}

cudaError_t launch_resample_bound_f32(const StreamArgs& a, int clusters, cudaStream_t s) {
  return launch_resample_bound_t<float>(a, clusters, s);
}

bool resample_bound_fits_bf16(int V);
bool resample_bound_fits(int dtype, int V) {
  return dtype == 0 ? resample_bound_fits_t<float>(V) : resample_bound_fits_bf16(V);
}

cudaError_t occupancy_resample(int dtype, bool sampled, int* nb) {
  return dtype == 0 ? occupancy_resample_t<float>(sampled, nb) : occupancy_resample_bf16(sampled, nb);
}

cudaError_t launch_stream_f32(int mode, bool sampled, bool second, const StreamArgs& a, int grid,
                              size_t smem, cudaStream_t s) {
  return launch_stream_t<float>(mode, sampled, second, a, grid, smem, s);
}

cudaError_t occupancy_stream(int dtype, int mode, bool sampled, bool second, size_t smem, int* nb) {
  return dtype == 0 ? occupancy_stream_t<float>(mode, sampled, second, smem, nb)
                    : occupancy_stream_bf16(mode, sampled, second, smem, nb);
}

__global__ void philox_fill_kernel(uint32_t k0, uint32_t k1, uint32_t c0, uint32_t c1, uint32_t c2,
                                   uint32_t c3, uint32_t* out, size_t n) {
  const size_t g = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (4 * g >= n) return;
  const U4 w = philox4x32_10(U4{c0 + (uint32_t)g, c1, c2, c3}, k0, k1);
  const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
  for (int j = 0; j < 4; ++j)
    if (4 * g + j < n) out[4 * g + j] = ws[j];
}

cudaError_t launch_philox_fill(unsigned long long seed, uint32_t c0, uint32_t c1, uint32_t c2,
                               uint32_t c3, uint32_t* out, size_t n, cudaStream_t s) {
  const size_t groups = (n + 3) / 4;
  if (groups == 0) return cudaSuccess;
  const unsigned grid = (unsigned)((groups + 255) / 256);
  philox_fill_kernel<<<grid, 256, 0, s>>>(seed_lo(seed), seed_hi(seed), c0, c1, c2, c3, out, n);
  return cudaGetLastError();
}

}  // namespace cmsd
