// Device generator of the decode-loop simulation's synthetic logits
// (include/cmsd_workload.h).  Input generation only: bit-identical to the
// host recipe (table lookups and IEEE float adds/multiplies with no
// contraction), so the CPU oracle can regenerate the same rows.
#include <cuda_runtime.h>
#include <stdint.h>

#include "cmsd_philox.cuh"
#include "cmsd_workload.h"

namespace {

constexpr uint32_t kGenDNoise = 0xC0000002u;
constexpr uint32_t kGenTNoise = 0xC0000003u;
constexpr uint32_t kGenSpike = 0xC0000004u;
constexpr int kThreads = 1024;   // one row per CTA; most slots of a window are idle
constexpr int kTableBits = 13;   // the normal table: 2^13 float32, staged in shared memory

__device__ __forceinline__ uint32_t half16(const cmsd::U4& w, int j) {
  const uint32_t word = (j >> 1) == 0 ? w.x : (j >> 1) == 1 ? w.y : (j >> 1) == 2 ? w.z : w.w;
  return (j & 1) ? (word >> 16) : (word & 0xFFFFu);
}

// One CTA per (b, i) slot of the [B][Kt] verifier layout.
__global__ void __launch_bounds__(kThreads) gen_rows_kernel(const float* __restrict__ table,
                                                            const float* __restrict__ heights_it,
                                                            uint32_t it, int B, int K_max, int Kt, int V,
                                                            const int32_t* __restrict__ k_row,
                                                            uint32_t k0, uint32_t k1, float* draft,
                                                            float* target, int32_t* tokens) {
  const int b = blockIdx.x / Kt;
  const int i = blockIdx.x - b * Kt;
  int k = K_max;
  if (k_row) {
    k = k_row[b];
    k = k < 0 ? 0 : (k > K_max ? K_max : k);
  }
  const bool has_draft = i < k;
  if (!has_draft && i >= k + (Kt - K_max)) return;
  __shared__ float s_table[1 << kTableBits];
  for (int j = threadIdx.x; j < (1 << kTableBits); j += kThreads) s_table[j] = table[j];
  __syncthreads();
  const int row = b * (K_max + 1) + i;          // generator row id
  const float h = heights_it[b];
  const cmsd::U4 sw = cmsd::philox4x32_10(cmsd::U4{0u, (uint32_t)row, it, kGenSpike}, k0, k1);
  const int spike = (int)(((uint64_t)sw.x * (uint64_t)V) >> 32);
  float* dz = draft + ((size_t)b * K_max + i) * V;
  float* tz = target + ((size_t)b * Kt + i) * V;

  float best = -__int_as_float(0x7F800000);
  int bidx = 0x7FFFFFFF;
  const int ngrp = (V + 7) / 8;
  // rows start on 16-byte boundaries when V is a multiple of 4: each thread
  // then writes its 8 logits as two 16-byte stores
  const bool vec = (V & 3) == 0;
  for (int g = threadIdx.x; g < ngrp; g += kThreads) {
    const cmsd::U4 wd = cmsd::philox4x32_10(cmsd::U4{(uint32_t)g, (uint32_t)row, it, kGenDNoise}, k0, k1);
    const cmsd::U4 wt = cmsd::philox4x32_10(cmsd::U4{(uint32_t)g, (uint32_t)row, it, kGenTNoise}, k0, k1);
    float zs[8], ts[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int v = 8 * g + j;
      float z = s_table[half16(wd, j) >> (16 - kTableBits)];
      if (v == spike) z = __fadd_rn(z, h);
      zs[j] = z;
      ts[j] = __fadd_rn(z, __fmul_rn(0.8f, s_table[half16(wt, j) >> (16 - kTableBits)]));
      if (v < V && z > best) { best = z; bidx = v; }
    }
    if (vec && 8 * g + 8 <= V) {
      float4* d4 = reinterpret_cast<float4*>(dz + 8 * g);
      float4* t4 = reinterpret_cast<float4*>(tz + 8 * g);
      if (has_draft) {
        d4[0] = make_float4(zs[0], zs[1], zs[2], zs[3]);
        d4[1] = make_float4(zs[4], zs[5], zs[6], zs[7]);
      }
      t4[0] = make_float4(ts[0], ts[1], ts[2], ts[3]);
      t4[1] = make_float4(ts[4], ts[5], ts[6], ts[7]);
    } else {
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const int v = 8 * g + j;
        if (v < V) {
          if (has_draft) dz[v] = zs[j];
          tz[v] = ts[j];
        }
      }
    }
  }
  if (!has_draft) return;     // the verifier's extra row has no drafted token
  // block argmax, lowest index among equal maxima
  for (int o = 16; o; o >>= 1) {
    const float ob = __shfl_xor_sync(0xFFFFFFFFu, best, o);
    const int oi = __shfl_xor_sync(0xFFFFFFFFu, bidx, o);
    if (ob > best || (ob == best && oi < bidx)) { best = ob; bidx = oi; }
  }
  __shared__ float sb[kThreads / 32];
  __shared__ int si[kThreads / 32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (lane == 0) { sb[warp] = best; si[warp] = bidx; }
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int w = 1; w < kThreads / 32; ++w)
      if (sb[w] > best || (sb[w] == best && si[w] < bidx)) { best = sb[w]; bidx = si[w]; }
    tokens[(size_t)b * K_max + i] = bidx;
  }
}

}  // namespace

extern "C" int cmsd_gen_decode_rows(const float* table, const float* heights_it, uint32_t it, int B,
                                    int K_max, int Kt, int V, const int32_t* k_row, uint64_t seed,
                                    float* draft, float* target, int32_t* tokens, void* stream) {
  if (B < 0 || K_max < 1 || V < 2 || (Kt != K_max && Kt != K_max + 1)) return -1;
  if (B == 0) return 0;
  if (!table || !heights_it || !draft || !target || !tokens) return -1;
  gen_rows_kernel<<<B * Kt, kThreads, 0, (cudaStream_t)stream>>>(
      table, heights_it, it, B, K_max, Kt, V, k_row, cmsd::seed_lo(seed), cmsd::seed_hi(seed), draft,
      target, tokens);
  return cudaGetLastError() == cudaSuccess ? 0 : -3;
}
