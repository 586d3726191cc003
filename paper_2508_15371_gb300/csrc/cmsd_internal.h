// Internal declarations shared by the kernels and the C-ABI layer of libcmsd.so.
#pragma once
#include <cuda_runtime.h>
#include <stdint.h>

namespace cmsd {

#ifndef CMSD_RES_THREADS
#define CMSD_RES_THREADS 256
#endif
constexpr int kThreads = CMSD_RES_THREADS;    // threads per CTA (resample kernel)
constexpr int kWarpsPerBlock = kThreads / 32;
// The streaming kernel runs as few, large CTAs (one per SM by default): warps
// of one CTA are scheduled evenly, warps of co-resident CTAs are not.
#ifndef CMSD_STREAM_THREADS
#define CMSD_STREAM_THREADS 768
#endif
constexpr int kStreamThreads = CMSD_STREAM_THREADS;
constexpr int kStreamWarps = kStreamThreads / 32;
constexpr int kMaxWarpsPerSM = 64;            // 2048 threads / SM
constexpr int kMaxRaggedB = 12000;            // B limit when k_row is given (prefix in smem)

enum Mode { kModeConf = 0, kModeVerify = 1, kModeFused = 2 };

// dynamic shared memory of one streaming CTA: the k_row prefix (ragged windows)
__host__ __device__ inline size_t stream_pref_bytes(int B, bool ragged) {
  return ragged ? (((size_t)(B + 1) * sizeof(int) + 127) / 128) * 128 : 0;
}
__host__ __device__ inline size_t stream_smem_bytes(int B, bool ragged) {
  return stream_pref_bytes(B, ragged);
}

// One warp's reduction over one row segment (or, in the row merge, the
// reduction over all segments).  Drafter: running max m, s = sum e^(z-m),
// t2 = sum e^(z-m) (z-m) log2(e), second largest logit, lowest argmax.
// Target: running max, s = sum e^(z-m), lowest argmax, count of logits
// strictly above the drafted token's (saturating at beta_rank).
struct __align__(16) Partial {
  float d_m, d_s, d_t2, d_top2;
  int d_idx;
  float t_m, t_s;
  int t_idx, t_cnt;
  int pad[3];
};

struct __align__(16) RacePartial {
  float key;   // least E_g / R_g of the warp's groups of one row
  int grp;     // its group (lowest on ties)
  int tok;     // the level-2 winner inside that group
  int pad;
};

// One rejected position queued for the residual draw (SAMPLED rule).
struct __align__(16) RejRec {
  int r;             // row index b*K + n
  int b, n;
  int targmax;       // verifier argmax (fallback for an empty residual)
  float MLt, invSt;  // verifier: max*log2e, 1 / sum e^(z-max)
  float MLd, invSd;  // drafter: the same
};

struct Workspace {
  // counters (zero at rest; each call returns them to zero)
  int* row_done;       // [B*K] logits of the row already reduced
  int* seq_done;       // [B]   rows of the sequence already merged
  int* res_done;       // [B]   groups of each queued residual row already raced
  int* rej_count;      // [1]   sequences queued for a residual draw
  int* res_cta_done;   // [1]   CTAs of the resample kernel that finished
  unsigned* err;       // [1]   sticky device-side input errors
  // per-call scratch
  RejRec* rej;         // [B]   queued rejected positions
  float* row_conf;     // [B*K]
  int* row_acc;        // [B*K]
  int* row_targmax;    // [B*K]
  float2* row_dstat;   // [B*K] drafter (m*log2e, sum e^(z-m))
  float2* row_tstat;   // [B*K] target  (m*log2e, sum e^(z-m))
  Partial* part;       // [B*K + warps]
  RacePartial* rpart;  // [B + warps]
};

struct StreamArgs {
  const void* draft;
  const void* target;
  const int* tokens;
  const int* k_row;
  int B, K, V;
  int k_min, k_max;
  float lam0, lam1, lam2, beta_sig;
  int beta_rank;
  float alpha, tau_base, gamma;
  int tau_sign;
  unsigned long long seed;
  unsigned iteration;
  const float* conf_in;   // verify-only
  const float* lse_in;    // verify-only, SAMPLED
  float* H;
  float* margin;
  int* argmax;
  float* conf;
  float* lse;
  int* k_next;
  int* n_accept;
  int* out_tokens;
  unsigned char* accept;
  Workspace ws;
  int nwarps;             // warps launched
};

// Kernel launchers (one translation unit per dtype).
cudaError_t launch_stream_f32(int mode, bool sampled, const StreamArgs& a, int grid, size_t smem,
                              cudaStream_t s);
cudaError_t launch_stream_bf16(int mode, bool sampled, const StreamArgs& a, int grid, size_t smem,
                               cudaStream_t s);
cudaError_t launch_resample_f32(const StreamArgs& a, int grid, cudaStream_t s);
cudaError_t launch_resample_bf16(const StreamArgs& a, int grid, cudaStream_t s);
cudaError_t occupancy_stream(int dtype, int mode, bool sampled, size_t smem, int* blocks_per_sm);
cudaError_t occupancy_resample(int dtype, int* blocks_per_sm);
cudaError_t launch_philox_fill(unsigned long long seed, uint32_t c0, uint32_t c1, uint32_t c2,
                               uint32_t c3, uint32_t* out, size_t n, cudaStream_t s);

}  // namespace cmsd
