// Internal declarations shared by the kernels and the C-ABI layer of libcmsd.so.
#pragma once
#include <cuda_runtime.h>
#include <stdint.h>

namespace cmsd {

// The streaming kernel runs as few, large CTAs (one per SM by default): warps
// of one CTA are scheduled evenly, warps of co-resident CTAs are not.
#ifndef CMSD_STREAM_THREADS
#define CMSD_STREAM_THREADS 768
#endif
constexpr int kStreamThreads = CMSD_STREAM_THREADS;
#ifndef CMSD_RES_THREADS
#define CMSD_RES_THREADS 256
#endif
constexpr int kResThreads = CMSD_RES_THREADS;   // threads per CTA of the resample kernel
constexpr int kResWarps = kResThreads / 32;
constexpr int kStreamWarps = kStreamThreads / 32;
constexpr int kMaxWarpsPerSM = 64;            // 2048 threads / SM
constexpr int kMaxRaggedB = 12000;            // B limit when k_row is given (prefix in smem)
constexpr int kPackedMaxK = 16;               // windows merged through one 64-bit counter

enum Mode { kModeConf = 0, kModeVerify = 1, kModeFused = 2 };

// Second pass over one row of a sequence, after its first-reject scan:
// the residual draw at a rejected position (sampled rule), or the token of
// the verifier's extra row when every draft was accepted (bonus row).
enum SeqKind { kSeqNone = 0, kSeqResidual = 1, kSeqBonus = 2 };

// Residual / bonus races run over groups of kGroup consecutive entries.
constexpr int kGroup = 32;

// dynamic shared memory of one streaming CTA: the k_row prefix (ragged windows)
__host__ __device__ inline size_t stream_smem_bytes(int B, bool ragged) {
  return ragged ? (((size_t)(B + 1) * sizeof(int) + 127) / 128) * 128 : 0;
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

// One resample warp's result for one queued row: its least race key (or, for
// the bonus argmax, minus its largest logit), its group and its token.
struct __align__(16) UnitResult {
  float key;
  float ref;   // bonus race: the warp's exponent reference (max * log2 e)
  int grp;
  int tok;
};

struct Workspace {
  // counters (zero at rest; each call returns them to zero)
  unsigned* err;                  // [1]   sticky device-side errors
  int* row_done;                  // [B*K] logits of the row already reduced
  unsigned long long* seq_word;   // [B]   K <= 16: rows merged | accept bits | sum of C (fixed point)
  int* seq_done;                  // [B]   K > 16: rows merged
  int* rec_count;                 // [1]   sequences queued for the second pass
  int* res_cta_done;              // [1]   CTAs of the resample kernel that finished
  int* res_done;                  // [B]   groups of each queued row already raced
  // per-call scratch
  int4* rec;                      // [B]   queued rows: (b, position, kind, 0)
  unsigned long long* row_conf;   // [B*K] C of each position, fixed point C * 2^36
  int* row_acc;                   // [B*K] accept bit (K > 16 epilogue)
  int* row_targmax;               // [B*K] verifier argmax
  float2* row_dstat;              // [B*K] drafter (max * log2e, sum e^(z-max))
  float2* row_tstat;              // [B*K] target  (the same)
  Partial* part;                  // [B*K + warps]
  UnitResult* rpart;              // [B + warps]
};

struct StreamArgs {
  const void* draft;
  const void* target;
  const int* tokens;
  const int* k_row;
  int B, K, V;
  int Kt;                 // verifier rows per sequence: K, or K + 1 with the bonus row
  int Ko;                 // out_tokens columns: K, or K + 1 with the bonus row
  int k_min, k_max, k_fixed;
  float lam0, lam1, lam2, beta_sig;
  float inv_log_v;        // 1 / ln V
  float soft_norm;        // 1 / (1 - 1/V)
  int beta_rank;
  float alpha, tau_base, gamma;
  int tau_sign;
  int bonus;
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
  int rec_by_seq;         // 1: second-pass records at each sequence's own slot rec[b], every sequence
                          // writing one (the bounded residual draw); 0: a compacted queue (rec_count)
};

// Kernel launchers (one translation unit per dtype).  `second`: this call
// queues rows for the resample kernel (sampled rule or bonus row).
cudaError_t launch_stream_f32(int mode, bool sampled, bool second, const StreamArgs& a, int grid,
                              size_t smem, cudaStream_t s);
cudaError_t launch_stream_bf16(int mode, bool sampled, bool second, const StreamArgs& a, int grid,
                               size_t smem, cudaStream_t s);
cudaError_t launch_resample_f32(bool sampled, const StreamArgs& a, int grid, cudaStream_t s);
cudaError_t launch_resample_bf16(bool sampled, const StreamArgs& a, int grid, cudaStream_t s);
// The residual draw by group bounds (sampled rule, no bonus row): clusters
// of CTAs, one queued row per cluster at a time; resample_bound_fits says
// whether a row's share fits its shared memory and such a cluster can be
// resident on the current device (else resample_kernel draws the residual).
cudaError_t launch_resample_bound_f32(const StreamArgs& a, int clusters, cudaStream_t s);
cudaError_t launch_resample_bound_bf16(const StreamArgs& a, int clusters, cudaStream_t s);
bool resample_bound_fits(int dtype, int V);
cudaError_t occupancy_stream(int dtype, int mode, bool sampled, bool second, size_t smem,
                             int* blocks_per_sm);
cudaError_t occupancy_resample(int dtype, bool sampled, int* blocks_per_sm);
cudaError_t launch_philox_fill(unsigned long long seed, uint32_t c0, uint32_t c1, uint32_t c2,
                               uint32_t c3, uint32_t* out, size_t n, cudaStream_t s);

// The drafter's LM head fused with its confidence signals (cmsd_lmhead.cu).
struct LmHeadArgs {
  const uint16_t* hidden;        // bf16 [R][d]
  const uint16_t* weight;        // bf16 [V][d]
  int R, d, V;
  int nb;                        // hidden rows per block (lmhead_block_rows(R))
  int nct;                       // CTAs per block (each owns a run of the vocabulary)
  float* logits;                 // nullable: f32 [R][V]
  Partial* part;                 // [ceil(R / nb)][nct][nb] per-CTA row statistics
  unsigned* err;                 // error word (bit 2: a wait for a load gave up)
};
int lmhead_block_rows(int R);
int lmhead_ctas_per_block(int sms, int R, int V);
// The GEMM + statistics kernel, then the per-row merge (a programmatic
// dependent on the same stream).  a carries the parameters, the output
// pointers and a workspace with row_conf [R].
cudaError_t launch_lmhead(const LmHeadArgs& h, const StreamArgs& a, cudaStream_t s);

// Host-side checks shared by the entry points (cmsd_api.cu).
int validate_fused(const void* draft_logits, const void* target_logits, const int32_t* draft_tokens,
                   const int32_t* k_row, int B, int K, int V, int dtype, const void* params,
                   const int32_t* n_accept, const int32_t* out_tokens);

}  // namespace cmsd
