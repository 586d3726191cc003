// C ABI of libcmsd.so: argument checks, workspace layout, launches, timing.
// The operations are specified in include/cmsd.h.
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>
#include <string.h>

#include <map>
#include <mutex>
#include <tuple>
#include <vector>

#include "cmsd.h"
#include "cmsd_internal.h"
#include "cmsd_philox.cuh"

using namespace cmsd;

namespace {

thread_local int g_last_cuda = 0;

int cuda_fail(cudaError_t e) {
  g_last_cuda = (int)e;
  return CMSD_ECUDA;
}

std::mutex g_mu;
std::map<int, int> g_sms;                                   // device -> SM count
std::map<std::tuple<int, int, int, int, int>, int> g_occ;   // (dev, dtype, mode, variant, smem) -> blocks/SM
std::map<std::tuple<int, int, int>, int> g_occ_res;          // (dev, dtype, sampled) -> blocks/SM

int device_sms(int* sms) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e);
  std::lock_guard<std::mutex> lk(g_mu);
  auto it = g_sms.find(dev);
  if (it == g_sms.end()) {
    int n = 0;
    e = cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return cuda_fail(e);
    it = g_sms.emplace(dev, n).first;
  }
  *sms = it->second;
  return CMSD_OK;
}

int stream_grid(int dtype, int mode, bool sampled, bool second, size_t smem, int* grid) {
  int sms = 0;
  int rc = device_sms(&sms);
  if (rc) return rc;
  int dev = 0;
  cudaGetDevice(&dev);
  const int variant = (sampled ? 1 : 0) | (second ? 2 : 0);
  const auto key = std::make_tuple(dev, dtype, mode, variant, (int)smem);
  std::lock_guard<std::mutex> lk(g_mu);
  auto it = g_occ.find(key);
  if (it == g_occ.end()) {
    int nb = 0;
    cudaError_t e = occupancy_stream(dtype, mode, sampled, second, smem, &nb);
    if (e != cudaSuccess) return cuda_fail(e);
    if (nb < 1) nb = 1;
    it = g_occ.emplace(key, nb).first;
  }
  *grid = sms * it->second;
  return CMSD_OK;
}

int resample_grid(int dtype, bool sampled, int* grid) {
  int sms = 0;
  int rc = device_sms(&sms);
  if (rc) return rc;
  int dev = 0;
  cudaGetDevice(&dev);
  const auto key = std::make_tuple(dev, dtype, sampled ? 1 : 0);
  std::lock_guard<std::mutex> lk(g_mu);
  auto it = g_occ_res.find(key);
  if (it == g_occ_res.end()) {
    int nb = 0;
    cudaError_t e = occupancy_resample(dtype, sampled, &nb);
    if (e != cudaSuccess) return cuda_fail(e);
    if (nb < 1) nb = 1;
    it = g_occ_res.emplace(key, nb).first;
  }
  *grid = sms * it->second;
  return CMSD_OK;
}

// ---------------------------------------------------------------- workspace

constexpr size_t kAlign = 256;
size_t up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }

struct Layout {
  size_t err, row_done, seq_word, seq_done, rec_count, res_cta_done, res_done;
  size_t rec, row_conf, row_acc, row_targmax, row_dstat, row_tstat, part, rpart;
  size_t total;
};

// The error word sits at offset 0 so that cmsd_workspace_errors needs no sizes;
// the two queue counters follow it (offsets 256 and 512).
Layout make_layout(int B, int K, int wmax) {
  Layout L;
  const size_t BK = (size_t)B * (size_t)K;
  size_t o = 0;
  L.err = o; o += up(sizeof(unsigned));
  L.rec_count = o; o += up(sizeof(int));
  L.res_cta_done = o; o += up(sizeof(int));
  L.row_done = o; o += up(BK * sizeof(int));
  L.seq_word = o; o += up((size_t)B * sizeof(unsigned long long));
  L.seq_done = o; o += up((size_t)B * sizeof(int));
  L.res_done = o; o += up((size_t)B * sizeof(int));
  L.rec = o; o += up((size_t)B * sizeof(int4));
  L.row_conf = o; o += up(BK * sizeof(unsigned long long));
  L.row_acc = o; o += up(BK * sizeof(int));
  L.row_targmax = o; o += up(BK * sizeof(int));
  L.row_dstat = o; o += up(BK * sizeof(float2));
  L.row_tstat = o; o += up(BK * sizeof(float2));
  L.part = o; o += up((BK + (size_t)wmax) * sizeof(Partial));
  L.rpart = o; o += up(((size_t)B + (size_t)wmax) * sizeof(UnitResult));
  L.total = o;
  return L;
}

Workspace carve(void* ws, const Layout& L) {
  char* p = (char*)ws;
  Workspace W;
  W.err = (unsigned*)(p + L.err);
  W.row_done = (int*)(p + L.row_done);
  W.seq_word = (unsigned long long*)(p + L.seq_word);
  W.seq_done = (int*)(p + L.seq_done);
  W.rec_count = (int*)(p + L.rec_count);
  W.res_cta_done = (int*)(p + L.res_cta_done);
  W.res_done = (int*)(p + L.res_done);
  W.rec = (int4*)(p + L.rec);
  W.row_conf = (unsigned long long*)(p + L.row_conf);
  W.row_acc = (int*)(p + L.row_acc);
  W.row_targmax = (int*)(p + L.row_targmax);
  W.row_dstat = (float2*)(p + L.row_dstat);
  W.row_tstat = (float2*)(p + L.row_tstat);
  W.part = (Partial*)(p + L.part);
  W.rpart = (UnitResult*)(p + L.rpart);
  return W;
}

int wmax_warps(int* wmax) {
  int sms = 0;
  int rc = device_sms(&sms);
  if (rc) return rc;
  *wmax = sms * kMaxWarpsPerSM;
  return CMSD_OK;
}

// ---------------------------------------------------------------- timing

struct Profiler {
  bool on = false;
  int max_calls = 0;
  int n = 0;
  std::vector<cudaEvent_t> ev;   // 3 per call: start, after the streaming kernel, after the resample kernel
} g_prof;

void prof_record(int slot, cudaStream_t s) {
  if (!g_prof.on || g_prof.n >= g_prof.max_calls) return;
  cudaEventRecord(g_prof.ev[3 * g_prof.n + slot], s);
  if (slot == 2) ++g_prof.n;
}

// ---------------------------------------------------------------- checks

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

int check_sizes(int B, int K, int V, int dtype, const int32_t* k_row) {
  if (dtype != CMSD_F32 && dtype != CMSD_BF16) return CMSD_EDTYPE;
  if (B < 0 || K < 0 || K > 1024 || V < 2) return CMSD_EINVAL;
  if ((long long)B * (long long)K > 0x7FFFFFFFLL) return CMSD_EINVAL;
  if ((double)B * (double)K * (double)V >= 70368744177664.0) return CMSD_EINVAL;   // 2^46
  if (k_row && B > kMaxRaggedB) return CMSD_EINVAL;
  return CMSD_OK;
}

int check_params(const cmsd_params* p, bool need_rule) {
  if (!p) return CMSD_EINVAL;
  if (need_rule && p->rule != CMSD_RULE_PAPER && p->rule != CMSD_RULE_SAMPLED) return CMSD_EDTYPE;
  if (p->k_min < 1 || p->k_max < p->k_min) return CMSD_EINVAL;
  float sum = 0.f;
  for (int j = 0; j < 3; ++j) {
    if (!(p->lambda[j] >= 0.f && p->lambda[j] <= 1.f)) return CMSD_EINVAL;
    sum += p->lambda[j];
  }
  if (fabsf(sum - 1.0f) > 1e-5f) return CMSD_EINVAL;
  if (!(p->beta_sig > 0.f) || !isfinite(p->beta_sig)) return CMSD_EINVAL;
  if (p->beta_rank < 0) return CMSD_EINVAL;
  if (!(p->alpha > 0.f && p->alpha <= 1.f)) return CMSD_EINVAL;
  if (!isfinite(p->tau_base) || !isfinite(p->gamma)) return CMSD_EINVAL;
  if (p->tau_sign != 1 && p->tau_sign != -1) return CMSD_EINVAL;
  if (p->k_fixed != 0 && (p->k_fixed < p->k_min || p->k_fixed > p->k_max)) return CMSD_EINVAL;
  if (p->bonus != 0 && p->bonus != 1) return CMSD_EINVAL;
  return CMSD_OK;
}

// With the bonus row the verifier tensor has K + 1 rows per sequence while the
// drafter's has K: their rows stay equally aligned only if a row is a whole
// number of 16-byte vectors.
int check_bonus_layout(const cmsd_params* p, int V, int dtype) {
  if (!p->bonus) return CMSD_OK;
  const size_t row_bytes = (size_t)V * (dtype == CMSD_F32 ? 4 : 2);
  return (row_bytes % 16) == 0 ? CMSD_OK : CMSD_EINVAL;
}

void fill_params(StreamArgs& a, const cmsd_params* p) {
  a.k_min = p->k_min;
  a.k_max = p->k_max;
  a.lam0 = p->lambda[0];
  a.lam1 = p->lambda[1];
  a.lam2 = p->lambda[2];
  a.beta_sig = p->beta_sig;
  a.beta_rank = p->beta_rank;
  a.alpha = p->alpha;
  a.tau_base = p->tau_base;
  a.gamma = p->gamma;
  a.tau_sign = p->tau_sign;
  a.k_fixed = p->k_fixed;
  a.bonus = p->bonus;
}

void fill_sizes(StreamArgs& a, int B, int K, int V) {
  a.B = B; a.K = K; a.V = V;
  a.inv_log_v = (float)(1.0 / log((double)V));
  a.soft_norm = (float)(1.0 / (1.0 - 1.0 / (double)V));
}

int launch(int dtype, int mode, bool sampled, StreamArgs& a, void* ws, size_t ws_bytes,
           cudaStream_t s) {
  int wmax = 0;
  int rc = wmax_warps(&wmax);
  if (rc) return rc;
  const Layout L = make_layout(a.B, a.K, wmax);
  if (!ws || ws_bytes < L.total) return CMSD_ENOWS;
  a.ws = carve(ws, L);
  const bool bonus = mode != kModeConf && a.bonus;
  a.Kt = bonus ? a.K + 1 : a.K;
  a.Ko = bonus ? a.K + 1 : a.K;
  const bool second = mode != kModeConf && (sampled || bonus);
  const size_t smem = stream_smem_bytes(a.B, a.k_row != nullptr);
  int grid = 0;
  rc = stream_grid(dtype, mode, sampled, second, smem, &grid);
  if (rc) return rc;
  int g2 = 0, nclu = 0;
  // the sampled rule's residual draw without the bonus row: by group bounds,
  // one cluster per queued row (up to two per SM pair's worth; more rows loop)
  const bool bound = second && sampled && !bonus && resample_bound_fits(dtype, a.V);
  if (second) {
    rc = resample_grid(dtype, sampled, &g2);
    if (rc) return rc;
    int sms = 0;
    rc = device_sms(&sms);
    if (rc) return rc;
    nclu = a.B < 2 * sms ? a.B : 2 * sms;
  }
  a.nwarps = grid * kStreamWarps;
  a.rec_by_seq = bound ? 1 : 0;
  prof_record(0, s);
  cudaError_t e = dtype == CMSD_F32 ? launch_stream_f32(mode, sampled, second, a, grid, smem, s)
                                    : launch_stream_bf16(mode, sampled, second, a, grid, smem, s);
  if (e != cudaSuccess) return cuda_fail(e);
  prof_record(1, s);
  if (second) {
    StreamArgs b = a;
    b.nwarps = g2 * kResWarps;
    if (bound)
      e = dtype == CMSD_F32 ? launch_resample_bound_f32(b, nclu, s) : launch_resample_bound_bf16(b, nclu, s);
    else
      e = dtype == CMSD_F32 ? launch_resample_f32(sampled, b, g2, s) : launch_resample_bf16(sampled, b, g2, s);
    if (e != cudaSuccess) {
      // the streaming kernel has queued rows that no resample kernel will
      // drain: return the queue counters to zero so the workspace stays usable
      cudaMemsetAsync(a.ws.rec_count, 0, sizeof(int), s);
      cudaMemsetAsync(a.ws.res_cta_done, 0, sizeof(int), s);
      if (bound) cudaMemsetAsync(a.ws.rec, 0, (size_t)a.B * sizeof(int4), s);   // the released record words
      return cuda_fail(e);
    }
  }
  prof_record(2, s);
  return CMSD_OK;
}

StreamArgs blank_args() {
  StreamArgs a;
  memset(&a, 0, sizeof(a));
  return a;
}

}  // namespace

namespace cmsd {

// Every host-side check of cmsd_confidence_verify (sizes, parameters, bonus
// layout, required pointers, alignment), without launching anything.
int validate_fused(const void* draft_logits, const void* target_logits, const int32_t* draft_tokens,
                   const int32_t* k_row, int B, int K, int V, int dtype, const void* params,
                   const int32_t* n_accept, const int32_t* out_tokens) {
  const cmsd_params* p = (const cmsd_params*)params;
  int rc = check_sizes(B, K, V, dtype, k_row);
  if (rc) return rc;
  rc = check_params(p, true);
  if (rc) return rc;
  rc = check_bonus_layout(p, V, dtype);
  if (rc) return rc;
  if (B == 0 || K == 0) return CMSD_OK;
  if (!draft_logits || !target_logits || !draft_tokens || !n_accept || !out_tokens) return CMSD_EINVAL;
  if (!aligned16(draft_logits) || !aligned16(target_logits)) return CMSD_EALIGN;
  return CMSD_OK;
}

}  // namespace cmsd

// ============================================================ C ABI

// ---------------------------------------------------------------- LM head

namespace {
struct LmLayout {
  size_t row_conf, part, total;
  int nct, nb;
};
int lm_layout(int R, int V, LmLayout* L) {
  int sms = 0;
  int rc = device_sms(&sms);
  if (rc) return rc;
  L->nct = lmhead_ctas_per_block(sms, R, V);
  L->nb = lmhead_block_rows(R);
  const size_t nrb = (size_t)(R + L->nb - 1) / L->nb;
  size_t o = up(sizeof(unsigned));
  L->row_conf = o; o += up((size_t)R * sizeof(unsigned long long));
  L->part = o; o += up(nrb * (size_t)L->nct * L->nb * sizeof(Partial));
  L->total = o;
  return CMSD_OK;
}
int check_lmhead(int R, int d, int V) {
  if (R < 0 || d < 64 || d % 64 != 0 || d > (1 << 20) || V < 2) return CMSD_EINVAL;
  if ((double)R * (double)V >= 70368744177664.0) return CMSD_EINVAL;   // 2^46 logits
  return CMSD_OK;
}
}  // namespace

extern "C" {

void cmsd_params_default(cmsd_params* p, int K, int rule) {
  if (!p) return;
  p->k_min = 1;
  p->k_max = K > 0 ? K : 1;
  p->lambda[0] = p->lambda[1] = p->lambda[2] = 1.0f / 3.0f;
  p->beta_sig = 1.0f;
  p->beta_rank = rule == CMSD_RULE_SAMPLED ? 0 : 3;
  p->alpha = 1.0f;
  p->tau_base = 0.1f;
  p->gamma = 1.0f;
  p->tau_sign = 1;
  p->rule = rule;
  p->k_fixed = 0;
  p->bonus = 0;
}

int cmsd_params_preset(cmsd_params* p, int K, int rule, int preset) {
  if (!p) return CMSD_EINVAL;
  cmsd_params_default(p, K, rule);
  switch (preset) {
    case CMSD_PRESET_FULL: break;
    case CMSD_PRESET_FIXED_K: p->k_fixed = p->k_max; break;
    case CMSD_PRESET_FIXED_TAU: p->gamma = 0.0f; break;
    case CMSD_PRESET_FIXED_K_TAU: p->k_fixed = p->k_max; p->gamma = 0.0f; break;
    case CMSD_PRESET_ENTROPY_ONLY: p->lambda[0] = 1.0f; p->lambda[1] = p->lambda[2] = 0.0f; break;
    case CMSD_PRESET_MARGIN_ONLY: p->lambda[1] = 1.0f; p->lambda[0] = p->lambda[2] = 0.0f; break;
    case CMSD_PRESET_SOFTMAX_ONLY: p->lambda[2] = 1.0f; p->lambda[0] = p->lambda[1] = 0.0f; break;
    default: return CMSD_EINVAL;
  }
  return CMSD_OK;
}


size_t cmsd_lmhead_workspace_bytes(int R, int d, int V) {
  if (check_lmhead(R, d, V)) return 0;
  LmLayout L;
  if (lm_layout(R, V, &L)) return 0;
  return L.total;
}

int cmsd_lmhead_confidence(const void* hidden, const void* weight, int R, int d, int V,
                           const cmsd_params* p, float* H, float* margin, int32_t* argmax, float* conf,
                           float* lse, float* logits, void* ws, size_t ws_bytes, void* stream) {
  int rc = check_lmhead(R, d, V);
  if (rc) return rc;
  rc = check_params(p, false);
  if (rc) return rc;
  if (R == 0) return CMSD_OK;
  if (!hidden || !weight) return CMSD_EINVAL;
  if (!aligned16(hidden) || !aligned16(weight)) return CMSD_EALIGN;
  LmLayout L;
  rc = lm_layout(R, V, &L);
  if (rc) return rc;
  if (!ws || ws_bytes < L.total) return CMSD_ENOWS;
  StreamArgs a = blank_args();
  fill_sizes(a, R, 1, V);
  fill_params(a, p);
  a.Kt = a.Ko = 1;
  a.H = H; a.margin = margin; a.argmax = argmax; a.conf = conf; a.lse = lse;
  char* w = (char*)ws;
  a.ws.err = (unsigned*)w;
  a.ws.row_conf = (unsigned long long*)(w + L.row_conf);
  LmHeadArgs h;
  h.hidden = (const uint16_t*)hidden;
  h.weight = (const uint16_t*)weight;
  h.R = R; h.d = d; h.V = V;
  h.nct = L.nct;
  h.nb = L.nb;
  h.logits = logits;
  h.part = (Partial*)(w + L.part);
  h.err = a.ws.err;
  cudaError_t e = launch_lmhead(h, a, (cudaStream_t)stream);
  return e == cudaSuccess ? CMSD_OK : cuda_fail(e);
}

size_t cmsd_workspace_bytes(int B, int K, int V) {
  if (B < 0 || K < 0 || V < 2) return 0;
  int wmax = 0;
  if (wmax_warps(&wmax)) return 0;
  return make_layout(B, K, wmax).total;
}

int cmsd_workspace_init(void* ws, size_t ws_bytes, void* stream) {
  if (!ws || ws_bytes == 0) return CMSD_ENOWS;
  cudaError_t e = cudaMemsetAsync(ws, 0, ws_bytes, (cudaStream_t)stream);
  return e == cudaSuccess ? CMSD_OK : cuda_fail(e);
}

int cmsd_workspace_errors(void* ws, size_t ws_bytes, void* stream, uint32_t* flags_out) {
  if (!ws || ws_bytes < sizeof(unsigned) || !flags_out) return CMSD_EINVAL;
  unsigned h = 0;
  cudaStream_t s = (cudaStream_t)stream;
  cudaError_t e = cudaMemcpyAsync(&h, ws, sizeof(unsigned), cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaMemsetAsync(ws, 0, sizeof(unsigned), s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return cuda_fail(e);
  *flags_out = h;
  return CMSD_OK;
}

int cmsd_test_record_wait_timeout(const void* draft_logits, const void* target_logits, int B, int K, int V,
                                  int dtype, int32_t* out_tokens, void* ws, size_t ws_bytes, void* stream) {
  int rc = check_sizes(B, K, V, dtype, nullptr);
  if (rc) return rc;
  if (B == 0 || K == 0) return CMSD_OK;
  if (!draft_logits || !target_logits || !out_tokens) return CMSD_EINVAL;
  if (!aligned16(draft_logits) || !aligned16(target_logits)) return CMSD_EALIGN;
  if (!resample_bound_fits(dtype, V)) return CMSD_EDTYPE;
  int wmax = 0;
  rc = wmax_warps(&wmax);
  if (rc) return rc;
  const Layout L = make_layout(B, K, wmax);
  if (!ws || ws_bytes < L.total) return CMSD_ENOWS;
  int sms = 0;
  rc = device_sms(&sms);
  if (rc) return rc;
  StreamArgs a = blank_args();
  fill_sizes(a, B, K, V);
  a.draft = draft_logits;
  a.target = target_logits;
  a.out_tokens = out_tokens;
  a.Kt = a.Ko = K;
  a.rec_by_seq = 1;
  a.ws = carve(ws, L);
  cudaStream_t s = (cudaStream_t)stream;
  // no record is released: every sequence's wait runs out
  cudaError_t e = cudaMemsetAsync(a.ws.rec, 0, (size_t)B * sizeof(int4), s);
  if (e != cudaSuccess) return cuda_fail(e);
  const int nclu = B < 2 * sms ? B : 2 * sms;
  e = dtype == CMSD_F32 ? launch_resample_bound_f32(a, nclu, s) : launch_resample_bound_bf16(a, nclu, s);
  return e == cudaSuccess ? CMSD_OK : cuda_fail(e);
}

int cmsd_confidence(const void* draft_logits, int B, int K, int V, int dtype, const int32_t* k_row,
                    const cmsd_params* p, float* H, float* margin, int32_t* argmax, float* conf,
                    float* lse, int32_t* k_next, void* ws, size_t ws_bytes, void* stream) {
  int rc = check_sizes(B, K, V, dtype, k_row);
  if (rc) return rc;
  rc = check_params(p, false);
  if (rc) return rc;
  if (B == 0 || K == 0) return CMSD_OK;
  if (!draft_logits) return CMSD_EINVAL;
  if (!aligned16(draft_logits)) return CMSD_EALIGN;
  StreamArgs a = blank_args();
  a.draft = draft_logits;
  a.k_row = k_row;
  fill_sizes(a, B, K, V);
  fill_params(a, p);
  a.H = H; a.margin = margin; a.argmax = argmax; a.conf = conf; a.lse = lse; a.k_next = k_next;
  return launch(dtype, kModeConf, false, a, ws, ws_bytes, (cudaStream_t)stream);
}

int cmsd_verify(const void* draft_logits, const void* target_logits, const int32_t* draft_tokens,
                const int32_t* k_row, int B, int K, int V, int dtype, const cmsd_params* p,
                const float* conf, const float* draft_lse, uint64_t seed, uint32_t iteration,
                int32_t* n_accept, int32_t* out_tokens, uint8_t* accept, void* ws, size_t ws_bytes,
                void* stream) {
  int rc = check_sizes(B, K, V, dtype, k_row);
  if (rc) return rc;
  rc = check_params(p, true);
  if (rc) return rc;
  rc = check_bonus_layout(p, V, dtype);
  if (rc) return rc;
  if (B == 0 || K == 0) return CMSD_OK;
  const bool sampled = p->rule == CMSD_RULE_SAMPLED;
  if (!draft_logits || !target_logits || !draft_tokens || !conf || !n_accept || !out_tokens)
    return CMSD_EINVAL;
  if (sampled && !draft_lse) return CMSD_EINVAL;
  if (!aligned16(draft_logits) || !aligned16(target_logits)) return CMSD_EALIGN;
  StreamArgs a = blank_args();
  a.draft = draft_logits;
  a.target = target_logits;
  a.tokens = draft_tokens;
  a.k_row = k_row;
  fill_sizes(a, B, K, V);
  fill_params(a, p);
  a.seed = seed;
  a.iteration = iteration;
  a.conf_in = conf;
  a.lse_in = draft_lse;
  a.n_accept = n_accept; a.out_tokens = out_tokens; a.accept = accept;
  return launch(dtype, kModeVerify, sampled, a, ws, ws_bytes, (cudaStream_t)stream);
}

int cmsd_confidence_verify(const void* draft_logits, const void* target_logits,
                           const int32_t* draft_tokens, const int32_t* k_row, int B, int K, int V,
                           int dtype, const cmsd_params* p, uint64_t seed, uint32_t iteration,
                           float* H, float* margin, int32_t* argmax, float* conf, float* lse,
                           int32_t* k_next, int32_t* n_accept, int32_t* out_tokens, uint8_t* accept,
                           void* ws, size_t ws_bytes, void* stream) {
  const int rc = validate_fused(draft_logits, target_logits, draft_tokens, k_row, B, K, V, dtype, p,
                                n_accept, out_tokens);
  if (rc) return rc;
  if (B == 0 || K == 0) return CMSD_OK;
  const bool sampled = p->rule == CMSD_RULE_SAMPLED;
  StreamArgs a = blank_args();
  a.draft = draft_logits;
  a.target = target_logits;
  a.tokens = draft_tokens;
  a.k_row = k_row;
  fill_sizes(a, B, K, V);
  fill_params(a, p);
  a.seed = seed;
  a.iteration = iteration;
  a.H = H; a.margin = margin; a.argmax = argmax; a.conf = conf; a.lse = lse; a.k_next = k_next;
  a.n_accept = n_accept; a.out_tokens = out_tokens; a.accept = accept;
  return launch(dtype, kModeFused, sampled, a, ws, ws_bytes, (cudaStream_t)stream);
}

uint32_t cmsd_philox_u32(uint64_t seed, uint32_t c0, uint32_t c1, uint32_t c2, uint32_t c3, int word) {
  const U4 w = philox4x32_10(U4{c0, c1, c2, c3}, seed_lo(seed), seed_hi(seed));
  switch (word & 3) {
    case 0: return w.x;
    case 1: return w.y;
    case 2: return w.z;
    default: return w.w;
  }
}

int cmsd_philox_fill(uint64_t seed, uint32_t c0, uint32_t c1, uint32_t c2, uint32_t c3, uint32_t* out,
                     size_t n, void* stream) {
  if (n == 0) return CMSD_OK;
  if (!out) return CMSD_EINVAL;
  cudaError_t e = launch_philox_fill(seed, c0, c1, c2, c3, out, n, (cudaStream_t)stream);
  return e == cudaSuccess ? CMSD_OK : cuda_fail(e);
}

int cmsd_profile_start(int max_calls) {
  if (max_calls < 0) return CMSD_EINVAL;
  const size_t need = (size_t)max_calls * 3;
  while (g_prof.ev.size() < need) {
    cudaEvent_t e;
    cudaError_t err = cudaEventCreate(&e);
    if (err != cudaSuccess) return cuda_fail(err);
    g_prof.ev.push_back(e);
  }
  g_prof.on = true;
  g_prof.max_calls = max_calls;
  g_prof.n = 0;
  return CMSD_OK;
}

int cmsd_profile_stop(float* stream_ms, float* resample_ms, int max_out, int* n_out) {
  g_prof.on = false;
  const int n = g_prof.n < max_out ? g_prof.n : max_out;
  for (int j = 0; j < n; ++j) {
    cudaError_t e = cudaEventSynchronize(g_prof.ev[3 * j + 2]);
    if (e != cudaSuccess) return cuda_fail(e);
    float x = 0.f, y = 0.f;
    e = cudaEventElapsedTime(&x, g_prof.ev[3 * j], g_prof.ev[3 * j + 1]);
    if (e == cudaSuccess) e = cudaEventElapsedTime(&y, g_prof.ev[3 * j + 1], g_prof.ev[3 * j + 2]);
    if (e != cudaSuccess) return cuda_fail(e);
    if (stream_ms) stream_ms[j] = x;
    if (resample_ms) resample_ms[j] = y;
  }
  if (n_out) *n_out = n;
  g_prof.n = 0;
  return CMSD_OK;
}

int cmsd_launch_info(int dtype, int* warps_out, int* sms_out) {
  if (dtype != CMSD_F32 && dtype != CMSD_BF16) return CMSD_EDTYPE;
  int sms = 0, grid = 0;
  int rc = device_sms(&sms);
  if (rc) return rc;
  rc = stream_grid(dtype, kModeFused, true, true, stream_smem_bytes(0, false), &grid);
  if (rc) return rc;
  if (warps_out) *warps_out = grid * kStreamWarps;
  if (sms_out) *sms_out = sms;
  return CMSD_OK;
}

const char* cmsd_strerror(int code) {
  switch (code) {
    case CMSD_OK: return "ok";
    case CMSD_EINVAL: return "invalid argument";
    case CMSD_EDTYPE: return "unknown dtype or rule";
    case CMSD_ECUDA: return "CUDA runtime error";
    case CMSD_ENOWS: return "workspace missing or too small";
    case CMSD_EALIGN: return "logit pointer not 16-byte aligned";
    case CMSD_ESCRATCH: return "problem too large for the static scratch (CMSD_STATIC_SCRATCH_BYTES)";
    default: return "unknown error";
  }
}

int cmsd_last_cuda_error(void) { return g_last_cuda; }

}  // extern "C"
