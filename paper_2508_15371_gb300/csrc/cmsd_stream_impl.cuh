// Streaming kernels of the CM-ASD logits pass (sm_103a).
//
// Work split.  The present rows (sequence b, drafted position i < k_row[b])
// are laid end to end into one stream of rows * V logits per tensor, and the
// launched warps (a persistent grid: every SM filled to its occupancy) each
// take an equal contiguous slice of that stream.  A slice crosses at most a
// few row boundaries; each piece of a row it covers is a "segment".  A warp
// reads its segments with 128-bit non-caching loads, keeps per-lane running
// statistics in registers, reduces them across the warp with shuffles and
// writes one Partial per segment.  Per-row and per-sequence arrival counters
// (atomics, no waiting) elect the warp that completes a row to merge its
// partials into the row's results, and the warp that completes a sequence to
// run the sequence epilogue (first-reject scan, next draft length, output
// tokens).  Every logit is read from HBM once.
//
// Per-element work (online softmax, Sec. III.B(1)): with running maximum m,
//   s  = sum e^(z - m)
//   t2 = sum e^(z - m) * (z - m) * log2(e)
// so that the entropy is H = -sum p log p = ln2 * (log2 s - t2 / s); when m
// grows to m', s and t2 are rescaled by e^(m - m') (t2 also shifted by
// s * (m - m') log2 e).  The exponent is evaluated as ex2(z*log2e - m*log2e)
// with the product m*log2e rounded once and shared by every term of the
// row, so that rounding cancels in p = e^(z-m)/s.
//
// -inf logits (masked vocabulary) are clamped to kNegClamp before the
// drafter arithmetic so that e^(z-m) * (z-m) is 0, not NaN.
#pragma once
#include <cuda_runtime.h>
#include <stdint.h>

#include "cmsd_internal.h"
#include "cmsd_philox.cuh"

namespace cmsd {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
constexpr uint32_t kNegClampBits = 0xF14A0000u;       // bf16 value nearest -1e30
constexpr uint32_t kNegClamp2 = 0xF14AF14Au;          // the same, two bf16 lanes
constexpr uint32_t kNegInf2 = 0xFF80FF80u;            // -inf, two bf16 lanes
constexpr float kNegInit = -2.0e30f;                  // below every clamped logit
constexpr unsigned kFull = 0xFFFFFFFFu;

__device__ __forceinline__ float neg_clamp() { return __uint_as_float(kNegClampBits); }

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ uint32_t bmax2(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("max.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}
__device__ __forceinline__ uint32_t bmin2(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("min.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}
__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

__device__ __forceinline__ uint4 ld_stream(const void* p) {
  uint4 r;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p));
  return r;
}

template <typename T> struct Elem;
template <> struct Elem<float> {
  static constexpr int kVec = 4;
  __device__ static float load(const float* p) { return __ldg(p); }
};
template <> struct Elem<uint16_t> {
  static constexpr int kVec = 8;
  __device__ static float load(const uint16_t* p) {
    return __uint_as_float(((uint32_t)__ldg(p)) << 16);
  }
};

// ---------------------------------------------------------------------------
// per-lane running state
// ---------------------------------------------------------------------------

struct DLane {               // drafter
  float m, negmL;            // running max and -(m*log2e)
  float s0, s1, t0, t1;      // two interleaved accumulators for ILP
  float f1, f2;              // top-2 of elements taken one at a time (all f32 data)
  uint32_t T1, T2;           // top-2 of bf16 vector elements, per half-word lane
  int pos, posw;             // first unit (start, width) that reached m
};

struct TLane {               // target
  float M, negML;
  float s0, s1;
  int pos, posw;
  int cnt;
};

__device__ __forceinline__ void dlane_init(DLane& d) {
  d.m = kNegInit;
  d.negmL = -(kNegInit * kLog2e);
  d.s0 = d.s1 = d.t0 = d.t1 = 0.f;
  d.f1 = d.f2 = kNegInit;
  d.T1 = d.T2 = kNegInf2;
  d.pos = 0x7FFFFFFF;
  d.posw = 0;
}
__device__ __forceinline__ void tlane_init(TLane& t) {
  t.M = kNegInit;
  t.negML = -(kNegInit * kLog2e);
  t.s0 = t.s1 = 0.f;
  t.pos = 0x7FFFFFFF;
  t.posw = 0;
  t.cnt = 0;
}

__device__ __forceinline__ void d_raise(DLane& d, float mx, int pos, int posw) {
  const float nmL = mx * kLog2e;
  const float dd = -d.negmL - nmL;            // (m_old - m_new) log2e <= 0
  const float sc = ex2(dd);
  d.t0 = sc * fmaf(d.s0, dd, d.t0);
  d.t1 = sc * fmaf(d.s1, dd, d.t1);
  d.s0 *= sc;
  d.s1 *= sc;
  d.m = mx;
  d.negmL = -nmL;
  d.pos = pos;
  d.posw = posw;
}
__device__ __forceinline__ void d_acc0(DLane& d, float z) {
  const float x = fmaf(z, kLog2e, d.negmL);
  const float e = ex2(x);
  d.s0 += e;
  d.t0 = fmaf(e, x, d.t0);
}
__device__ __forceinline__ void d_acc1(DLane& d, float z) {
  const float x = fmaf(z, kLog2e, d.negmL);
  const float e = ex2(x);
  d.s1 += e;
  d.t1 = fmaf(e, x, d.t1);
}

__device__ __forceinline__ void t_raise(TLane& t, float mx, int pos, int posw, bool sampled) {
  const float nmL = mx * kLog2e;
  if (sampled) {
    const float sc = ex2(-t.negML - nmL);
    t.s0 *= sc;
    t.s1 *= sc;
  }
  t.M = mx;
  t.negML = -nmL;
  t.pos = pos;
  t.posw = posw;
}

// --- drafter: one element at a time (head/tail, or every f32 element) -------
__device__ __forceinline__ void d_scalar(DLane& d, float z, int v) {
  z = fmaxf(z, neg_clamp());
  d.f2 = fmaxf(d.f2, fminf(d.f1, z));
  d.f1 = fmaxf(d.f1, z);
  if (z > d.m) d_raise(d, z, v, 1);
  d_acc0(d, z);
}

// --- drafter: 8 bf16 ---------------------------------------------------------
__device__ __forceinline__ void d_vec(DLane& d, uint4 q, int v) {
  const uint32_t w0 = bmax2(q.x, kNegClamp2), w1 = bmax2(q.y, kNegClamp2);
  const uint32_t w2 = bmax2(q.z, kNegClamp2), w3 = bmax2(q.w, kNegClamp2);
  d.T2 = bmax2(d.T2, bmin2(d.T1, w0)); d.T1 = bmax2(d.T1, w0);
  d.T2 = bmax2(d.T2, bmin2(d.T1, w1)); d.T1 = bmax2(d.T1, w1);
  d.T2 = bmax2(d.T2, bmin2(d.T1, w2)); d.T1 = bmax2(d.T1, w2);
  d.T2 = bmax2(d.T2, bmin2(d.T1, w3)); d.T1 = bmax2(d.T1, w3);
  const float mx = fmaxf(bf_lo(d.T1), bf_hi(d.T1));
  if (mx > d.m) d_raise(d, mx, v, 8);
  d_acc0(d, bf_lo(w0)); d_acc1(d, bf_hi(w0));
  d_acc0(d, bf_lo(w1)); d_acc1(d, bf_hi(w1));
  d_acc0(d, bf_lo(w2)); d_acc1(d, bf_hi(w2));
  d_acc0(d, bf_lo(w3)); d_acc1(d, bf_hi(w3));
}

// --- drafter: 4 f32 ------------------------------------------------------------
__device__ __forceinline__ void d_vec(DLane& d, float4 q, int v) {
  const float nc = neg_clamp();
  const float z0 = fmaxf(q.x, nc), z1 = fmaxf(q.y, nc), z2 = fmaxf(q.z, nc), z3 = fmaxf(q.w, nc);
  d.f2 = fmaxf(d.f2, fminf(d.f1, z0)); d.f1 = fmaxf(d.f1, z0);
  d.f2 = fmaxf(d.f2, fminf(d.f1, z1)); d.f1 = fmaxf(d.f1, z1);
  d.f2 = fmaxf(d.f2, fminf(d.f1, z2)); d.f1 = fmaxf(d.f1, z2);
  d.f2 = fmaxf(d.f2, fminf(d.f1, z3)); d.f1 = fmaxf(d.f1, z3);
  if (d.f1 > d.m) d_raise(d, d.f1, v, 4);
  d_acc0(d, z0); d_acc1(d, z1); d_acc0(d, z2); d_acc1(d, z3);
}

// --- target: one element --------------------------------------------------------
template <bool SAMPLED>
__device__ __forceinline__ void t_scalar(TLane& t, float z, int v, float c, int beta) {
  if (z > t.M) t_raise(t, z, v, 1, SAMPLED);
  if (t.cnt < beta && z > c) ++t.cnt;
  if (SAMPLED) t.s0 += ex2(fmaf(z, kLog2e, t.negML));
}

template <bool SAMPLED>
__device__ __forceinline__ void t_vec(TLane& t, uint4 q, int v, float c, int beta) {
  const uint32_t a = bmax2(bmax2(q.x, q.y), bmax2(q.z, q.w));
  const float vmax = fmaxf(bf_lo(a), bf_hi(a));
  if (vmax > t.M) t_raise(t, vmax, v, 8, SAMPLED);
  if (t.cnt < beta && vmax > c) {
    const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      t.cnt += (bf_lo(w[k]) > c) + (bf_hi(w[k]) > c);
    }
  }
  if (SAMPLED) {
    const float n = t.negML;
    t.s0 += ex2(fmaf(bf_lo(q.x), kLog2e, n)); t.s1 += ex2(fmaf(bf_hi(q.x), kLog2e, n));
    t.s0 += ex2(fmaf(bf_lo(q.y), kLog2e, n)); t.s1 += ex2(fmaf(bf_hi(q.y), kLog2e, n));
    t.s0 += ex2(fmaf(bf_lo(q.z), kLog2e, n)); t.s1 += ex2(fmaf(bf_hi(q.z), kLog2e, n));
    t.s0 += ex2(fmaf(bf_lo(q.w), kLog2e, n)); t.s1 += ex2(fmaf(bf_hi(q.w), kLog2e, n));
  }
}

template <bool SAMPLED>
__device__ __forceinline__ void t_vec(TLane& t, float4 q, int v, float c, int beta) {
  const float vmax = fmaxf(fmaxf(q.x, q.y), fmaxf(q.z, q.w));
  if (vmax > t.M) t_raise(t, vmax, v, 4, SAMPLED);
  if (t.cnt < beta && vmax > c) t.cnt += (q.x > c) + (q.y > c) + (q.z > c) + (q.w > c);
  if (SAMPLED) {
    const float n = t.negML;
    t.s0 += ex2(fmaf(q.x, kLog2e, n)); t.s1 += ex2(fmaf(q.y, kLog2e, n));
    t.s0 += ex2(fmaf(q.z, kLog2e, n)); t.s1 += ex2(fmaf(q.w, kLog2e, n));
  }
}

template <typename T> struct VecT;
template <> struct VecT<float> { using type = float4; };
template <> struct VecT<uint16_t> { using type = uint4; };

template <typename T>
__device__ __forceinline__ typename VecT<T>::type as_vec(uint4 r);
template <> __device__ __forceinline__ float4 as_vec<float>(uint4 r) {
  return make_float4(__uint_as_float(r.x), __uint_as_float(r.y), __uint_as_float(r.z),
                     __uint_as_float(r.w));
}
template <> __device__ __forceinline__ uint4 as_vec<uint16_t>(uint4 r) { return r; }

// First index in the unit (start pos, width w) whose value equals m (drafter
// values clamped as in the streaming pass when `clamp`).
template <typename T>
__device__ __forceinline__ int first_equal(const T* row, int pos, int w, float m, bool clamp) {
  if (w <= 1) return pos;
  const float nc = neg_clamp();
  for (int k = 0; k < w; ++k) {
    float z = Elem<T>::load(row + pos + k);
    if (clamp) z = fmaxf(z, nc);
    if (z == m) return pos + k;
  }
  return pos;   // not reached
}

// ---------------------------------------------------------------------------
// warp reductions (results identical in every lane)
// ---------------------------------------------------------------------------

__device__ __forceinline__ float warp_max(float x) {
#pragma unroll
  for (int o = 16; o; o >>= 1) x = fmaxf(x, __shfl_xor_sync(kFull, x, o));
  return x;
}
__device__ __forceinline__ int warp_min_i(int x) {
#pragma unroll
  for (int o = 16; o; o >>= 1) x = min(x, __shfl_xor_sync(kFull, x, o));
  return x;
}
__device__ __forceinline__ int warp_sum_i(int x) {
#pragma unroll
  for (int o = 16; o; o >>= 1) x += __shfl_xor_sync(kFull, x, o);
  return x;
}
// Sum with a fixed tree, broadcast from lane 0 (same bits in every lane).
__device__ __forceinline__ float warp_sum_f(float x) {
#pragma unroll
  for (int o = 16; o; o >>= 1) x += __shfl_down_sync(kFull, x, o);
  return __shfl_sync(kFull, x, 0);
}

struct DRed { float m, s, t2, top2; int idx; };
struct TRed { float m, s; int idx, cnt; };

// Merge per-lane drafter statistics (m, s, t2 relative to m, top2, idx).
__device__ __forceinline__ DRed reduce_d(float m, float s, float t2, float top2, int idx) {
  DRed r;
  r.m = warp_max(m);
  const float ML = r.m * kLog2e;
  const float dd = m * kLog2e - ML;
  const float sc = ex2(dd);
  const float s_ = s * sc;
  const float t_ = sc * fmaf(s, dd, t2);
  r.s = warp_sum_f(s_);
  r.t2 = warp_sum_f(t_);
  r.idx = warp_min_i(m == r.m ? idx : 0x7FFFFFFF);
  r.top2 = warp_max((m == r.m && idx == r.idx) ? top2 : m);
  return r;
}
__device__ __forceinline__ TRed reduce_t(float m, float s, int idx, int cnt) {
  TRed r;
  r.m = warp_max(m);
  const float sc = ex2(m * kLog2e - r.m * kLog2e);
  r.s = warp_sum_f(s * sc);
  r.idx = warp_min_i(m == r.m ? idx : 0x7FFFFFFF);
  r.cnt = warp_sum_i(cnt);
  return r;
}

// ---------------------------------------------------------------------------
// work split
// ---------------------------------------------------------------------------

__device__ __forceinline__ int64_t min_len(int V) {
  const int64_t a = (int64_t)V / 24 + 64;
  return a > 1024 ? a : 1024;
}
__device__ __forceinline__ int eff_warps(int64_t N, int V, int nwarps) {
  int64_t w = N / min_len(V);
  if (w < 1) w = 1;
  if (w > nwarps) w = nwarps;
  return (int)w;
}
__device__ __forceinline__ int64_t split_start(int w, int64_t N, int W, int vec) {
  if (w >= W) return N;
  return ((int64_t)w * N / W) & ~(int64_t)(vec - 1);
}
__device__ __forceinline__ int find_warp(int64_t e, int64_t N, int W, int vec) {
  int w = (int)((e * (int64_t)W) / N);
  if (w >= W) w = W - 1;
  while (w + 1 < W && split_start(w + 1, N, W, vec) <= e) ++w;
  while (w > 0 && split_start(w, N, W, vec) > e) --w;
  return w;
}

__device__ __forceinline__ int k_of(const StreamArgs& a, int b) {
  if (!a.k_row) return a.K;
  int k = __ldg(a.k_row + b);
  return k < 0 ? 0 : (k > a.K ? a.K : k);
}

// active row index -> (b, i); pref = exclusive prefix of k_row in smem
__device__ __forceinline__ void map_row(const StreamArgs& a, const int* pref, int ar, int& b, int& i) {
  if (!a.k_row) {
    b = ar / a.K;
    i = ar - b * a.K;
    return;
  }
  int lo = 0, hi = a.B;              // pref[lo] <= ar < pref[hi]
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (pref[mid] <= ar) lo = mid; else hi = mid;
  }
  b = lo;
  i = ar - pref[lo];
}

template <typename T>
__device__ __forceinline__ int checked_token(const StreamArgs& a, int r) {
  int tok = __ldg(a.tokens + r);
  if (tok < 0 || tok >= a.V) {
    atomicOr(a.ws.err, 1u);
    tok = 0;
  }
  return tok;
}

// ---------------------------------------------------------------------------
// sequence epilogue: first-reject scan, next draft length, output tokens
// ---------------------------------------------------------------------------

template <int MODE, bool SAMPLED>
__device__ void seq_epilogue(const StreamArgs& a, int b, int kb, int lane) {
  const Workspace& W = a.ws;
  const int base = b * a.K;
  int n = kb;
  float csum = 0.f;
  for (int i0 = 0; i0 < kb; i0 += 32) {
    const int i = i0 + lane;
    const bool valid = i < kb;
    int acc = 1;
    float cf = 0.f;
    if (valid) {
      if (MODE != kModeConf) acc = __ldcg(W.row_acc + base + i);
      if (MODE != kModeVerify) cf = __ldcg(W.row_conf + base + i);
    }
    const unsigned rej = __ballot_sync(kFull, valid && !acc);
    if (n == kb && rej) n = i0 + __ffs(rej) - 1;
    csum += cf;
  }
  if (MODE != kModeVerify) {
    csum = warp_sum_f(csum);
    if (lane == 0 && a.k_next) {
      int k = a.k_min;
      if (kb > 0) {
        const float cbar = csum / (float)kb;
        const float x = a.alpha * cbar * (float)a.k_max;
        k = (int)floorf(x);
        k = k < a.k_min ? a.k_min : (k > a.k_max ? a.k_max : k);
      }
      a.k_next[b] = k;
    }
  }
  if (MODE != kModeConf) {
    for (int i = lane; i < a.K; i += 32) {
      int tok = -1;
      if (i < n) {
        tok = __ldg(a.tokens + base + i);
      } else if (i == n && n < kb) {
        tok = SAMPLED ? -1 : __ldcg(W.row_targmax + base + n);
      }
      a.out_tokens[base + i] = tok;
      if (a.accept) a.accept[base + i] = (i < kb) ? (unsigned char)(__ldcg(W.row_acc + base + i) != 0) : 0;
    }
    if (lane == 0) {
      a.n_accept[b] = n;
      if (SAMPLED && n < kb) {
        const int slot = atomicAdd(W.rej_count, 1);
        if (slot < a.B) {
          W.rej_list[slot] = b;
          W.seq_n[b] = n;
        } else {
          atomicOr(W.err, 4u);   // queue not drained by a previous call: workspace misuse
        }
      }
    }
  }
  if (lane == 0) W.seq_done[b] = 0;
}

// ---------------------------------------------------------------------------
// row results from the merged statistics
// ---------------------------------------------------------------------------

template <typename T, int MODE, bool SAMPLED>
__device__ void row_results(const StreamArgs& a, int r, int b, int i, const DRed& d, const TRed& t,
                            float c_tgt) {
  const Workspace& W = a.ws;
  float C = 0.f, MLd = 0.f, Sd = 1.f;
  if (MODE != kModeVerify) {
    MLd = d.m * kLog2e;
    Sd = d.s;
    const float H = kLn2 * (log2f(d.s) - d.t2 / d.s);
    const float margin = (d.top2 <= neg_clamp()) ? __int_as_float(0x7F800000) : d.m - d.top2;
    const float psm = (1.0f - exp2f(fmaf(d.top2, kLog2e, -MLd))) / d.s;
    const float Vf = (float)a.V;
    const float c_ent = 1.0f - H / logf(Vf);
    const float c_mar = 1.0f / (1.0f + expf(-a.beta_sig * margin));
    const float c_soft = psm / (1.0f - 1.0f / Vf);
    C = a.lam0 * c_ent + a.lam1 * c_mar + a.lam2 * c_soft;
    C = fminf(1.0f, fmaxf(0.0f, C));
    if (a.H) a.H[r] = H;
    if (a.margin) a.margin[r] = margin;
    if (a.argmax) a.argmax[r] = d.idx;
    if (a.conf) a.conf[r] = C;
    if (a.lse) a.lse[r] = d.m + kLn2 * log2f(d.s);
  } else {
    C = __ldg(a.conf_in + r);
  }
  W.row_conf[r] = C;
  if (MODE != kModeConf) {
    const float tau = (a.tau_sign >= 0) ? a.tau_base + a.gamma * (1.0f - C)
                                        : a.tau_base + a.gamma * C;
    const bool rank_ok = a.beta_rank <= 0 || t.cnt < a.beta_rank;
    bool acc;
    const float MLt = t.m * kLog2e;
    if (!SAMPLED) {
      const float gap = t.m - c_tgt;
      acc = rank_ok && gap <= tau;
    } else {
      const int tok = checked_token<T>(a, r);
      const float zd = Elem<T>::load((const T*)a.draft + (size_t)r * a.V + tok);
      const float p = exp2f(fmaf(c_tgt, kLog2e, -MLt)) / t.s;
      float q;
      if (MODE == kModeFused) {
        q = exp2f(fmaf(zd, kLog2e, -MLd)) / Sd;
      } else {
        const float lse = __ldg(a.lse_in + r);
        q = expf(zd - lse);
        MLd = lse * kLog2e;
        Sd = 1.0f;
      }
      const U4 w = philox4x32_10(U4{0u, (uint32_t)b, (uint32_t)i, iter_word(a.iteration, kPurposeAccept)},
                                 seed_lo(a.seed), seed_hi(a.seed));
      const float u = word_to_unit(w.x);
      acc = rank_ok && (u * q < expf(tau) * p);
      W.row_dstat[r] = make_float2(MLd, Sd);
      W.row_tstat[r] = make_float2(MLt, t.s);
    }
    W.row_acc[r] = acc ? 1 : 0;
    W.row_targmax[r] = t.idx;
  }
}

// ---------------------------------------------------------------------------
// the streaming kernel
// ---------------------------------------------------------------------------

template <typename T, int MODE, bool SAMPLED>
__global__ void __launch_bounds__(kThreads) stream_kernel(const StreamArgs a) {
  constexpr bool HAS_D = MODE != kModeVerify;
  constexpr bool HAS_T = MODE != kModeConf;
  constexpr int VEC = Elem<T>::kVec;
  using V4 = typename VecT<T>::type;
  extern __shared__ int s_pref[];

  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  const Workspace& W = a.ws;

  // -- present rows: exclusive prefix of k_row (ragged windows) -------------
  int nrows;
  if (a.k_row) {
    // per-thread serial chunks, then a scan over thread totals
    const int per = (a.B + kThreads - 1) / kThreads;
    const int b0 = threadIdx.x * per;
    int tot = 0;
    for (int b = b0; b < b0 + per && b < a.B; ++b) tot += k_of(a, b);
    // block exclusive scan of tot (warp scan + warp totals)
    int incl = tot;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(kFull, incl, o);
      if (lane >= o) incl += y;
    }
    __shared__ int s_wsum[kWarpsPerBlock];
    if (lane == 31) s_wsum[warp] = incl;
    __syncthreads();
    int wofs = 0;
    for (int k = 0; k < warp; ++k) wofs += s_wsum[k];
    int run = wofs + incl - tot;
    for (int b = b0; b < b0 + per && b < a.B; ++b) {
      s_pref[b] = run;
      run += k_of(a, b);
    }
    if (threadIdx.x == kThreads - 1) s_pref[a.B] = run;
    __syncthreads();
    nrows = s_pref[a.B];
  } else {
    nrows = a.B * a.K;
  }

  // -- sequences with no present position, and k_row range errors -----------
  if (a.k_row) {
    const int gt = blockIdx.x * kThreads + threadIdx.x;
    const int gn = gridDim.x * kThreads;
    for (int b = gt; b < a.B; b += gn) {
      const int raw = __ldg(a.k_row + b);
      if (raw < 0 || raw > a.K) atomicOr(W.err, 2u);
      if (k_of(a, b) == 0) {
        if (HAS_D && a.k_next) a.k_next[b] = a.k_min;
        if (HAS_T) {
          a.n_accept[b] = 0;
          for (int i = 0; i < a.K; ++i) {
            a.out_tokens[b * a.K + i] = -1;
            if (a.accept) a.accept[b * a.K + i] = 0;
          }
        }
      }
    }
  }

  const int64_t N = (int64_t)nrows * a.V;
  if (N == 0) return;
  const int Weff = eff_warps(N, a.V, a.nwarps);
  const int w = blockIdx.x * kWarpsPerBlock + warp;
  if (w >= Weff) return;

  int64_t e0 = split_start(w, N, Weff, VEC);
  const int64_t e1 = split_start(w + 1, N, Weff, VEC);
  const int beta = a.beta_rank > 0 ? a.beta_rank : 0;

  while (e0 < e1) {
    const int ar = (int)(e0 / a.V);
    const int v0 = (int)(e0 - (int64_t)ar * a.V);
    const int len = (int)min((int64_t)(a.V - v0), e1 - e0);
    const int v1 = v0 + len;
    int b, i;
    map_row(a, s_pref, ar, b, i);
    const int r = b * a.K + i;
    const size_t rowoff = (size_t)r * (size_t)a.V;
    const T* dp = (const T*)a.draft + rowoff;
    const T* tp = HAS_T ? (const T*)a.target + rowoff : nullptr;

    float c_tgt = 0.f;
    if (HAS_T) c_tgt = Elem<T>::load(tp + checked_token<T>(a, r));

    DLane d;
    TLane t;
    dlane_init(d);
    tlane_init(t);

    const T* ap = HAS_D ? dp : tp;
    const int mis = (int)(((uintptr_t)(ap + v0) & 15) / sizeof(T));
    const int head = mis ? min(VEC - mis, len) : 0;
    const int va = v0 + head;
    const int nvec = (v1 - va) / VEC;
    const int vb = va + nvec * VEC;

    if (lane < head) {
      const int v = v0 + lane;
      if (HAS_D) d_scalar(d, Elem<T>::load(dp + v), v);
      if (HAS_T) t_scalar<SAMPLED>(t, Elem<T>::load(tp + v), v, c_tgt, beta);
    }
    {
      const uint4* dv = reinterpret_cast<const uint4*>(dp + va);
      const uint4* tv = HAS_T ? reinterpret_cast<const uint4*>(tp + va) : nullptr;
      int j = lane;
      constexpr int U = 4;
      for (; j + (U - 1) * 32 < nvec; j += U * 32) {
        uint4 qd[U], qt[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
          if (HAS_D) qd[u] = ld_stream(dv + j + u * 32);
          if (HAS_T) qt[u] = ld_stream(tv + j + u * 32);
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
          const int v = va + (j + u * 32) * VEC;
          if (HAS_D) d_vec(d, as_vec<T>(qd[u]), v);
          if (HAS_T) t_vec<SAMPLED>(t, as_vec<T>(qt[u]), v, c_tgt, beta);
        }
      }
      for (; j < nvec; j += 32) {
        const int v = va + j * VEC;
        if (HAS_D) d_vec(d, as_vec<T>(ld_stream(dv + j)), v);
        if (HAS_T) t_vec<SAMPLED>(t, as_vec<T>(ld_stream(tv + j)), v, c_tgt, beta);
      }
    }
    if (lane < v1 - vb) {
      const int v = vb + lane;
      if (HAS_D) d_scalar(d, Elem<T>::load(dp + v), v);
      if (HAS_T) t_scalar<SAMPLED>(t, Elem<T>::load(tp + v), v, c_tgt, beta);
    }

    // -- segment reduction ------------------------------------------------
    DRed dr{};
    TRed tr{};
    if (HAS_D) {
      float top1 = d.f1, top2 = d.f2;
      if (sizeof(T) == 2) {
        const float a1 = bf_lo(d.T1), a2 = bf_lo(d.T2), b1 = bf_hi(d.T1), b2 = bf_hi(d.T2);
        const float u1 = fmaxf(a1, b1), u2 = fmaxf(fminf(a1, b1), fmaxf(a2, b2));
        top2 = fmaxf(fminf(u1, top1), fmaxf(u2, top2));
        top1 = fmaxf(u1, top1);
      }
      const int idx = d.posw ? first_equal<T>(dp, d.pos, d.posw, d.m, true) : 0x7FFFFFFF;
      dr = reduce_d(d.m, d.s0 + d.s1, d.t0 + d.t1, top2, idx);
    }
    if (HAS_T) {
      const int idx = t.posw ? first_equal<T>(tp, t.pos, t.posw, t.M, false) : 0x7FFFFFFF;
      tr = reduce_t(t.M, t.s0 + t.s1, idx, t.cnt);
    }

    Partial* slot = W.part + ar + w;
    if (lane == 0) {
      Partial p;
      p.d_m = dr.m; p.d_s = dr.s; p.d_t2 = dr.t2; p.d_top2 = dr.top2; p.d_idx = dr.idx;
      p.t_m = tr.m; p.t_s = tr.s; p.t_idx = tr.idx; p.t_cnt = tr.cnt;
      p.pad[0] = p.pad[1] = p.pad[2] = 0;
      *slot = p;
    }
    __threadfence();
    int old = 0;
    if (lane == 0) old = atomicAdd(W.row_done + r, len);
    old = __shfl_sync(kFull, old, 0);

    if (old + len == a.V) {
      // -- this warp completed row r: merge every segment's partial ----------
      __threadfence();
      const int wf = find_warp((int64_t)ar * a.V, N, Weff, VEC);
      const int wl = find_warp((int64_t)ar * a.V + a.V - 1, N, Weff, VEC);
      const int np = wl - wf + 1;      // <= 26 by the minimum slice length
      Partial p;
      if (lane < np) {
        const float4* src = reinterpret_cast<const float4*>(W.part + ar + wf + lane);
        const float4 x0 = __ldcg(src), x1 = __ldcg(src + 1), x2 = __ldcg(src + 2);
        p.d_m = x0.x; p.d_s = x0.y; p.d_t2 = x0.z; p.d_top2 = x0.w;
        p.d_idx = __float_as_int(x1.x); p.t_m = x1.y; p.t_s = x1.z; p.t_idx = __float_as_int(x1.w);
        p.t_cnt = __float_as_int(x2.x);
      } else {
        p.d_m = kNegInit; p.d_s = 0.f; p.d_t2 = 0.f; p.d_top2 = kNegInit; p.d_idx = 0x7FFFFFFF;
        p.t_m = kNegInit; p.t_s = 0.f; p.t_idx = 0x7FFFFFFF; p.t_cnt = 0;
      }
      if (HAS_D) dr = reduce_d(p.d_m, p.d_s, p.d_t2, p.d_top2, p.d_idx);
      if (HAS_T) tr = reduce_t(p.t_m, p.t_s, p.t_idx, p.t_cnt);
      if (lane == 0) {
        W.row_done[r] = 0;
        row_results<T, MODE, SAMPLED>(a, r, b, i, dr, tr, c_tgt);
      }
      __threadfence();
      const int kb = k_of(a, b);
      int sold = 0;
      if (lane == 0) sold = atomicAdd(W.seq_done + b, 1);
      sold = __shfl_sync(kFull, sold, 0);
      if (sold + 1 == kb) {
        __threadfence();
        seq_epilogue<MODE, SAMPLED>(a, b, kb, lane);
      }
    }
    e0 += len;
  }
}

// ---------------------------------------------------------------------------
// residual draw: exponential race over max(0, p - q) at each rejected position
// ---------------------------------------------------------------------------

struct Race {
  float key;
  int idx;
  uint32_t grp;
  U4 words;
};

__device__ __forceinline__ void race_elem(Race& rc, float zt, float zd, int v, float MLt, float invSt,
                                          float MLd, float invSd, uint32_t b, uint32_t n,
                                          uint32_t cw, uint32_t k0, uint32_t k1) {
  const float p = ex2(fmaf(zt, kLog2e, -MLt)) * invSt;
  const float q = ex2(fmaf(zd, kLog2e, -MLd)) * invSd;
  const float rr = p - q;
  if (rr > 0.f) {
    const uint32_t g = (uint32_t)v >> 2;
    if (g != rc.grp) {
      rc.words = philox4x32_10(U4{g, b, n, cw}, k0, k1);
      rc.grp = g;
    }
    const uint32_t sel = (uint32_t)v & 3u;
    const uint32_t word = sel == 0 ? rc.words.x : sel == 1 ? rc.words.y : sel == 2 ? rc.words.z : rc.words.w;
    const float u = word_to_unit(word);
    // E = -log(1 - u) >= u: skip entries that cannot beat the current best
    if (u < rc.key * rr) {
      const float E = -log1pf(-u);
      const float key = E / rr;
      if (key < rc.key) {
        rc.key = key;
        rc.idx = v;
      }
    }
  }
}

template <typename T>
__global__ void __launch_bounds__(kThreads) resample_kernel(const StreamArgs a) {
  constexpr int VEC = Elem<T>::kVec;
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  const Workspace& W = a.ws;
  int R = __ldcg(W.rej_count);
  R = R < 0 ? 0 : (R > a.B ? a.B : R);
  const int64_t N = (int64_t)R * a.V;
  if (N > 0) {
    const int Weff = eff_warps(N, a.V, a.nwarps);
    const int w = blockIdx.x * kWarpsPerBlock + warp;
    if (w < Weff) {
      int64_t e0 = split_start(w, N, Weff, VEC);
      const int64_t e1 = split_start(w + 1, N, Weff, VEC);
      const uint32_t k0 = seed_lo(a.seed), k1 = seed_hi(a.seed);
      const uint32_t cw = iter_word(a.iteration, kPurposeResidual);
      while (e0 < e1) {
        const int rr_ = (int)(e0 / a.V);
        const int v0 = (int)(e0 - (int64_t)rr_ * a.V);
        const int len = (int)min((int64_t)(a.V - v0), e1 - e0);
        const int v1 = v0 + len;
        const int b = __ldcg(W.rej_list + rr_);
        const int n = __ldcg(W.seq_n + b);
        const int r = b * a.K + n;
        const float2 ds = __ldcg(W.row_dstat + r);
        const float2 ts = __ldcg(W.row_tstat + r);
        const float invSd = 1.0f / ds.y, invSt = 1.0f / ts.y;
        const size_t rowoff = (size_t)r * (size_t)a.V;
        const T* dp = (const T*)a.draft + rowoff;
        const T* tp = (const T*)a.target + rowoff;

        Race rc;
        rc.key = __int_as_float(0x7F800000);
        rc.idx = 0x7FFFFFFF;
        rc.grp = 0xFFFFFFFFu;
        rc.words = U4{0, 0, 0, 0};

        const int mis = (int)(((uintptr_t)(tp + v0) & 15) / sizeof(T));
        const int head = mis ? min(VEC - mis, len) : 0;
        const int va = v0 + head;
        const int nvec = (v1 - va) / VEC;
        const int vb = va + nvec * VEC;
        if (lane < head) {
          const int v = v0 + lane;
          race_elem(rc, Elem<T>::load(tp + v), Elem<T>::load(dp + v), v, ts.x, invSt, ds.x, invSd,
                    b, n, cw, k0, k1);
        }
        const uint4* dv = reinterpret_cast<const uint4*>(dp + va);
        const uint4* tv = reinterpret_cast<const uint4*>(tp + va);
        for (int j = lane; j < nvec; j += 32) {
          const uint4 qd = ld_stream(dv + j), qt = ld_stream(tv + j);
          const int v = va + j * VEC;
          if (sizeof(T) == 2) {
            const uint32_t wd[4] = {qd.x, qd.y, qd.z, qd.w};
            const uint32_t wt[4] = {qt.x, qt.y, qt.z, qt.w};
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              race_elem(rc, bf_lo(wt[k]), bf_lo(wd[k]), v + 2 * k, ts.x, invSt, ds.x, invSd, b, n, cw, k0, k1);
              race_elem(rc, bf_hi(wt[k]), bf_hi(wd[k]), v + 2 * k + 1, ts.x, invSt, ds.x, invSd, b, n, cw, k0, k1);
            }
          } else {
            const uint32_t wd[4] = {qd.x, qd.y, qd.z, qd.w};
            const uint32_t wt[4] = {qt.x, qt.y, qt.z, qt.w};
#pragma unroll
            for (int k = 0; k < 4; ++k)
              race_elem(rc, __uint_as_float(wt[k]), __uint_as_float(wd[k]), v + k, ts.x, invSt, ds.x,
                        invSd, b, n, cw, k0, k1);
          }
        }
        if (lane < v1 - vb) {
          const int v = vb + lane;
          race_elem(rc, Elem<T>::load(tp + v), Elem<T>::load(dp + v), v, ts.x, invSt, ds.x, invSd,
                    b, n, cw, k0, k1);
        }
        // warp: smallest key, lowest index among equal keys
        float kmin = rc.key;
#pragma unroll
        for (int o = 16; o; o >>= 1) kmin = fminf(kmin, __shfl_xor_sync(kFull, kmin, o));
        const int imin = warp_min_i(rc.key == kmin ? rc.idx : 0x7FFFFFFF);
        if (lane == 0) W.rpart[rr_ + w] = RacePartial{kmin, imin};
        __threadfence();
        int old = 0;
        if (lane == 0) old = atomicAdd(W.res_done + b, len);
        old = __shfl_sync(kFull, old, 0);
        if (old + len == a.V) {
          __threadfence();
          const int wf = find_warp((int64_t)rr_ * a.V, N, Weff, VEC);
          const int wl = find_warp((int64_t)rr_ * a.V + a.V - 1, N, Weff, VEC);
          float key = __int_as_float(0x7F800000);
          int idx = 0x7FFFFFFF;
          if (lane < wl - wf + 1) {
            const float2 x = __ldcg(reinterpret_cast<const float2*>(W.rpart + rr_ + wf + lane));
            key = x.x;
            idx = __float_as_int(x.y);
          }
          float km = key;
#pragma unroll
          for (int o = 16; o; o >>= 1) km = fminf(km, __shfl_xor_sync(kFull, km, o));
          const int im = warp_min_i(key == km ? idx : 0x7FFFFFFF);
          if (lane == 0) {
            W.res_done[b] = 0;
            a.out_tokens[r] = (im != 0x7FFFFFFF) ? im : __ldcg(W.row_targmax + r);
          }
        }
        e0 += len;
      }
    }
  }
  // the last CTA to finish clears the queue for the next call
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    const int done = atomicAdd(W.res_cta_done, 1);
    if (done == (int)gridDim.x - 1) {
      *W.rej_count = 0;
      *W.res_cta_done = 0;
      __threadfence();
    }
  }
}

template <typename T>
cudaError_t launch_stream_t(int mode, bool sampled, const StreamArgs& a, int grid, size_t smem,
                            cudaStream_t s) {
#define CMSD_L(M, S) stream_kernel<T, M, S><<<grid, kThreads, smem, s>>>(a)
  if (mode == kModeConf) CMSD_L(kModeConf, false);
  else if (mode == kModeVerify) { if (sampled) CMSD_L(kModeVerify, true); else CMSD_L(kModeVerify, false); }
  else { if (sampled) CMSD_L(kModeFused, true); else CMSD_L(kModeFused, false); }
#undef CMSD_L
  return cudaGetLastError();
}

template <typename T>
cudaError_t occupancy_stream_t(int mode, bool sampled, size_t smem, int* nb) {
#define CMSD_O(M, S) cudaOccupancyMaxActiveBlocksPerMultiprocessor(nb, stream_kernel<T, M, S>, kThreads, smem)
  if (mode == kModeConf) return CMSD_O(kModeConf, false);
  if (mode == kModeVerify) return sampled ? CMSD_O(kModeVerify, true) : CMSD_O(kModeVerify, false);
  return sampled ? CMSD_O(kModeFused, true) : CMSD_O(kModeFused, false);
#undef CMSD_O
}

}  // namespace cmsd
