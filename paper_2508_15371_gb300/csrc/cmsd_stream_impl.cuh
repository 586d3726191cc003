// Streaming kernels of the CM-ASD logits pass (sm_103a).
//
// Work split.  The present rows (sequence b, drafted position i < k_row[b])
// are laid end to end into one stream of rows * V logits per tensor, and the
// launched warps (a persistent grid: every SM filled to its occupancy) each
// take an equal contiguous slice of that stream.  A slice crosses at most a
// few row boundaries; each piece of a row it covers is a "segment".
//
// Memory pipeline.  Each warp owns a ring of kStages shared-memory stages; a
// stage holds a 1 KB chunk of the drafter row and the matching 1 KB of the
// target row, filled by bulk copies (cp.async.bulk, TMA) that complete on the
// stage's mbarrier.  Lane 0 keeps kStages chunks in flight ahead of the warp,
// across segment boundaries; the warp reads each landed chunk with 128-bit
// shared loads.  The unaligned head and tail of a segment (fewer than 16
// bytes each) are read directly from global memory.
//
// Per-element work (online softmax, Sec. III.B(1)): with running maximum m,
//   s  = sum e^(z - m)
//   t2 = sum e^(z - m) * (z - m) * log2(e)
// so that the entropy is H = -sum p log p = ln2 * (log2 s - t2 / s); when m
// grows to m', s and t2 are rescaled by e^(m - m') (t2 also shifted by
// s * (m - m') log2 e).  The exponent is evaluated as ex2(z*log2e - m*log2e)
// with the product m*log2e rounded once and shared by every term of the
// row, so that rounding cancels in p = e^(z-m)/s.  Pairs of elements go
// through the packed f32x2 FMA/ADD pipes.  The target row keeps its maximum,
// lowest argmax, the count of logits above the drafted token's (saturating at
// beta_rank) and, for the sampled rule, its own sum of e^(z - m).
//
// Reduction.  At the end of a segment the warp merges its lanes with
// shuffles and writes one Partial.  Per-row and per-sequence arrival
// counters (atomics, no waiting on other warps) elect the warp that completes
// a row to merge its partials into the row's results, and the warp that
// completes a sequence to run the sequence epilogue (first-reject scan, next
// draft length, output tokens).  Every logit is read from HBM once.
//
// -inf logits (masked vocabulary) are clamped to -2^100 before the drafter
// arithmetic so that e^(z-m) * (z-m) is 0, not NaN.
#pragma once
#include <cuda_runtime.h>
#include <stdint.h>

#include "cmsd_device.cuh"
#include "cmsd_internal.h"
#include "cmsd_philox.cuh"

namespace cmsd {

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
//
// Each lane walks its elements in increasing index order and keeps, without
// branches: the exact running maximum and the first vector (or single
// element) in which it was reached; the exact index inside that vector is
// resolved at the end of the segment by the lane(s) holding the segment
// maximum, so the lowest index among equal maxima survives.  The exponent
// reference `ref` of the sums moves only when the maximum has grown more
// than kRefSlack above it (rare), so every term is e^(z - ref) <= e^kRefSlack
// and the final shift to the exact maximum loses no precision.

constexpr float kRefSlack = 4.0f;   // nats

#ifndef CMSD_DRAFT_PACKED
#define CMSD_DRAFT_PACKED 1
#endif
#ifndef CMSD_TARGET_PACKED
#define CMSD_TARGET_PACKED 1
#endif

struct DLane {               // drafter
  float m;                   // exact running max (of clamped logits)
  float ref;                 // exponent reference of s and t
  u64 negrL;                 // -(ref*log2e) in both halves
  u64 s, t;                  // packed (even, odd) sums of e and of e*x, relative to ref
  float f1, f2;              // top-2 of elements taken one at a time (all f32 data)
  uint32_t T1, T2;           // top-2 of bf16 vector elements, per half-word lane
  int pos, posw;             // first unit (start, width) that reached m
};

struct TLane {               // target
  float M;                   // exact running max
  float ref;
  u64 negrL;
  u64 s;                     // packed partial sums of e^(z - ref)
  float thr;                 // PAPER rule: elements above thr may be counted
  int pos, posw;
  int cnt;
};

__device__ __forceinline__ void dlane_init(DLane& d) {
  d.m = kNegInit;
  d.ref = kNegInit;
  d.negrL = dup2(-mlog2e(kNegInit));
  d.s = d.t = 0ull;
  d.f1 = d.f2 = kNegInit;
  d.T1 = d.T2 = kNegInf2;
  d.pos = kIntMax;
  d.posw = 0;
}
__device__ __forceinline__ void tlane_init(TLane& t, float c, int beta) {
  t.M = kNegInit;
  t.ref = kNegInit;
  t.negrL = dup2(-mlog2e(kNegInit));
  t.s = 0ull;
  t.pos = kIntMax;
  t.posw = 0;
  t.cnt = 0;
  t.thr = pos_inf();
  if (beta > 0) t.thr = c;   // c is a pending load: read it only when needed
}

// move the exponent reference up to mx: s *= e^(ref - mx), t likewise
// (shifted by s * (ref - mx) log2e)
__device__ __forceinline__ void d_reref(DLane& d, float mx) {
  const float nrL = mlog2e(mx);
  const float dd = __fsub_rn(-lo32f(d.negrL), nrL);    // (ref_old - ref_new) log2e <= 0
  const u64 sc = dup2(ex2(dd));
  d.t = mul2(sc, fma2(d.s, dup2(dd), d.t));
  d.s = mul2(d.s, sc);
  d.ref = mx;
  d.negrL = dup2(-nrL);
}
__device__ __forceinline__ void t_reref(TLane& t, float mx) {
  const float nrL = mlog2e(mx);
  t.s = mul2(t.s, dup2(ex2(__fsub_rn(-lo32f(t.negrL), nrL))));
  t.ref = mx;
  t.negrL = dup2(-nrL);
}

// accumulate a pair of (clamped) drafter logits given as packed floats
__device__ __forceinline__ void d_acc(DLane& d, u64 z) {
#if CMSD_DRAFT_PACKED
  const u64 x = fma2(z, dup2(kLog2e), d.negrL);
  const u64 e = ex2_2(x);
  d.s = add2(d.s, e);
  d.t = fma2(e, x, d.t);
#else
  const float nr = lo32f(d.negrL);
  const float xa = fmaf(lo32f(z), kLog2e, nr), xb = fmaf(hi32f(z), kLog2e, nr);
  const float ea = ex2(xa), eb = ex2(xb);
  d.s = pack2(lo32f(d.s) + ea, hi32f(d.s) + eb);
  d.t = pack2(fmaf(ea, xa, lo32f(d.t)), fmaf(eb, xb, hi32f(d.t)));
#endif
}
__device__ __forceinline__ void t_acc(TLane& t, u64 z) {
#if CMSD_TARGET_PACKED
  t.s = add2(t.s, ex2_2(fma2(z, dup2(kLog2e), t.negrL)));
#else
  const float nr = lo32f(t.negrL);
  t.s = pack2(lo32f(t.s) + ex2(fmaf(lo32f(z), kLog2e, nr)), hi32f(t.s) + ex2(fmaf(hi32f(z), kLog2e, nr)));
#endif
}

// --- drafter: one element at a time (segment heads/tails) --------------------
__device__ __forceinline__ void d_scalar(DLane& d, float z, int v) {
  z = fmaxf(z, neg_clamp());
  d.f2 = fmaxf(d.f2, fminf(d.f1, z));
  d.f1 = fmaxf(d.f1, z);
  if (z > d.m) { d.pos = v; d.posw = 1; }
  d.m = fmaxf(d.m, z);
  if (z > d.ref + kRefSlack) d_reref(d, z);
  d_acc(d, pack2(z, kNegInit));          // the second half adds e = 0
}

// --- drafter: 8 bf16 ---------------------------------------------------------
__device__ __forceinline__ void d_vec(DLane& d, uint4 q, int v) {
  const uint32_t w[4] = {bmax2(q.x, kNegClamp2), bmax2(q.y, kNegClamp2), bmax2(q.z, kNegClamp2),
                         bmax2(q.w, kNegClamp2)};
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    d.T2 = bmax2(d.T2, bmin2(d.T1, w[k]));
    d.T1 = bmax2(d.T1, w[k]);
  }
  const float mx = fmaxf(bf_lo(d.T1), bf_hi(d.T1));
  const bool up = mx > d.m;
  d.pos = up ? v : d.pos;
  d.posw = up ? 8 : d.posw;
  d.m = fmaxf(d.m, mx);
  if (mx > d.ref + kRefSlack) d_reref(d, mx);
#pragma unroll
  for (int k = 0; k < 4; ++k) d_acc(d, bf2_to_f2(w[k]));
}

// --- drafter: 4 f32 ------------------------------------------------------------
__device__ __forceinline__ void d_vec(DLane& d, float4 q, int v) {
  const float nc = neg_clamp();
  const float z[4] = {fmaxf(q.x, nc), fmaxf(q.y, nc), fmaxf(q.z, nc), fmaxf(q.w, nc)};
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    d.f2 = fmaxf(d.f2, fminf(d.f1, z[k]));
    d.f1 = fmaxf(d.f1, z[k]);
  }
  const bool up = d.f1 > d.m;
  d.pos = up ? v : d.pos;
  d.posw = up ? 4 : d.posw;
  d.m = fmaxf(d.m, d.f1);
  if (d.f1 > d.ref + kRefSlack) d_reref(d, d.f1);
  d_acc(d, pack2(z[0], z[1]));
  d_acc(d, pack2(z[2], z[3]));
}

// --- target -----------------------------------------------------------------------
template <bool SAMPLED>
__device__ __forceinline__ void t_scalar(TLane& t, float z, int v, float c, int beta) {
  if (z > t.M) { t.pos = v; t.posw = 1; }
  t.M = fmaxf(t.M, z);
  if (t.cnt < beta && z > c) ++t.cnt;
  if (SAMPLED) {
    if (z > t.ref + kRefSlack) t_reref(t, z);
    t_acc(t, pack2(z, -pos_inf()));
  }
}

template <bool SAMPLED>
__device__ __forceinline__ void t_vec(TLane& t, uint4 q, int v, float c, int beta) {
  const uint32_t w[4] = {q.x, q.y, q.z, q.w};
  const uint32_t a = bmax2(bmax2(w[0], w[1]), bmax2(w[2], w[3]));
  const float vmax = fmaxf(bf_lo(a), bf_hi(a));
  const bool up = vmax > t.M;
  t.pos = up ? v : t.pos;
  t.posw = up ? 8 : t.posw;
  t.M = fmaxf(t.M, vmax);
  if (vmax > t.thr) {          // PAPER rule, rank gate: count logits above the draft's
#pragma unroll
    for (int k = 0; k < 4; ++k) t.cnt += (bf_lo(w[k]) > c) + (bf_hi(w[k]) > c);
    if (t.cnt >= beta) t.thr = pos_inf();
  }
  if (SAMPLED) {
    if (vmax > t.ref + kRefSlack) t_reref(t, vmax);
#pragma unroll
    for (int k = 0; k < 4; ++k) t_acc(t, bf2_to_f2(w[k]));
  }
}

template <bool SAMPLED>
__device__ __forceinline__ void t_vec(TLane& t, float4 q, int v, float c, int beta) {
  const float z[4] = {q.x, q.y, q.z, q.w};
  const float vmax = fmaxf(fmaxf(z[0], z[1]), fmaxf(z[2], z[3]));
  const bool up = vmax > t.M;
  t.pos = up ? v : t.pos;
  t.posw = up ? 4 : t.posw;
  t.M = fmaxf(t.M, vmax);
  if (vmax > t.thr) {
    t.cnt += (z[0] > c) + (z[1] > c) + (z[2] > c) + (z[3] > c);
    if (t.cnt >= beta) t.thr = pos_inf();
  }
  if (SAMPLED) {
    if (vmax > t.ref + kRefSlack) t_reref(t, vmax);
    t_acc(t, pack2(z[0], z[1]));
    t_acc(t, pack2(z[2], z[3]));
  }
}

// s and t of a drafter lane relative to its exact maximum m
__device__ __forceinline__ void d_final(const DLane& d, float& s, float& t2) {
  const float dd = __fsub_rn(-lo32f(d.negrL), mlog2e(d.m));   // (ref - m) log2e <= 0
  const float sc = ex2(dd);
  const float s0 = lo32f(d.s) + hi32f(d.s);
  s = s0 * sc;
  t2 = sc * fmaf(s0, dd, lo32f(d.t) + hi32f(d.t));
}
__device__ __forceinline__ float t_final(const TLane& t) {
  return (lo32f(t.s) + hi32f(t.s)) * ex2(__fsub_rn(-lo32f(t.negrL), mlog2e(t.M)));
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

// Entry k of a 16-byte vector (k may be a run-time value: selects, no local array).
template <typename T>
__device__ __forceinline__ float logit_at(uint4 q, int k) {
  const int j = sizeof(T) == 2 ? (k >> 1) : k;
  const uint32_t w = j == 0 ? q.x : j == 1 ? q.y : j == 2 ? q.z : q.w;
  if (sizeof(T) == 2) return (k & 1) ? bf_hi(w) : bf_lo(w);
  return __uint_as_float(w);
}

// First index in the unit (start pos, width w) whose value equals m (drafter
// values clamped as in the streaming pass when `clamp`).  A unit of width > 1
// is one aligned 16-byte vector of the row: it is read with a single load
// and searched in registers.
template <typename T>
__device__ __forceinline__ int first_in_vec(uint4 q, float m, bool clamp) {
  const float nc = neg_clamp();
  int k = 0;
#pragma unroll
  for (int j = Elem<T>::kVec - 1; j >= 0; --j) {
    float z = logit_at<T>(q, j);
    if (clamp) z = fmaxf(z, nc);
    k = (z == m) ? j : k;
  }
  return k;
}
template <typename T>
__device__ __forceinline__ int first_equal(const T* row, int pos, int w, float m, bool clamp) {
  if (w <= 1) return pos;
  return pos + first_in_vec<T>(__ldcg(reinterpret_cast<const uint4*>(row + pos)), m, clamp);
}

// ---------------------------------------------------------------------------
// warp reductions (results identical in every lane)
// ---------------------------------------------------------------------------

__device__ __forceinline__ float warp_max(float x) {
#pragma unroll
  for (int o = 16; o; o >>= 1) x = fmaxf(x, __shfl_xor_sync(kFull, x, o));
  return x;
}
__device__ __forceinline__ float warp_min(float x) {
#pragma unroll
  for (int o = 16; o; o >>= 1) x = fminf(x, __shfl_xor_sync(kFull, x, o));
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

__device__ __forceinline__ DRed dred_empty() { return DRed{kNegInit, 0.f, 0.f, kNegInit, kIntMax}; }
__device__ __forceinline__ TRed tred_empty() { return TRed{kNegInit, 0.f, kIntMax, 0}; }

// Merge per-lane drafter statistics (m, s, t2 relative to m, top2, idx).
__device__ __forceinline__ DRed reduce_d(const DRed& x) {
  DRed r;
  r.m = warp_max(x.m);
  const float ML = mlog2e(r.m);
  const float dd = __fsub_rn(mlog2e(x.m), ML);
  const float sc = ex2(dd);
  r.s = warp_sum_f(x.s * sc);
  r.t2 = warp_sum_f(sc * fmaf(x.s, dd, x.t2));
  r.idx = warp_min_i(x.m == r.m ? x.idx : kIntMax);
  r.top2 = warp_max((x.m == r.m && x.idx == r.idx) ? x.top2 : x.m);
  return r;
}
__device__ __forceinline__ TRed reduce_t(const TRed& x) {
  TRed r;
  r.m = warp_max(x.m);
  const float sc = ex2(__fsub_rn(mlog2e(x.m), mlog2e(r.m)));
  r.s = warp_sum_f(x.s * sc);
  r.idx = warp_min_i(x.m == r.m ? x.idx : kIntMax);
  r.cnt = warp_sum_i(x.cnt);
  return r;
}

// Lane-local merge of two partial statistics (used when a row has more
// partials than a warp has lanes).
__device__ __forceinline__ void fold_d(DRed& a, const DRed& b) {
  const float M = fmaxf(a.m, b.m);
  const float ML = mlog2e(M);
  const float da = __fsub_rn(mlog2e(a.m), ML), db = __fsub_rn(mlog2e(b.m), ML);
  const float sa = ex2(da), sb = ex2(db);
  const float t2 = sa * fmaf(a.s, da, a.t2) + sb * fmaf(b.s, db, b.t2);
  const float s = a.s * sa + b.s * sb;
  if (a.m > b.m) {
    a.top2 = fmaxf(a.top2, b.m);
  } else if (b.m > a.m) {
    a.top2 = fmaxf(b.top2, a.m);
    a.idx = b.idx;
  } else {
    a.top2 = a.m;
    a.idx = min(a.idx, b.idx);
  }
  a.m = M;
  a.s = s;
  a.t2 = t2;
}
__device__ __forceinline__ void fold_t(TRed& a, const TRed& b) {
  const float M = fmaxf(a.m, b.m);
  const float ML = mlog2e(M);
  const float s = a.s * ex2(__fsub_rn(mlog2e(a.m), ML)) + b.s * ex2(__fsub_rn(mlog2e(b.m), ML));
  if (b.m > a.m) a.idx = b.idx;
  else if (b.m == a.m) a.idx = min(a.idx, b.idx);
  a.m = M;
  a.s = s;
  a.cnt += b.cnt;
}

// ---------------------------------------------------------------------------
// work split
// ---------------------------------------------------------------------------

__device__ __forceinline__ int eff_warps(int64_t N, int64_t min_len, int nwarps) {
  int64_t w = N / min_len;
  if (w < 1) w = 1;
  if (w > nwarps) w = nwarps;
  return (int)w;
}
__device__ __forceinline__ int64_t stream_min_len(int V) {
  const int64_t a = (int64_t)V / 64 + 64;
  return a > 2048 ? a : 2048;
}
// a / b for 0 <= a, 0 < b, in 32-bit arithmetic when both fit.
__device__ __forceinline__ int64_t div_nn(int64_t a, int64_t b) {
  if (a <= 0x7FFFFFFF && b <= 0x7FFFFFFF) return (int64_t)((uint32_t)a / (uint32_t)b);
  return a / b;
}

// N units over W warps, contiguous and in order: the first rem warps get q+1.
struct EvenSplit {
  int64_t q;
  int rem;
  __device__ EvenSplit(int64_t N, int W) {
    q = div_nn(N, W);
    rem = (int)(N - q * W);
  }
  __device__ int64_t start(int w) const { return (int64_t)w * q + (w < rem ? w : rem); }
  __device__ int owner(int64_t u) const {
    const int64_t big = (q + 1) * rem;
    return u < big ? (int)div_nn(u, q + 1) : rem + (int)div_nn(u - big, q);
  }
};

// How the present-row stream (R rows of V logits, N = R*V elements) is cut
// into warp slices.  When there are at least as many warps as rows, each row
// is cut into wpr pieces of one warp each (no slice crosses a row end, so
// every warp streams one segment); otherwise the stream is cut into W equal
// runs of 16-byte vectors.  Slices start on multiples of VEC elements (the
// last one ends at N).
struct StreamSplit {
  int64_t N;
  int W;          // warps with work
  int V, VEC;
  int wpr;        // > 0: row-aligned split with wpr warps per row
  int qv, rv;     // row-aligned: V / wpr, V % wpr
  int64_t q;      // flat: vectors per warp (the first rem warps one more)
  int rem;
  __device__ StreamSplit(int R, int V_, int vec, int nwarps, int64_t min_len) {
    V = V_;
    VEC = vec;
    N = (int64_t)R * V;
    int64_t want = N / min_len;
    if (want < 1) want = 1;
    const int Wmax = (int)(want < nwarps ? want : nwarps);
    int p = nwarps / R;                              // pieces per row that fit
    const int64_t pm = (int64_t)V / min_len;
    const int pmax = pm > 0 ? (int)pm : 1;
    if (p > pmax) p = pmax;
    if (p >= 1 && (int64_t)p * R * 8 >= (int64_t)Wmax * 7) {   // uses at least 7/8 of the warps
      wpr = p;
      W = p * R;
      qv = V / p;
      rv = V - qv * p;
      q = 0;
      rem = 0;
    } else {
      wpr = 0;
      W = Wmax;
      qv = rv = 0;
      const int64_t nv = N / VEC;
      q = div_nn(nv, W);
      rem = (int)(nv - q * W);
    }
  }
  __device__ int64_t start(int w) const {
    if (w >= W) return N;
    if (wpr > 0) {
      const int row = w / wpr, k = w - row * wpr;
      const int off = k * qv + (k < rv ? k : rv);
      return (int64_t)row * V + (off & ~(VEC - 1));
    }
    return ((int64_t)w * q + (w < rem ? w : rem)) * VEC;
  }
  // warps holding the first and the last element of row ar
  __device__ int first_warp(int ar) const { return wpr > 0 ? ar * wpr : owner_flat((int64_t)ar * V); }
  __device__ int last_warp(int ar) const {
    return wpr > 0 ? ar * wpr + wpr - 1 : owner_flat((int64_t)ar * V + V - 1);
  }
  __device__ int owner_flat(int64_t e) const {
    const int64_t ev = e / VEC;
    const int64_t big = (q + 1) * rem;
    const int w = ev < big ? (int)div_nn(ev, q + 1) : rem + (int)div_nn(ev - big, q);
    return w < W ? w : W - 1;
  }
};

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

// Geometry of one segment: row elements [v0, v1), with the 16-byte aligned
// body [va, vb) (a whole number of vectors) between a head and a tail.
struct Seg {
  int ar, b, i, r;
  int v0, v1, va, vb;
};

template <typename T>
__device__ __forceinline__ Seg make_seg(const StreamArgs& a, const int* pref, int64_t e, int64_t e_end,
                                        const void* base) {
  constexpr int VEC = Elem<T>::kVec;
  Seg s;
  s.ar = (int)(e / a.V);
  s.v0 = (int)(e - (int64_t)s.ar * a.V);
  const int len = (int)min((int64_t)(a.V - s.v0), e_end - e);
  s.v1 = s.v0 + len;
  map_row(a, pref, s.ar, s.b, s.i);
  s.r = s.b * a.K + s.i;
  const uintptr_t addr = (uintptr_t)((const T*)base + (size_t)s.r * (size_t)a.V + s.v0);
  const int mis = (int)((addr & 15) / sizeof(T));
  const int head = mis ? min(VEC - mis, len) : 0;
  s.va = s.v0 + head;
  s.vb = s.va + ((s.v1 - s.va) / VEC) * VEC;
  return s;
}

// ---------------------------------------------------------------------------
// sequence epilogue: first-reject scan, next draft length, output tokens
// ---------------------------------------------------------------------------

template <int MODE, bool SAMPLED>
__device__ void seq_epilogue(const StreamArgs& a, int b, int kb, int lane) {
  const Workspace& W = a.ws;
  const int base = b * a.K;
  if (a.K <= 32) {
    // one position per lane: every value the outputs need is requested at once
    const int i = lane;
    const bool valid = i < kb;
    int acc = 1, tok = -1, tmx = 0;
    float cf = 0.f;
    float2 ts = make_float2(0.f, 1.f), ds = make_float2(0.f, 1.f);
    if (valid) {
      if (MODE != kModeConf) {
        acc = __ldcg(W.row_acc + base + i);
        tok = __ldg(a.tokens + base + i);
        tmx = __ldcg(W.row_targmax + base + i);
        if (SAMPLED) {
          ts = __ldcg(W.row_tstat + base + i);
          ds = __ldcg(W.row_dstat + base + i);
        }
      }
      if (MODE != kModeVerify) cf = __ldcg(W.row_conf + base + i);
    }
    const unsigned rej = __ballot_sync(kFull, valid && !acc);
    const int n = rej ? __ffs(rej) - 1 : kb;
    if (MODE != kModeVerify) {
      const float csum = warp_sum_f(cf);
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
      if (i < a.K) {
        int ot = -1;
        if (i < n) ot = tok;
        else if (i == n && n < kb) ot = SAMPLED ? -1 : tmx;
        a.out_tokens[base + i] = ot;
        if (a.accept) a.accept[base + i] = valid ? (unsigned char)(acc != 0) : 0;
      }
      if (lane == 0) a.n_accept[b] = n;
      if (SAMPLED && i == n && n < kb) {
        const int slot = atomicAdd(W.rej_count, 1);
        if (slot < a.B) {
          RejRec q;
          q.r = base + n; q.b = b; q.n = n;
          q.targmax = tmx;
          q.MLt = ts.x; q.invSt = 1.0f / ts.y;
          q.MLd = ds.x; q.invSd = 1.0f / ds.y;
          W.rej[slot] = q;
        } else {
          atomicOr(W.err, 4u);   // queue not drained by a previous call: workspace misuse
        }
      }
    }
    if (lane == 0) W.seq_done[b] = 0;
    return;
  }
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
          const int r = base + n;
          const float2 ts = __ldcg(W.row_tstat + r);
          const float2 ds = __ldcg(W.row_dstat + r);
          RejRec q;
          q.r = r; q.b = b; q.n = n;
          q.targmax = __ldcg(W.row_targmax + r);
          q.MLt = ts.x; q.invSt = 1.0f / ts.y;
          q.MLd = ds.x; q.invSd = 1.0f / ds.y;
          W.rej[slot] = q;
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
                            float c_tgt, float zd) {
  const Workspace& W = a.ws;
  float C = 0.f, MLd = 0.f, Sd = 1.f;
  if (MODE != kModeVerify) {
    MLd = mlog2e(d.m);
    Sd = d.s;
    const float H = kLn2 * (log2f(d.s) - d.t2 / d.s);
    const float margin = (d.top2 <= neg_clamp()) ? pos_inf() : d.m - d.top2;
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
    const float MLt = mlog2e(t.m);
    if (!SAMPLED) {
      const float gap = t.m - c_tgt;
      acc = rank_ok && gap <= tau;
    } else {
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
//
// Every warp owns one contiguous slice of the stream.  Within each segment
// (the part of one row inside the slice) a lane's 16-byte vectors are those
// with index lane + 32 t, CMSD_UNROLL of each tensor per stage; the loads of
// stage s+1 are issued into registers before stage s is reduced, so every
// lane keeps one stage in flight and no lane waits on another.  A segment's
// unaligned head and tail (under 16 bytes each) are read directly.
// At the end of a segment the warp reduces its lanes and writes one Partial;
// the warp that completes a row merges the row and, when it completes a
// sequence, runs the sequence epilogue.  Warps never wait on each other.

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

#ifndef CMSD_MIN_BLOCKS
#define CMSD_MIN_BLOCKS 1
#endif

// Running state of the segment a warp is reducing.
template <typename T>
struct SegState {
  DLane d;
  TLane t;
  float c;          // target logit at the drafted token
  float zd;         // drafter logit at the drafted token (SAMPLED rule)
};

template <typename T, int MODE, bool SAMPLED>
__device__ __forceinline__ void seg_begin(SegState<T>& ss, float c_tgt, float zd, int beta) {
  dlane_init(ss.d);
  tlane_init(ss.t, c_tgt, beta);
  ss.c = c_tgt;
  ss.zd = zd;
}

// End of a segment (row ar / storage row r / sequence b, position i, len
// logits): warp-reduce, publish the partial, and merge the row / run the
// sequence epilogue if this warp completes them.
template <typename T, int MODE, bool SAMPLED>
__device__ void seg_finish(const StreamArgs& a, SegState<T>& ss, int ar, int r, int b, int i, int len,
                           const StreamSplit& sp, int w, int lane) {
  const T* dp = (const T*)a.draft + (size_t)r * (size_t)a.V;
  const T* tp = (MODE != kModeConf) ? (const T*)a.target + (size_t)r * (size_t)a.V : nullptr;
  constexpr bool HAS_D = MODE != kModeVerify;
  constexpr bool HAS_T = MODE != kModeConf;
  const Workspace& W = a.ws;
  DRed dr = dred_empty();
  TRed tr = tred_empty();
  if (HAS_D) {
    const DLane& d = ss.d;
    float top1 = d.f1, top2 = d.f2;
    if (sizeof(T) == 2) {
      const float a1 = bf_lo(d.T1), a2 = bf_lo(d.T2), b1 = bf_hi(d.T1), b2 = bf_hi(d.T2);
      const float u1 = fmaxf(a1, b1), u2 = fmaxf(fminf(a1, b1), fmaxf(a2, b2));
      top2 = fmaxf(fminf(u1, top1), fmaxf(u2, top2));
      top1 = fmaxf(u1, top1);
    }
    float s, t2;
    d_final(d, s, t2);
    // only lanes holding the segment maximum resolve their exact index
    const float M = warp_max(d.m);
    const int idx = (d.m == M && d.posw) ? first_equal<T>(dp, d.pos, d.posw, d.m, true) : kIntMax;
    dr = reduce_d(DRed{d.m, s, t2, top2, idx});
  }
  if (HAS_T) {
    const TLane& t = ss.t;
    const float M = warp_max(t.M);
    const int idx = (t.M == M && t.posw) ? first_equal<T>(tp, t.pos, t.posw, t.M, false) : kIntMax;
    tr = reduce_t(TRed{t.M, SAMPLED ? t_final(t) : 0.f, idx, t.cnt});
  }
  // lane 0 stores the partial and counts it with a release; the warp that
  // completes the row sees every other slice's partial through the acquire
  // of its own count (extended to the other lanes by __syncwarp)
  int old = 0;
  if (lane == 0) {
    Partial p;
    p.d_m = dr.m; p.d_s = dr.s; p.d_t2 = dr.t2; p.d_top2 = dr.top2; p.d_idx = dr.idx;
    p.t_m = tr.m; p.t_s = tr.s; p.t_idx = tr.idx; p.t_cnt = tr.cnt;
    p.pad[0] = p.pad[1] = p.pad[2] = 0;
    W.part[ar + w] = p;
    old = atom_add_acq_rel(W.row_done + r, len);
  }
  old = __shfl_sync(kFull, old, 0);
  if (old + len != a.V) return;
  // -- this warp completed row r: merge every slice's partial -----------------
  __syncwarp();
  const int wf = sp.first_warp(ar);
  const int wl = sp.last_warp(ar);
  DRed dm = dred_empty();
  TRed tm = tred_empty();
  for (int k = wf + lane; k <= wl; k += 32) {
    const float4* src = reinterpret_cast<const float4*>(W.part + ar + k);
    const float4 x0 = __ldcg(src), x1 = __ldcg(src + 1), x2 = __ldcg(src + 2);
    if (HAS_D) fold_d(dm, DRed{x0.x, x0.y, x0.z, x0.w, __float_as_int(x1.x)});
    if (HAS_T) fold_t(tm, TRed{x1.y, x1.z, __float_as_int(x1.w), __float_as_int(x2.x)});
  }
  if (HAS_D) dr = reduce_d(dm);
  if (HAS_T) tr = reduce_t(tm);
  const int kb = k_of(a, b);
  int sold = 0;
  if (lane == 0) {
    W.row_done[r] = 0;
    row_results<T, MODE, SAMPLED>(a, r, b, i, dr, tr, ss.c, ss.zd);
    sold = atom_add_acq_rel(W.seq_done + b, 1);
  }
  sold = __shfl_sync(kFull, sold, 0);
  if (sold + 1 == kb) {
    __syncwarp();
    seq_epilogue<MODE, SAMPLED>(a, b, kb, lane);
  }
}

// ---- one segment body, pipelined ----------------------------------------------
// The lane's vectors of the aligned body [va, vb) are j = lane + 32 t,
// t = 0, 1, ...; stage s holds t in [s*U, s*U + U) and is loaded (streaming,
// no L1 allocation) while stage s-1 is reduced.
#ifndef CMSD_UNROLL
#define CMSD_UNROLL 2
#endif
template <typename T>
struct Pipe {
  uint4 d[CMSD_UNROLL], t[CMSD_UNROLL];   // the stage in flight
  const uint4* gd;
  const uint4* gt;
  int nt, nst;                            // this lane's vectors; warp-uniform stages
};

// issue the loads of stage 0
template <typename T, int MODE>
__device__ __forceinline__ void pipe_start(Pipe<T>& p, const T* dp, const T* tp, int va, int vb, int lane) {
  constexpr bool HAS_D = MODE != kModeVerify;
  constexpr bool HAS_T = MODE != kModeConf;
  constexpr int VEC = Elem<T>::kVec;
  constexpr int U = CMSD_UNROLL;
  const int nvec = (vb - va) / VEC;
  p.nt = nvec > lane ? (nvec - lane + 31) / 32 : 0;
  p.nst = (nvec + 32 * U - 1) / (32 * U);
  p.gd = reinterpret_cast<const uint4*>(dp + va) + lane;
  p.gt = HAS_T ? reinterpret_cast<const uint4*>(tp + va) + lane : nullptr;
#pragma unroll
  for (int u = 0; u < U; ++u) {
    if (u < p.nt) {
      if (HAS_D) p.d[u] = ld_stream(p.gd + 32 * u);
      if (HAS_T) p.t[u] = ld_stream(p.gt + 32 * u);
    }
  }
}

template <typename T, int MODE, bool SAMPLED>
__device__ __forceinline__ void pipe_run(Pipe<T>& p, SegState<T>& ss, int va, int beta, int lane) {
  constexpr bool HAS_D = MODE != kModeVerify;
  constexpr bool HAS_T = MODE != kModeConf;
  constexpr int VEC = Elem<T>::kVec;
  constexpr int U = CMSD_UNROLL;
  for (int s = 0; s < p.nst; ++s) {
    uint4 nd[U], nx[U];
    const int t1 = (s + 1) * U;
#pragma unroll
    for (int u = 0; u < U; ++u) {
      if (t1 + u < p.nt) {
        if (HAS_D) nd[u] = ld_stream(p.gd + 32 * (t1 + u));
        if (HAS_T) nx[u] = ld_stream(p.gt + 32 * (t1 + u));
      }
    }
    const int t0 = s * U;
#pragma unroll
    for (int u = 0; u < U; ++u) {
      if (t0 + u < p.nt) {
        const int v = va + (lane + 32 * (t0 + u)) * VEC;
        if (HAS_D) d_vec(ss.d, as_vec<T>(p.d[u]), v);
        if (HAS_T) t_vec<SAMPLED>(ss.t, as_vec<T>(p.t[u]), v, ss.c, beta);
      }
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      if (HAS_D) p.d[u] = nd[u];
      if (HAS_T) p.t[u] = nx[u];
    }
  }
}

// ---- a warp's slice, segment by segment ------------------------------------------
// Order of a segment's start: its first stage of logits is requested, then
// the logits at its drafted token (whose index was requested one segment
// earlier), so the slice's first loads are not held up behind the token.
template <typename T, int MODE, bool SAMPLED>
__device__ void walk_slice(const StreamArgs& a, const int* s_pref, int64_t e_begin, int64_t e_end,
                           const StreamSplit& sp, int w, int lane) {
  constexpr bool HAS_D = MODE != kModeVerify;
  constexpr bool HAS_T = MODE != kModeConf;
  const int beta = a.beta_rank > 0 ? a.beta_rank : 0;
  const void* base = HAS_D ? a.draft : a.target;
  int tok_next = 0;
  if (HAS_T) tok_next = __ldg(a.tokens + make_seg<T>(a, s_pref, e_begin, e_end, base).r);
  for (int64_t e0 = e_begin; e0 < e_end;) {
    const Seg sg = make_seg<T>(a, s_pref, e0, e_end, base);
    const int len = sg.v1 - sg.v0;
    e0 += len;
    const size_t rowoff = (size_t)sg.r * (size_t)a.V;
    const T* dp = (const T*)a.draft + rowoff;
    const T* tp = HAS_T ? (const T*)a.target + rowoff : nullptr;
    Pipe<T> pp;
    pipe_start<T, MODE>(pp, dp, tp, sg.va, sg.vb, lane);
    float c = 0.f, zd = 0.f;
    if (HAS_T) {
      int tok = tok_next;
      if (e0 < e_end) tok_next = __ldg(a.tokens + make_seg<T>(a, s_pref, e0, e_end, base).r);
      if (tok < 0 || tok >= a.V) {
        if (lane == 0) atomicOr(a.ws.err, 1u);
        tok = 0;
      }
      c = Elem<T>::load(tp + tok);
      if (SAMPLED) zd = Elem<T>::load(dp + tok);
    }
    SegState<T> ss;
    seg_begin<T, MODE, SAMPLED>(ss, c, zd, beta);
    if (lane < sg.va - sg.v0) {
      const int v = sg.v0 + lane;
      if (HAS_D) d_scalar(ss.d, Elem<T>::load(dp + v), v);
      if (HAS_T) t_scalar<SAMPLED>(ss.t, Elem<T>::load(tp + v), v, ss.c, beta);
    }
    pipe_run<T, MODE, SAMPLED>(pp, ss, sg.va, beta, lane);
    if (lane < sg.v1 - sg.vb) {
      const int v = sg.vb + lane;
      if (HAS_D) d_scalar(ss.d, Elem<T>::load(dp + v), v);
      if (HAS_T) t_scalar<SAMPLED>(ss.t, Elem<T>::load(tp + v), v, ss.c, beta);
    }
    seg_finish<T, MODE, SAMPLED>(a, ss, sg.ar, sg.r, sg.b, sg.i, len, sp, w, lane);
  }
}

template <typename T, int MODE, bool SAMPLED>
__global__ void __launch_bounds__(kStreamThreads, CMSD_MIN_BLOCKS) stream_kernel(const StreamArgs a) {
  constexpr bool HAS_D = MODE != kModeVerify;
  constexpr bool HAS_T = MODE != kModeConf;
  constexpr int VEC = Elem<T>::kVec;
  extern __shared__ __align__(128) unsigned char smem[];
  // the resample kernel (launched as a programmatic dependent) may be
  // scheduled now; it waits for this grid's completion before reading anything
  if (SAMPLED) asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  const Workspace& W = a.ws;
  const bool ragged = a.k_row != nullptr;
  int* s_pref = reinterpret_cast<int*>(smem);

  // -- present rows: exclusive prefix of k_row (ragged windows) -------------
  int nrows;
  if (ragged) {
    const int per = (a.B + kStreamThreads - 1) / kStreamThreads;
    const int b0 = threadIdx.x * per;
    int tot = 0;
    for (int b = b0; b < b0 + per && b < a.B; ++b) tot += k_of(a, b);
    int incl = tot;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(kFull, incl, o);
      if (lane >= o) incl += y;
    }
    __shared__ int s_wsum[kStreamWarps];
    if (lane == 31) s_wsum[warp] = incl;
    __syncthreads();
    int wofs = 0;
    for (int k = 0; k < warp; ++k) wofs += s_wsum[k];
    int run = wofs + incl - tot;
    for (int b = b0; b < b0 + per && b < a.B; ++b) {
      s_pref[b] = run;
      run += k_of(a, b);
    }
    if (threadIdx.x == kStreamThreads - 1) s_pref[a.B] = run;
    __syncthreads();
    nrows = s_pref[a.B];
  } else {
    nrows = a.B * a.K;
  }

  // -- sequences with no present position, and k_row range errors -----------
  if (ragged) {
    const int gt = blockIdx.x * kStreamThreads + threadIdx.x;
    const int gn = gridDim.x * kStreamThreads;
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

  if (nrows == 0) return;
  const StreamSplit sp(nrows, a.V, VEC, a.nwarps, stream_min_len(a.V));
  const int w = blockIdx.x * kStreamWarps + warp;
  if (w >= sp.W) return;
  const int64_t e_begin = sp.start(w);
  const int64_t e_end = sp.start(w + 1);
  if (e_begin >= e_end) return;
  walk_slice<T, MODE, SAMPLED>(a, s_pref, e_begin, e_end, sp, w, lane);
}

// ---------------------------------------------------------------------------
// residual draw at each rejected position: two-level exponential race over
// r_v = max(0, p_v - q_v).  Level 1 races the groups of kGroup consecutive
// entries on their masses R_g = sum of r_v (key E_g / R_g, E_g = -log(1-U_g));
// level 2 races the entries of the winning group (key E_v / r_v).  The group
// wins with probability R_g / R and the entry within it with r_v / R_g, so the
// token has the law r_v / R of the normalised residual.
//
// Work is split over warps in units of (rejected row, group); a warp walks its
// groups GPI at a time, LPG lanes per group with one 16-byte vector each.
// Its best (key, group) goes to a partial slot; the warp that completes a row
// merges the partials and runs level 2 on the winning group (one lane per
// entry).
// ---------------------------------------------------------------------------

#ifndef CMSD_RES_MIN_BLOCKS
#define CMSD_RES_MIN_BLOCKS 3
#endif
constexpr int kGroup = 32;
constexpr int kGroupBatch = 128;       // groups whose E_g one warp draws at once (4 per lane)
constexpr int kResMinGroups = 48;      // fewest groups per warp
constexpr int kResStageBytes = 8192;   // shared-memory stage per warp (both tensors)
constexpr float kRaceFilter = 0.99999f;  // 1 - 1e-5

struct RowStat {
  float MLt, invSt;    // verifier: max*log2e, 1 / sum
  float MLd, ninvSd;   // drafter: max*log2e, -1 / sum
};

// r = max(0, p - q), p = e^(zt - Mt) / St, q = e^(zd - Md) / Sd, with every
// operation rounded on its own (p - q formed as p + (-q), which is the same
// rounding), so that the packed form below gives the same bits per entry.
__device__ __forceinline__ float resid(float zt, float zd, const RowStat& s) {
  const float p = __fmul_rn(ex2(__fmaf_rn(zt, kLog2e, -s.MLt)), s.invSt);
  const float qn = __fmul_rn(ex2(__fmaf_rn(zd, kLog2e, -s.MLd)), s.ninvSd);
  return fmaxf(__fadd_rn(p, qn), 0.f);
}

__device__ __forceinline__ float expo(uint32_t word) { return -log1pf(-word_to_unit(word)); }

// resid() of two entries at once (packed f32x2), accumulated into acc.
__device__ __forceinline__ void resid2(u64& acc, u64 zt, u64 zd, const RowStat& s) {
  const u64 p = mul2(ex2_2(fma2(zt, dup2(kLog2e), dup2(-s.MLt))), dup2(s.invSt));
  const u64 qn = mul2(ex2_2(fma2(zd, dup2(kLog2e), dup2(-s.MLd))), dup2(s.ninvSd));
  const u64 r = add2(p, qn);
  acc = add2(acc, pack2(fmaxf(lo32f(r), 0.f), fmaxf(hi32f(r), 0.f)));
}

// Sum of r over the entries of one 16-byte vector pair.
template <typename T>
__device__ __forceinline__ float resid_vec(uint4 qt, uint4 qd, const RowStat& s) {
  u64 acc = 0ull;
  if (sizeof(T) == 2) {
    resid2(acc, bf2_to_f2(qt.x), bf2_to_f2(qd.x), s);
    resid2(acc, bf2_to_f2(qt.y), bf2_to_f2(qd.y), s);
    resid2(acc, bf2_to_f2(qt.z), bf2_to_f2(qd.z), s);
    resid2(acc, bf2_to_f2(qt.w), bf2_to_f2(qd.w), s);
  } else {
    resid2(acc, pack2(__uint_as_float(qt.x), __uint_as_float(qt.y)),
           pack2(__uint_as_float(qd.x), __uint_as_float(qd.y)), s);
    resid2(acc, pack2(__uint_as_float(qt.z), __uint_as_float(qt.w)),
           pack2(__uint_as_float(qd.z), __uint_as_float(qd.w)), s);
  }
  return lo32f(acc) + hi32f(acc);
}


// 16 bytes of logits at entry v of one row: one vector load when the vector is
// aligned and inside the row, else element loads with entries past the row
// end read as -inf (p = q = 0, so r = 0).
template <typename T>
__device__ __forceinline__ uint4 load_logits(const T* p, int v, int V, bool vec_ok) {
  constexpr int VEC = Elem<T>::kVec;
  if (vec_ok && v + VEC <= V) return ld_stream(p + v);
  uint32_t w[4];
  if (sizeof(T) == 2) {
    const unsigned short* q = reinterpret_cast<const unsigned short*>(p);
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const uint32_t lo = (v + 2 * k < V) ? (uint32_t)__ldg(q + v + 2 * k) : 0xFF80u;
      const uint32_t hi = (v + 2 * k + 1 < V) ? (uint32_t)__ldg(q + v + 2 * k + 1) : 0xFF80u;
      w[k] = lo | (hi << 16);
    }
  } else {
    const uint32_t* q = reinterpret_cast<const uint32_t*>(p);
#pragma unroll
    for (int k = 0; k < 4; ++k) w[k] = (v + k < V) ? __ldg(q + v + k) : 0xFF800000u;
  }
  return make_uint4(w[0], w[1], w[2], w[3]);
}

template <typename T>
__device__ __forceinline__ uint4 neg_inf_vec() {
  return sizeof(T) == 2 ? make_uint4(kNegInf2, kNegInf2, kNegInf2, kNegInf2)
                        : make_uint4(0xFF800000u, 0xFF800000u, 0xFF800000u, 0xFF800000u);
}



// Level 2 on group gm, whose logits sit in lanes own .. own+LPG-1 (vector
// `sub` of the group in lane own+sub): every lane takes one entry, gathers its
// logit pair by shuffles and races E_v / r_v.  Returns the warp's least key
// (lowest entry on ties) as the entry index, or -1 if no entry has r_v > 0.
template <typename T>
__device__ __forceinline__ int race_group_entries(uint4 qt, uint4 qd, int gm, int own, int lane,
                                                  const RowStat& st, uint32_t b, uint32_t n,
                                                  uint32_t cw, uint32_t k0, uint32_t k1) {
  constexpr int VEC = Elem<T>::kVec;
  const int src = own + lane / VEC;
  const int k = lane % VEC;
  const uint32_t t0 = __shfl_sync(kFull, qt.x, src), t1 = __shfl_sync(kFull, qt.y, src);
  const uint32_t t2 = __shfl_sync(kFull, qt.z, src), t3 = __shfl_sync(kFull, qt.w, src);
  const uint32_t d0 = __shfl_sync(kFull, qd.x, src), d1 = __shfl_sync(kFull, qd.y, src);
  const uint32_t d2 = __shfl_sync(kFull, qd.z, src), d3 = __shfl_sync(kFull, qd.w, src);
  const float zt = logit_at<T>(make_uint4(t0, t1, t2, t3), k);
  const float zd = logit_at<T>(make_uint4(d0, d1, d2, d3), k);
  const int v = gm * kGroup + lane;
  const float rv = resid(zt, zd, st);
  const U4 wd = philox4x32_10(U4{(uint32_t)v >> 2, b, n, cw}, k0, k1);
  const uint32_t sel = (uint32_t)v & 3u;
  const uint32_t word = sel == 0 ? wd.x : sel == 1 ? wd.y : sel == 2 ? wd.z : wd.w;
  const float key = rv > 0.f ? expo(word) / rv : pos_inf();
  const float km = warp_min(key);
  const int vm = warp_min_i(key == km ? v : kIntMax);
  return km != pos_inf() ? vm : -1;
}

template <typename T>
__global__ void __launch_bounds__(kThreads, CMSD_RES_MIN_BLOCKS) resample_kernel(const StreamArgs a) {
  constexpr int VEC = Elem<T>::kVec;
  constexpr int LPG = kGroup / VEC;    // lanes per group
  constexpr int GPI = 32 / LPG;        // groups per warp iteration
  constexpr int CG = kResStageBytes / (2 * kGroup * (int)sizeof(T));   // groups per chunk
  extern __shared__ __align__(16) unsigned char res_smem[];
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  const unsigned char* stage = res_smem + warp * kResStageBytes;
  const uint32_t st_t = smem_u32(stage), st_d = st_t + kResStageBytes / 2;
  // everything below reads what the streaming kernel wrote: wait until that
  // grid has completed and its memory is visible
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const Workspace& W = a.ws;
  int R = __ldcg(W.rej_count);
  R = R < 0 ? 0 : (R > a.B ? a.B : R);
  const int ng = (a.V + kGroup - 1) / kGroup;
  const int64_t NU = (int64_t)R * ng;
  if (NU > 0) {
    const int Weff = eff_warps(NU, kResMinGroups, a.nwarps);
    const int w = blockIdx.x * kWarpsPerBlock + warp;
    if (w < Weff) {
      const EvenSplit sp(NU, Weff);
      int64_t u0 = sp.start(w);
      const int64_t u1 = sp.start(w + 1);
      const uint32_t k0 = seed_lo(a.seed), k1 = seed_hi(a.seed);
      const uint32_t cw_grp = iter_word(a.iteration, kPurposeGroup);
      const uint32_t cw_ent = iter_word(a.iteration, kPurposeResidual);
      const int sub = lane % LPG;
      while (u0 < u1) {
        const int rr_ = (int)div_nn(u0, ng);
        const int g0 = (int)(u0 - (int64_t)rr_ * ng);
        const int cnt = (int)min((int64_t)(ng - g0), u1 - u0);
        const int g1 = g0 + cnt;
        const int4 rq0 = __ldcg(reinterpret_cast<const int4*>(W.rej + rr_));
        const float4 rq1 = __ldcg(reinterpret_cast<const float4*>(W.rej + rr_) + 1);
        const int r = rq0.x, b = rq0.y, n = rq0.z;
        const RowStat st{rq1.x, rq1.y, rq1.z, -rq1.w};
        const size_t rowoff = (size_t)r * (size_t)a.V;
        const T* dp = (const T*)a.draft + rowoff;
        const T* tp = (const T*)a.target + rowoff;
        const bool vec_ok = ((((uintptr_t)tp) | ((uintptr_t)dp)) & 15) == 0;

        // level 1, one chunk of CG groups at a time: the chunk's logits are
        // copied to this warp's shared-memory stage in one batch of cp.async
        // (all in flight together), then raced GPI groups per iteration
        float best = pos_inf();              // this lane set's least key
        float thr = pos_inf();               // the warp's least key so far (filter bound)
        int bestg = kIntMax;
        uint4 bqt = neg_inf_vec<T>(), bqd = neg_inf_vec<T>();
        int gb = -kGroupBatch;               // first group of the drawn batch
        uint32_t U0 = 0, U1 = 0, U2 = 0, U3 = 0;
        for (int gc = g0; gc < g1; gc += CG) {
          const int ge = min(g1, gc + CG);
          const int v_base = gc * kGroup;
          // vectors of the chunk lying wholly inside the row (aligned rows only)
          const int nfull = vec_ok ? min((ge - gc) * LPG, (a.V - v_base) / VEC) : 0;
          for (int j = lane; j < nfull; j += 32) {
            cp_async16(st_t + 16u * (uint32_t)j, tp + v_base + j * VEC);
            cp_async16(st_d + 16u * (uint32_t)j, dp + v_base + j * VEC);
          }
          cp_async_commit();
          cp_async_wait<0>();
          __syncwarp();
          for (int gi = gc; gi < ge; gi += GPI) {
            const int g = gi + lane / LPG;
            const int j = (g - gc) * LPG + sub;
            uint4 qt = neg_inf_vec<T>(), qd = neg_inf_vec<T>();
            if (g < ge) {
              if (j < nfull) {
                qt = *reinterpret_cast<const uint4*>(stage + 16 * j);
                qd = *reinterpret_cast<const uint4*>(stage + kResStageBytes / 2 + 16 * j);
              } else {   // ragged row end or unaligned row: element loads, -inf past the end
                qt = load_logits<T>(tp, g * kGroup + sub * VEC, a.V, false);
                qd = load_logits<T>(dp, g * kGroup + sub * VEC, a.V, false);
              }
            }
            if (gi + GPI > gb + kGroupBatch) {   // warp-uniform
              gb = gi & ~3;
              const U4 wds = philox4x32_10(U4{(uint32_t)(gb >> 2) + (uint32_t)lane, (uint32_t)b,
                                              (uint32_t)n, cw_grp}, k0, k1);
              U0 = wds.x; U1 = wds.y; U2 = wds.z; U3 = wds.w;
            }
            float acc = resid_vec<T>(qt, qd, st);
#pragma unroll
            for (int o = 1; o < LPG; o <<= 1) acc += __shfl_xor_sync(kFull, acc, o);
            const int off = min(g - gb, kGroupBatch - 1);
            const int src = off >> 2, sel = off & 3;
            const uint32_t x0 = __shfl_sync(kFull, U0, src), x1 = __shfl_sync(kFull, U1, src);
            const uint32_t x2 = __shfl_sync(kFull, U2, src), x3 = __shfl_sync(kFull, U3, src);
            const uint32_t word = sel == 0 ? x0 : sel == 1 ? x1 : sel == 2 ? x2 : x3;
            // E_g >= U_g, so a group with U_g >= thr * R_g has a key above the
            // warp's best so far and cannot win (the factor keeps the filter
            // safe against the rounding of E and of the product)
            bool improved = false;
            if (g < ge && acc > 0.f && word_to_unit(word) * kRaceFilter < thr * acc) {
              const float key = expo(word) / acc;
              if (key < best) {          // groups are visited in increasing order
                best = key;
                bestg = g;
                bqt = qt;
                bqd = qd;
                improved = true;
              }
            }
            if (__any_sync(kFull, improved)) thr = warp_min(best);
          }
          __syncwarp();                  // the stage is rewritten by the next chunk
        }
        const float kmin = warp_min(best);
        const int gmin = warp_min_i(best == kmin ? bestg : kIntMax);
        // level 2 on this warp's winning group (its lanes are the ones whose
        // best group it is)
        int tok = -1;
        if (gmin != kIntMax) {
          const int own = ((gmin - g0) % GPI) * LPG;
          tok = race_group_entries<T>(bqt, bqd, gmin, own, lane, st, (uint32_t)b, (uint32_t)n,
                                      cw_ent, k0, k1);
        }
        int old = 0;
        if (lane == 0) {
          W.rpart[rr_ + w] = RacePartial{kmin, gmin, tok, 0};
          old = atom_add_acq_rel(W.res_done + rr_, cnt);
        }
        old = __shfl_sync(kFull, old, 0);
        if (old + cnt == ng) {
          __syncwarp();
          const int wf = sp.owner((int64_t)rr_ * ng);
          const int wl = sp.owner((int64_t)rr_ * ng + ng - 1);
          float key = pos_inf();
          int gw = kIntMax, tw = -1;
          for (int k = wf + lane; k <= wl; k += 32) {
            const int4 x = __ldcg(reinterpret_cast<const int4*>(W.rpart + rr_ + k));
            const float xk = __int_as_float(x.x);
            if (xk < key || (xk == key && x.y < gw)) {
              key = xk;
              gw = x.y;
              tw = x.z;
            }
          }
          const float km = warp_min(key);
          const int gm = warp_min_i(key == km ? gw : kIntMax);
          const int tm = warp_min_i((key == km && gw == gm && tw >= 0) ? tw : kIntMax);
          if (lane == 0) {
            W.res_done[rr_] = 0;
            a.out_tokens[r] = (gm != kIntMax && tm != kIntMax) ? tm : rq0.w;   // empty residual: argmax
          }
        }
        u0 += cnt;
      }
    }
  }
  // the last CTA to finish clears the queue for the next call
  __syncthreads();
  if (threadIdx.x == 0) {
    const int done = atom_add_acq_rel(W.res_cta_done, 1);
    if (done == (int)gridDim.x - 1) {
      *W.rej_count = 0;
      *W.res_cta_done = 0;
      __threadfence();
    }
  }
}

constexpr size_t kResSmemBytes = (size_t)kWarpsPerBlock * kResStageBytes;

// Launched as a programmatic dependent of the streaming kernel just before it
// on the same stream: its CTAs may be scheduled as the streaming kernel's CTAs
// retire, and griddepcontrol.wait at its top orders it after that grid.
template <typename T>
cudaError_t launch_resample_t(const StreamArgs& a, int grid, cudaStream_t s) {
  cudaFuncSetAttribute(resample_kernel<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kResSmemBytes);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = kResSmemBytes;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, resample_kernel<T>, a);
}

template <typename T>
cudaError_t occupancy_resample_t(int* nb) {
  cudaFuncSetAttribute(resample_kernel<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kResSmemBytes);
  return cudaOccupancyMaxActiveBlocksPerMultiprocessor(nb, resample_kernel<T>, kThreads, kResSmemBytes);
}

template <typename T>
cudaError_t launch_stream_t(int mode, bool sampled, const StreamArgs& a, int grid, size_t smem,
                            cudaStream_t s) {
#define CMSD_L(M, S)                                                                          \
  do {                                                                                        \
    cudaFuncSetAttribute(stream_kernel<T, M, S>, cudaFuncAttributeMaxDynamicSharedMemorySize, \
                         (int)smem);                                                          \
    stream_kernel<T, M, S><<<grid, kStreamThreads, smem, s>>>(a);                                   \
  } while (0)
  if (mode == kModeConf) CMSD_L(kModeConf, false);
  else if (mode == kModeVerify) { if (sampled) CMSD_L(kModeVerify, true); else CMSD_L(kModeVerify, false); }
  else { if (sampled) CMSD_L(kModeFused, true); else CMSD_L(kModeFused, false); }
#undef CMSD_L
  return cudaGetLastError();
}

template <typename T>
cudaError_t occupancy_stream_t(int mode, bool sampled, size_t smem, int* nb) {
#define CMSD_O(M, S)                                                                            \
  (cudaFuncSetAttribute(stream_kernel<T, M, S>, cudaFuncAttributeMaxDynamicSharedMemorySize,   \
                        (int)smem),                                                            \
   cudaOccupancyMaxActiveBlocksPerMultiprocessor(nb, stream_kernel<T, M, S>, kStreamThreads, smem))
  if (mode == kModeConf) return CMSD_O(kModeConf, false);
  if (mode == kModeVerify) return sampled ? CMSD_O(kModeVerify, true) : CMSD_O(kModeVerify, false);
  return sampled ? CMSD_O(kModeFused, true) : CMSD_O(kModeFused, false);
#undef CMSD_O
}

}  // namespace cmsd
