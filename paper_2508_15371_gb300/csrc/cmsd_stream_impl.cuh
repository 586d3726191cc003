// Streaming kernel of the CM-ASD logits pass (sm_103a).
//
// Work split.  The present rows (sequence b, drafted position i < k_row[b])
// are laid end to end into one stream of rows * V logits per tensor, and the
// launched warps (a persistent grid: one 768-thread CTA per SM) each take one
// contiguous slice of that stream: whole-warp pieces of one row when there are
// at least as many warps as rows, equal runs of 16-byte vectors otherwise.
// Each piece of a row inside a slice is a "segment".
//
// Memory pipeline.  A lane's 16-byte vectors in a segment are those with index
// lane + 32 t; it reads CMSD_UNROLL of each tensor per stage with streaming
// loads (ld.global.nc, no L1 allocation) into registers, and issues the loads
// of stage s + 1 before it reduces stage s, so one stage is always in flight.
// The unaligned head and tail of a segment (under 16 bytes each) are read
// element by element.
//
// Per-element work (online softmax, Sec. III.B(1)): with exponent reference
// ref (a lane's running maximum, moved only when the maximum exceeds it by
// kRefSlack), each term is e = 2^(z log2e - ref log2e) and a lane keeps
//   s  = sum e,   t2 = sum e * (z - ref) log2e
// so that the entropy is H = -sum p log p = ln2 (log2 s - t2 / s) once s and
// t2 are shifted to the exact maximum.  A stage first updates the maxima
// (one reference check per stage), then sums its terms among themselves
// (pairs of elements through the packed f32x2 FMA/ADD pipes) and adds that
// stage sum to the lane's sums with compensated (Kahan) addition: after a
// spike, a lane adds many terms near 1e-6 to a sum near 1, and plain
// addition would lose most of their bits.  The verifier row keeps its maximum,
// lowest argmax, the count of logits above the drafted token's (saturating at
// beta_rank) and, for the sampled rule, its own sum of exponentials.
//
// Reduction.  At the end of a segment the warp merges its lanes with shuffles
// and writes one Partial; per-row and per-sequence counters (acquire-release
// atomics, no waiting) elect the warp that completes a row to merge the row's
// partials and take its decisions, and the warp that
// completes a sequence to run the sequence epilogue: first-reject scan, next
// draft length, output tokens.  For windows of up to 16 positions the
// sequence counter is one 64-bit word that also carries every position's
// accept bit and confidence (fixed point), so the epilogue needs no loads.
//
// Second pass.  Under the sampled rule the rejected position's token is drawn
// from the residual max(0, p - q), and with the bonus row the verifier's extra
// row gives a token when every draft was accepted; both need one more pass
// over one row of the sequence after its epilogue.  The epilogue queues a
// record for each sequence that needs one; a second kernel, launched as a
// programmatic dependent of this one, drains the queue: under the sampled rule
// without the bonus row, resample_bound_kernel (a cluster of CTAs per row that
// bounds each group's residual mass by its largest target logit and races
// only the groups the bound leaves in play); otherwise resample_kernel (the
// queued rows' groups split evenly over its warps, every group raced).  Every
// logit of the pass proper is read once.
//
// -inf logits (masked vocabulary) are clamped to -2^100 before the drafter
// arithmetic so that e^(z-m) * (z-m) is 0, not NaN.
#pragma once
#include <cooperative_groups.h>
#include <map>
#include <mutex>
#include <utility>
#include <cuda_runtime.h>
#include <stdint.h>

#include "cmsd_device.cuh"
#include "cmsd_internal.h"
#include "cmsd_philox.cuh"

namespace cg = cooperative_groups;

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

constexpr int kFixedShift = 36;          // confidence in the sequence word: C * 2^36

// ---------------------------------------------------------------------------
// per-lane running state
// ---------------------------------------------------------------------------
//
// Each lane walks its elements in increasing index order and keeps, without
// branches: the exact running maximum and the first vector (or single
// element) in which it was reached; the exact index inside that vector is
// resolved at the end of the segment, so the lowest index among equal maxima
// survives.  The exponent reference `ref` of the sums moves only when the
// maximum has grown more than kRefSlack above it (rare), so every term is
// e^(z - ref) <= e^kRefSlack and the final shift to the exact maximum loses
// no precision.

constexpr float kRefSlack = 4.0f;   // nats

struct DLane {               // drafter
  float m;                   // exact running max of the raw logits (kNegInit: none yet)
  float ref;                 // exponent reference of s and t
  u64 negrL;                 // -(ref*log2e) in both halves
  float s, cs;               // sum of e, and its compensation (Kahan)
  float t, ct;               // sum of e*x, and its compensation
  float f1, f2;              // top-2 of elements taken one at a time (all f32 data)
  uint32_t T1, T2;           // top-2 of bf16 vector elements, per half-word lane
  int pos, posw;             // first unit (start, width) that reached m
};

struct TLane {               // target
  float M;                   // exact running max
  float ref;
  u64 negrL;
  float s, cs;               // sum of e^(z - ref), and its compensation
  float thr;                 // PAPER rule: elements above thr may be counted
  int pos, posw;
  int cnt;
};

__device__ __forceinline__ void dlane_init(DLane& d) {
  d.m = kNegInit;
  d.ref = kNegInit;
  d.negrL = dup2(-mlog2e(kNegInit));
  d.s = d.cs = d.t = d.ct = 0.f;
  d.f1 = d.f2 = kNegInit;
  d.T1 = d.T2 = kNegInf2;
  d.pos = kIntMax;
  d.posw = 0;
}
__device__ __forceinline__ void tlane_init(TLane& t, float c, int beta) {
  t.M = kNegInit;
  t.ref = kNegInit;
  t.negrL = dup2(-mlog2e(kNegInit));
  t.s = t.cs = 0.f;
  t.pos = kIntMax;
  t.posw = 0;
  t.cnt = 0;
  t.thr = pos_inf();
  if (beta > 0) t.thr = c;   // c is a pending load: read it only when needed
}

// Compensated (Kahan) accumulation s += x; the sum is s - c.
__device__ __forceinline__ void kahan(float& s, float& c, float x) {
  const float y = __fsub_rn(x, c);
  const float u = __fadd_rn(s, y);
  c = __fsub_rn(__fsub_rn(u, s), y);
  s = u;
}

// The drafter's maximum as the exponent arithmetic sees it: masked (-inf)
// logits count as -2^100.
__device__ __forceinline__ float d_mexp(const DLane& d) { return fmaxf(d.m, neg_clamp()); }

// move the exponent reference up to mx: s *= e^(ref - mx), t likewise
// (shifted by s * (ref - mx) log2e); the compensations are folded in
__device__ __forceinline__ void d_reref(DLane& d, float mx) {
  const float nrL = mlog2e(mx);
  const float dd = __fsub_rn(-lo32f(d.negrL), nrL);    // (ref_old - ref_new) log2e <= 0
  const float sc = ex2(dd);
  const float s0 = __fsub_rn(d.s, d.cs), t0 = __fsub_rn(d.t, d.ct);
  d.t = sc * fmaf(s0, dd, t0);
  d.s = s0 * sc;
  d.cs = d.ct = 0.f;
  d.ref = mx;
  d.negrL = dup2(-nrL);
}
__device__ __forceinline__ void t_reref(TLane& t, float mx) {
  const float nrL = mlog2e(mx);
  t.s = __fsub_rn(t.s, t.cs) * ex2(__fsub_rn(-lo32f(t.negrL), nrL));
  t.cs = 0.f;
  t.ref = mx;
  t.negrL = dup2(-nrL);
}

// --- drafter: one element at a time (segment heads/tails) --------------------
__device__ __forceinline__ void d_scalar(DLane& d, float z, int v) {
  d.f2 = fmaxf(d.f2, fminf(d.f1, z));
  d.f1 = fmaxf(d.f1, z);
  if (z > d.m) { d.pos = v; d.posw = 1; }
  d.m = fmaxf(d.m, z);
  const float me = d_mexp(d);
  if (me > d.ref + kRefSlack) d_reref(d, me);
  const float x = fmaf(fmaxf(z, neg_clamp()), kLog2e, lo32f(d.negrL));
  const float e = ex2(x);
  kahan(d.s, d.cs, e);
  kahan(d.t, d.ct, e * x);
}

// --- drafter, maximum phase: top-2 and the first vector of the maximum --------
__device__ __forceinline__ void d_vmax(DLane& d, uint4 q, int v) {
  const uint32_t w[4] = {q.x, q.y, q.z, q.w};
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
}
__device__ __forceinline__ void d_vmax(DLane& d, float4 q, int v) {
  const float z[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    d.f2 = fmaxf(d.f2, fminf(d.f1, z[k]));
    d.f1 = fmaxf(d.f1, z[k]);
  }
  const bool up = d.f1 > d.m;
  d.pos = up ? v : d.pos;
  d.posw = up ? 4 : d.posw;
  d.m = fmaxf(d.m, d.f1);
}

// --- drafter, exponent phase: the vector's terms, summed among themselves ----
__device__ __forceinline__ void d_vexp(const DLane& d, uint4 q, u64& ss, u64& ts) {
  const uint32_t w[4] = {bmax2(q.x, kNegClamp2), bmax2(q.y, kNegClamp2), bmax2(q.z, kNegClamp2),
                         bmax2(q.w, kNegClamp2)};
  const u64 L = dup2(kLog2e);
  const u64 x0 = fma2(bf2_to_f2(w[0]), L, d.negrL), x1 = fma2(bf2_to_f2(w[1]), L, d.negrL);
  const u64 x2 = fma2(bf2_to_f2(w[2]), L, d.negrL), x3 = fma2(bf2_to_f2(w[3]), L, d.negrL);
  const u64 e0 = ex2_2(x0), e1 = ex2_2(x1), e2 = ex2_2(x2), e3 = ex2_2(x3);
  ss = add2(ss, add2(add2(e0, e1), add2(e2, e3)));
  ts = add2(ts, fma2(e3, x3, fma2(e2, x2, fma2(e1, x1, mul2(e0, x0)))));
}
__device__ __forceinline__ void d_vexp(const DLane& d, float4 q, u64& ss, u64& ts) {
  const float nc = neg_clamp();
  const u64 L = dup2(kLog2e);
  const u64 x0 = fma2(pack2(fmaxf(q.x, nc), fmaxf(q.y, nc)), L, d.negrL);
  const u64 x1 = fma2(pack2(fmaxf(q.z, nc), fmaxf(q.w, nc)), L, d.negrL);
  const u64 e0 = ex2_2(x0), e1 = ex2_2(x1);
  ss = add2(ss, add2(e0, e1));
  ts = add2(ts, fma2(e1, x1, mul2(e0, x0)));
}

// --- target -----------------------------------------------------------------------
template <bool SAMPLED>
__device__ __forceinline__ void t_scalar(TLane& t, float z, int v, float c, int beta) {
  if (z > t.M) { t.pos = v; t.posw = 1; }
  t.M = fmaxf(t.M, z);
  if (t.cnt < beta && z > c) ++t.cnt;
  if (SAMPLED) {
    if (t.M > t.ref + kRefSlack) t_reref(t, t.M);
    kahan(t.s, t.cs, ex2(fmaf(z, kLog2e, lo32f(t.negrL))));
  }
}

__device__ __forceinline__ void t_vmax(TLane& t, uint4 q, int v, float c, int beta) {
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
}
__device__ __forceinline__ void t_vmax(TLane& t, float4 q, int v, float c, int beta) {
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
}

__device__ __forceinline__ void t_vexp(const TLane& t, uint4 q, u64& ss) {
  const u64 L = dup2(kLog2e);
  const u64 e0 = ex2_2(fma2(bf2_to_f2(q.x), L, t.negrL)), e1 = ex2_2(fma2(bf2_to_f2(q.y), L, t.negrL));
  const u64 e2 = ex2_2(fma2(bf2_to_f2(q.z), L, t.negrL)), e3 = ex2_2(fma2(bf2_to_f2(q.w), L, t.negrL));
  ss = add2(ss, add2(add2(e0, e1), add2(e2, e3)));
}
__device__ __forceinline__ void t_vexp(const TLane& t, float4 q, u64& ss) {
  const u64 L = dup2(kLog2e);
  const u64 e0 = ex2_2(fma2(pack2(q.x, q.y), L, t.negrL));
  const u64 e1 = ex2_2(fma2(pack2(q.z, q.w), L, t.negrL));
  ss = add2(ss, add2(e0, e1));
}

// s and t of a drafter lane relative to its maximum (as the exponents see it)
__device__ __forceinline__ void d_final(const DLane& d, float& s, float& t2) {
  const float dd = __fsub_rn(-lo32f(d.negrL), mlog2e(d_mexp(d)));   // (ref - m) log2e <= 0
  const float sc = ex2(dd);
  const float s0 = __fsub_rn(d.s, d.cs);
  s = s0 * sc;
  t2 = sc * fmaf(s0, dd, __fsub_rn(d.t, d.ct));
}
__device__ __forceinline__ float t_final(const TLane& t) {
  return __fsub_rn(t.s, t.cs) * ex2(__fsub_rn(-lo32f(t.negrL), mlog2e(t.M)));
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

// First index in a 16-byte vector whose value equals m (drafter values
// clamped as in the streaming pass when `clamp`).
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

// Fewest logits per warp slice: small problems are cut finely (latency), large
// rows into at most about 128 pieces (each piece costs one partial to merge).
// Measured on one-call latencies: 1024 beat 2048 by 2-3 us at B=1 K=4
// V=32000, and 512 or 256 gained nothing more.
__device__ __forceinline__ int64_t stream_min_len(int V) {
  const int64_t a = (int64_t)V / 128 + 64;
  return a > 1024 ? a : 1024;
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
// runs of 128-byte lines.  Slices start on multiples of 128 bytes from the
// row (or stream) start, so that a warp's 512-byte loads cover whole 32-byte
// sectors when the rows themselves are 128-byte aligned; a 16-byte offset
// would make every load touch one sector more (the last slice ends at N).
constexpr int kLineVecs = 8;   // 16-byte vectors per 128-byte line
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
      const int64_t nv = N / (VEC * kLineVecs);
      q = div_nn(nv, W);
      rem = (int)(nv - q * W);
    }
  }
  __device__ int64_t start(int w) const {
    if (w >= W) return N;
    if (wpr > 0) {
      const int row = w / wpr, k = w - row * wpr;
      const int off = k * qv + (k < rv ? k : rv);
      return (int64_t)row * V + (off & ~(VEC * kLineVecs - 1));
    }
    return ((int64_t)w * q + (w < rem ? w : rem)) * VEC * kLineVecs;
  }
  // warps holding the first and the last element of row ar
  __device__ int first_warp(int ar) const { return wpr > 0 ? ar * wpr : owner_flat((int64_t)ar * V); }
  __device__ int last_warp(int ar) const {
    return wpr > 0 ? ar * wpr + wpr - 1 : owner_flat((int64_t)ar * V + V - 1);
  }
  __device__ int owner_flat(int64_t e) const {
    const int64_t ev = e / (VEC * kLineVecs);
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
// r = b*K + i indexes positions (drafter rows, tokens, per-position outputs);
// the verifier row of the position is b*Kt + i.
struct Seg {
  int ar, b, i, r;
  int v0, v1, va, vb;
};

template <typename T>
__device__ __forceinline__ Seg make_seg(const StreamArgs& a, const int* pref, int64_t e, int64_t e_end,
                                        const void* base, bool base_is_target) {
  constexpr int VEC = Elem<T>::kVec;
  Seg s;
  s.ar = (int)(e / a.V);
  s.v0 = (int)(e - (int64_t)s.ar * a.V);
  const int len = (int)min((int64_t)(a.V - s.v0), e_end - e);
  s.v1 = s.v0 + len;
  map_row(a, pref, s.ar, s.b, s.i);
  s.r = s.b * a.K + s.i;
  const size_t row = base_is_target ? (size_t)s.b * a.Kt + s.i : (size_t)s.r;
  const uintptr_t addr = (uintptr_t)((const T*)base + row * (size_t)a.V + s.v0);
  const int mis = (int)((addr & 15) / sizeof(T));
  const int head = mis ? min(VEC - mis, len) : 0;
  s.va = s.v0 + head;
  s.vb = s.va + ((s.v1 - s.va) / VEC) * VEC;
  return s;
}

// ---------------------------------------------------------------------------
// sequence epilogue: first-reject scan, next draft length, output tokens
// ---------------------------------------------------------------------------

// Sec. III.B(b): k = min(k_max, max(k_min, floor(alpha * Cbar * k_max))), with
// Cbar = csum 2^-36 / kb from the window's confidences in fixed point: with
// alpha = ma 2^ea, floor(alpha csum 2^-36 k_max / kb) is formed exactly in
// integer arithmetic.  A constant k when k_fixed > 0 (the fixed-k variants of
// the ablation, Table III).
__device__ __forceinline__ int next_k(const StreamArgs& a, unsigned long long csum, int kb) {
  if (a.k_fixed > 0) return a.k_fixed;
  if (kb <= 0) return a.k_min;
  const uint32_t bits = __float_as_uint(a.alpha);                    // 0 < alpha <= 1, normal
  const int ea = (int)((bits >> 23) & 0xFFu) - 150;                  // alpha = ma 2^ea, ea <= -23
  const unsigned long long t = (unsigned long long)((bits & 0x7FFFFFu) | 0x800000u) *
                               (unsigned long long)a.k_max;           // < 2^35
  const unsigned long long lo = t * csum, hi = __umul64hi(t, csum);
  const int sh = kFixedShift - ea;                                    // >= 59
  const unsigned long long q = sh >= 128 ? 0ull
                             : sh >= 64 ? (hi >> (sh - 64))
                                        : ((lo >> sh) | (hi << (64 - sh)));
  const unsigned long long kk = q / (unsigned long long)kb;
  const int k = kk > (unsigned long long)a.k_max ? a.k_max : (int)kk;
  return k < a.k_min ? a.k_min : k;
}

// The word of sequence b's record that the bounded residual draw polls:
// valid bit | kind << 1 | rejected position << 3.
__device__ __forceinline__ unsigned* rec_word(const Workspace& W, int b) {
  return reinterpret_cast<unsigned*>(W.rec + b) + 3;
}

// Queue the sequence's second-pass record, if it needs one; or, for the
// bounded residual draw, release it (kSeqNone included) at the sequence's own
// slot: one word that the draw polls, written after every other write of the
// epilogue (the caller's warp has synchronised) and, through the row
// counters, of the sequence's rows.
__device__ __forceinline__ void publish(const StreamArgs& a, int b, int kind, int pos) {
  if (a.rec_by_seq) {
    const unsigned w = 1u | ((unsigned)kind << 1) | ((unsigned)pos << 3);
    asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(rec_word(a.ws, b)), "r"(w) : "memory");
    return;
  }
  if (kind == kSeqNone) return;
  const int slot = atomicAdd(a.ws.rec_count, 1);
  if (slot < a.B) a.ws.rec[slot] = make_int4(b, pos, kind, 0);
}

template <int MODE, bool SAMPLED>
__device__ __forceinline__ int seq_kind(const StreamArgs& a, int n, int kb) {
  if (SAMPLED && n < kb) return kSeqResidual;
  if (a.bonus && n == kb) return kSeqBonus;
  return kSeqNone;
}

// One position per lane; write the outputs of sequence b given n, the accept
// bits and the drafted tokens (tok: this lane's position's token).
//   out_tokens: accepted drafts, then at n the correction (PAPER rule: already
//   written by the row merge of position n; sampled rule: -1 until the second
//   pass writes it), -1 after; with the bonus row, slot k_b holds -1 until the
//   second pass writes the verifier's token.
template <int MODE, bool SAMPLED>
__device__ __forceinline__ void write_outputs(const StreamArgs& a, int b, int kb, int n, int i, int tok,
                                              bool acc_i) {
  if (i < a.Ko) {
    const bool mine = (i == n && n < kb && !SAMPLED);
    if (!mine) a.out_tokens[(size_t)b * a.Ko + i] = (i < n) ? tok : -1;
  }
  if (a.accept && i < a.K) a.accept[(size_t)b * a.K + i] = (i < kb && acc_i) ? 1 : 0;
}

// Epilogue of a window of at most 16 positions: everything comes in the
// sequence word (rows merged | accept bits << 6 | sum of C * 2^36 << 22);
// tok is this lane's prefetched drafted token.
template <int MODE, bool SAMPLED, bool PH2>
__device__ __forceinline__ void seq_epilogue_packed(const StreamArgs& a, int b, int kb, unsigned long long word, int tok,
                                    int lane) {
  const unsigned bits = (unsigned)(word >> 6) & 0xFFFFu;
  const unsigned rej = ~bits & ((1u << kb) - 1u);
  const int n = rej ? __ffs(rej) - 1 : kb;
  if (lane == 0) {
    if (MODE != kModeVerify && a.k_next) a.k_next[b] = next_k(a, word >> 22, kb);
    if (MODE != kModeConf) a.n_accept[b] = n;
    a.ws.seq_word[b] = 0ull;
  }
  if (MODE != kModeConf) {
    write_outputs<MODE, SAMPLED>(a, b, kb, n, lane, tok, (bits >> lane) & 1u);
    if (PH2) __syncwarp();                 // the lanes' writes precede lane 0's release
    if (PH2 && lane == 0) publish(a, b, seq_kind<MODE, SAMPLED>(a, n, kb), n);
  }
}

// Epilogue of a longer window: reads the accept bits and confidences of the
// window's positions from the workspace.
template <int MODE, bool SAMPLED, bool PH2>
__device__ __forceinline__ void seq_epilogue_loads(const StreamArgs& a, int b, int kb, int lane) {
  const Workspace& W = a.ws;
  const int base = b * a.K;
  int n = kb;
  unsigned long long csum = 0ull;
  for (int i0 = 0; i0 < kb; i0 += 32) {
    const int i = i0 + lane;
    const bool valid = i < kb;
    int acc = 1;
    unsigned long long cf = 0ull;
    if (valid) {
      if (MODE != kModeConf) acc = __ldcg(W.row_acc + base + i);
      if (MODE != kModeVerify) cf = __ldcg(W.row_conf + base + i);
    }
    const unsigned rej = __ballot_sync(kFull, valid && !acc);
    if (n == kb && rej) n = i0 + __ffs(rej) - 1;
    csum += cf;
  }
  if (MODE != kModeVerify) {
#pragma unroll
    for (int o = 16; o; o >>= 1) csum += __shfl_xor_sync(kFull, csum, o);
    if (lane == 0 && a.k_next) a.k_next[b] = next_k(a, csum, kb);
  }
  if (MODE != kModeConf) {
    for (int i = lane; i < a.Ko; i += 32) {
      const int tok = (i < n) ? __ldg(a.tokens + base + i) : -1;
      const bool acc_i = (i < kb) ? (__ldcg(W.row_acc + base + i) != 0) : false;
      write_outputs<MODE, SAMPLED>(a, b, kb, n, i, tok, acc_i);
    }
    if (lane == 0) a.n_accept[b] = n;
  }
  if (lane == 0) W.seq_done[b] = 0;
  if (MODE != kModeConf && PH2) __syncwarp();   // the lanes' writes precede lane 0's release
  if (MODE != kModeConf && PH2 && lane == 0) publish(a, b, seq_kind<MODE, SAMPLED>(a, n, kb), n);
}

// ---------------------------------------------------------------------------
// row results from the merged statistics (lane 0 of the merging warp)
// ---------------------------------------------------------------------------
//
// All in fp32 (fp64 issues slowly on this part), arranged so that no step
// loses more than a rounding: exponentials take arguments that are exact
// differences of logits, the sums' scale 2^(m log2e - fl(m log2e)) is the
// exact rounding residual of one product, log2 s is split into the exponent
// of s and the log2 of its mantissa, and the confidence is summed with
// error-free transformations into fixed point (C * 2^36).

// log2 s = e + log2(mantissa), mantissa in [1, 2)
__device__ __forceinline__ float log2_split(float s) {
  int e;
  const float m = frexpf(s, &e);      // s = m 2^e, m in [0.5, 1)
  return (float)(e - 1) + log2f(2.0f * m);
}
// 2^(a - b) for floats a, b with a - b in the normal range: the difference
// is formed exactly as hi + lo (TwoSum), then 2^n ex2(hi - n + lo)
__device__ __forceinline__ float exp2_diff(float a, float b) {
  const float nb = -b;
  const float hi = __fadd_rn(a, nb);
  const float z = __fsub_rn(hi, a);
  const float lo = __fadd_rn(__fsub_rn(a, __fsub_rn(hi, z)), __fsub_rn(nb, z));
  const float n = rintf(hi);
  return ldexpf(exp2f(__fadd_rn(__fsub_rn(hi, n), lo)), (int)n);
}

// lambda . c as an unevaluated sum hi + lo (error-free products and sums)
__device__ __forceinline__ void dot3_exact(float l0, float c0, float l1, float c1, float l2, float c2,
                                           float& hi, float& lo) {
  const float p0 = __fmul_rn(l0, c0), p1 = __fmul_rn(l1, c1), p2 = __fmul_rn(l2, c2);
  float err = fmaf(l0, c0, -p0) + fmaf(l1, c1, -p1) + fmaf(l2, c2, -p2);
  float s = __fadd_rn(p0, p1);
  float bb = __fsub_rn(s, p0);
  err += __fadd_rn(__fsub_rn(p0, __fsub_rn(s, bb)), __fsub_rn(p1, bb));
  const float s2 = __fadd_rn(s, p2);
  bb = __fsub_rn(s2, s);
  err += __fadd_rn(__fsub_rn(s, __fsub_rn(s2, bb)), __fsub_rn(p2, bb));
  hi = __fadd_rn(s2, err);
  lo = __fsub_rn(err, __fsub_rn(hi, s2));
}

constexpr float kFixedScale = 68719476736.0f;   // 2^36

// Called by the whole warp (statistics identical in every lane): the row's
// exponentials and reciprocals are spread one per lane, so each costs one
// instruction sequence instead of a chain on one lane.  Lane 0 writes.
template <typename T, int MODE, bool SAMPLED>
__device__ __forceinline__ void row_results(const StreamArgs& a, int r, int b, int i, const DRed& d, const TRed& t,
                                         float c_tgt, float zd, int lane, bool& acc_out,
                                         unsigned long long& cfx_out) {
  constexpr bool HAS_D = MODE != kModeVerify;
  constexpr bool HAS_T = MODE != kModeConf;
  const Workspace& W = a.ws;
  const float MLd0 = HAS_D ? mlog2e(d.m) : 0.f;
  const float MLt = HAS_T ? mlog2e(t.m) : 0.f;
  const float res_m = HAS_D ? fmaf(d.m, kLog2e, -MLd0) : 0.f;   // exact rounding residuals of m log2e
  const float res_t = HAS_T ? fmaf(t.m, kLog2e, -MLt) : 0.f;
  const bool has2 = HAS_D && d.top2 > neg_clamp();
  const float margin = has2 ? d.m - d.top2 : pos_inf();
  const float lse_in = (MODE == kModeVerify && SAMPLED) ? __ldg(a.lse_in + r) : 0.f;
  // one exponential per lane
  float x = 0.f;
  if (lane == 0) x = has2 ? d.top2 - d.m : -pos_inf();        // e^(z(2) - m)
  if (lane == 1) x = -a.beta_sig * margin;                     // sigmoid of the margin
  if (lane == 2) x = c_tgt - t.m;                              // p, unnormalised
  if (lane == 3) x = MODE == kModeVerify ? zd - lse_in : zd - d.m;   // q
  if (lane == 4) x = res_m * kLn2;                             // the sums' scales
  if (lane == 5) x = res_t * kLn2;
  const float ex = expf(x);
  const float e_mar = __shfl_sync(kFull, ex, 1);
  // one reciprocal per lane
  float den = 1.f;
  if (lane == 0 && HAS_D) den = d.s;
  if (lane == 1) den = 1.0f + e_mar;
  if (lane == 2 && HAS_T) den = t.s;
  const float rc = 1.0f / den;
  const float inv_s = __shfl_sync(kFull, rc, 0), c_mar = __shfl_sync(kFull, rc, 1);
  const float inv_st = __shfl_sync(kFull, rc, 2);
  const float e2 = __shfl_sync(kFull, ex, 0), e_p = __shfl_sync(kFull, ex, 2), e_q = __shfl_sync(kFull, ex, 3);
  const float sc_d = __shfl_sync(kFull, ex, 4), sc_t = __shfl_sync(kFull, ex, 5);
  float C = 0.f;
  unsigned long long cfx = 0ull;
  const float qscale = sc_d * inv_s;                            // 2^(res_m) / s
  if (HAS_D) {
    // H = -sum p ln p = ln2 (log2 s - t2 / s)                      (Sec. III.B(1))
    const float l2s = log2_split(d.s);
    const float H = kLn2 * (l2s - d.t2 * inv_s);
    // P(1) - P(2) = (1 - e^(z(2) - m)) / sum e^(z - m)
    const float psm = (1.0f - e2) * qscale;
    const float c_ent = 1.0f - H * a.inv_log_v;
    const float c_soft = psm * a.soft_norm;
    float hi, lo;
    dot3_exact(a.lam0, c_ent, a.lam1, c_mar, a.lam2, c_soft, hi, lo);
    if (hi + lo >= 1.0f) { C = 1.0f; cfx = 1ull << kFixedShift; }
    else if (hi + lo <= 0.0f) { C = 0.0f; cfx = 0ull; }
    else {
      C = hi;
      const long long f = __float2ll_rn(hi * kFixedScale) + __float2ll_rn(lo * kFixedScale);
      cfx = f < 0 ? 0ull : (unsigned long long)f;
    }
    if (lane == 0) {
      if (a.H) a.H[r] = H;
      if (a.margin) a.margin[r] = margin;
      if (a.argmax) a.argmax[r] = d.idx;
      if (a.conf) a.conf[r] = C;
      // ln sum e^z = m + ln2 (log2 s - res_m)
      if (a.lse) a.lse[r] = d.m + kLn2 * (l2s - res_m);
    }
  } else {
    C = __ldg(a.conf_in + r);
    cfx = __float2ull_rn(fminf(1.0f, fmaxf(0.0f, C)) * kFixedScale);
  }
  bool acc = false;
  if (HAS_T) {
    // Sec. III.B(c): tau_t = tau_base + gamma (1 - C_t) (tau_sign = -1: + gamma C_t)
    const float tau = (a.tau_sign >= 0) ? fmaf(a.gamma, 1.0f - C, a.tau_base) : fmaf(a.gamma, C, a.tau_base);
    const bool rank_ok = a.beta_rank <= 0 || t.cnt < a.beta_rank;
    if (!SAMPLED) {
      // gap-bounded acceptance: log P(y1) - log P(draft) = M - z_draft <= tau
      acc = rank_ok && (t.m - c_tgt <= tau);
      if (lane == 0 && !acc) a.out_tokens[(size_t)b * a.Ko + i] = t.idx;   // the correction, if first failure
    } else {
      const float p = e_p * sc_t * inv_st;                      // e^(c - M) / sum e^(z - M)
      const float q = MODE == kModeVerify ? e_q : e_q * qscale;
      const U4 w = philox4x32_10(U4{0u, (uint32_t)b, (uint32_t)i, iter_word(a.iteration, kPurposeAccept)},
                                 seed_lo(a.seed), seed_hi(a.seed));
      acc = rank_ok && (word_to_unit(w.x) * q < expf(tau) * p);
      if (lane == 0) {
        float MLd = MLd0, Sd = d.s;
        if (MODE == kModeVerify) {            // q_v = 2^(z log2e - MLd) / Sd with MLd = lse log2e
          MLd = lse_in * kLog2e;
          Sd = exp2f(fmaf(lse_in, kLog2e, -MLd));
        }
        W.row_dstat[r] = make_float2(MLd, Sd);
        W.row_tstat[r] = make_float2(MLt, t.s);
      }
    }
    if (lane == 0) {
      W.row_acc[r] = acc ? 1 : 0;
      W.row_targmax[r] = t.idx;
    }
  }
  if (lane == 0) W.row_conf[r] = cfx;
  acc_out = acc;
  cfx_out = cfx;
}

// ---------------------------------------------------------------------------
// the streaming pass
// ---------------------------------------------------------------------------

// Running state of the segment a warp is reducing.
struct SegState {
  DLane d;
  TLane t;
  float c;          // target logit at the drafted token
  float zd;         // drafter logit at the drafted token (SAMPLED rule)
};

// End of a segment (row ar, position r = b*K + i, len logits): warp-reduce,
// publish the partial, and merge the row / run the sequence epilogue if this
// warp completes them.
template <typename T, int MODE, bool SAMPLED, bool PH2>
__device__ void seg_finish(const StreamArgs& a, SegState& ss, int ar, int r, int b, int i, int len,
                           const StreamSplit& sp, int w, int lane, const T* dp, const T* tp) {
  constexpr bool HAS_D = MODE != kModeVerify;
  constexpr bool HAS_T = MODE != kModeConf;
  const Workspace& W = a.ws;
  // The exact index of a lane's maximum inside its first 16-byte vector needs
  // that vector again.  Under the sampled rule only the lanes holding the
  // segment maximum request it (one sector each, usually one lane; this saved
  // 19 MB of the 263 MB per launch at B=64 K=8 V=128256 and 2 us).  Under the
  // PAPER rule every lane requests its vector before the warp reductions, so
  // the loads overlap the shuffles: there the kernel's tail is this latency,
  // and the early requests measured 3 us faster than the late ones.
  const float me = HAS_D ? d_mexp(ss.d) : 0.f;
  // Under the sampled rule the exact indices feed only the drafter's argmax
  // output and resample_kernel's empty-residual fallback (the bounded draw
  // finds that argmax itself): without them a lane's vector start stands in
  // (distinct per lane and ordered like the index, so the merges still tell
  // the maximum's lane from a duplicate of its value) and nothing is re-read.
  const bool want_didx = !SAMPLED || a.argmax != nullptr;
  const bool want_tidx = !SAMPLED || !a.rec_by_seq;
  uint4 dq = make_uint4(0, 0, 0, 0), tq = make_uint4(0, 0, 0, 0);
  if (!SAMPLED) {
    if (HAS_D && ss.d.posw > 1) dq = __ldcg(reinterpret_cast<const uint4*>(dp + ss.d.pos));
    if (HAS_T && ss.t.posw > 1) tq = __ldcg(reinterpret_cast<const uint4*>(tp + ss.t.pos));
  }
  const float Md = HAS_D ? warp_max(me) : 0.f;
  const float Mt = HAS_T ? warp_max(ss.t.M) : 0.f;
  const bool dhit = HAS_D && me == Md && ss.d.posw, thit = HAS_T && ss.t.M == Mt && ss.t.posw;
  if (SAMPLED) {
    if (want_didx && dhit && ss.d.posw > 1) dq = __ldcg(reinterpret_cast<const uint4*>(dp + ss.d.pos));
    if (want_tidx && thit && ss.t.posw > 1) tq = __ldcg(reinterpret_cast<const uint4*>(tp + ss.t.pos));
  }
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
    int idx = kIntMax;
    if (dhit) idx = (want_didx && d.posw > 1) ? d.pos + first_in_vec<T>(dq, me, true) : d.pos;
    dr = reduce_d(DRed{me, s, t2, top2, idx});
  }
  if (HAS_T) {
    const TLane& t = ss.t;
    int idx = kIntMax;
    if (thit) idx = (want_tidx && t.posw > 1) ? t.pos + first_in_vec<T>(tq, t.M, false) : t.pos;
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
  const int kb = k_of(a, b);
  const bool packed = a.K <= kPackedMaxK;
  // the drafted tokens of the window, needed if this row completes the sequence
  int tok = -1;
  if (HAS_T && packed && lane < kb) tok = __ldg(a.tokens + b * a.K + lane);
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
  if (packed) {
    unsigned long long word = 0ull;
    bool acc;
    unsigned long long cfx;
    row_results<T, MODE, SAMPLED>(a, r, b, i, dr, tr, ss.c, ss.zd, lane, acc, cfx);
    if (lane == 0) {
      W.row_done[r] = 0;
      const unsigned long long mine = 1ull | ((unsigned long long)(acc ? 1u : 0u) << (6 + i)) | (cfx << 22);
      word = atom_add_acq_rel_u64(W.seq_word + b, mine) + mine;
    }
    word = __shfl_sync(kFull, word, 0);
    if ((int)(word & 63ull) == kb) {
      __syncwarp();
      seq_epilogue_packed<MODE, SAMPLED, PH2>(a, b, kb, word, tok, lane);
    }
  } else {
    int sold = 0;
    bool acc;
    unsigned long long cfx;
    row_results<T, MODE, SAMPLED>(a, r, b, i, dr, tr, ss.c, ss.zd, lane, acc, cfx);
    if (lane == 0) {
      W.row_done[r] = 0;
      sold = atom_add_acq_rel(W.seq_done + b, 1);
    }
    sold = __shfl_sync(kFull, sold, 0);
    if (sold + 1 == kb) {
      __syncwarp();
      seq_epilogue_loads<MODE, SAMPLED, PH2>(a, b, kb, lane);
    }
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
  p.gd = HAS_D ? reinterpret_cast<const uint4*>(dp + va) + lane : nullptr;
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
__device__ __forceinline__ void pipe_run(Pipe<T>& p, SegState& ss, int va, int beta, int lane) {
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
    // maximum phase: running maxima, top-2, rank count
#pragma unroll
    for (int u = 0; u < U; ++u) {
      if (t0 + u < p.nt) {
        const int v = va + (lane + 32 * (t0 + u)) * VEC;
        if (HAS_D) d_vmax(ss.d, as_vec<T>(p.d[u]), v);
        if (HAS_T) t_vmax(ss.t, as_vec<T>(p.t[u]), v, ss.c, beta);
      }
    }
    // one reference check per stage, then the stage's exponentials
    if (HAS_D) {
      const float me = d_mexp(ss.d);
      if (me > ss.d.ref + kRefSlack) d_reref(ss.d, me);
    }
    if (HAS_T && SAMPLED && ss.t.M > ss.t.ref + kRefSlack) t_reref(ss.t, ss.t.M);
    u64 ds = 0ull, dt = 0ull, ts = 0ull;
#pragma unroll
    for (int u = 0; u < U; ++u) {
      if (t0 + u < p.nt) {
        if (HAS_D) d_vexp(ss.d, as_vec<T>(p.d[u]), ds, dt);
        if (HAS_T && SAMPLED) t_vexp(ss.t, as_vec<T>(p.t[u]), ts);
      }
    }
    if (HAS_D) {
      kahan(ss.d.s, ss.d.cs, lo32f(ds) + hi32f(ds));
      kahan(ss.d.t, ss.d.ct, lo32f(dt) + hi32f(dt));
    }
    if (HAS_T && SAMPLED) kahan(ss.t.s, ss.t.cs, lo32f(ts) + hi32f(ts));
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
template <typename T, int MODE, bool SAMPLED, bool PH2>
__device__ void walk_slice(const StreamArgs& a, const int* s_pref, int64_t e_begin, int64_t e_end,
                           const StreamSplit& sp, int w, int lane) {
  constexpr bool HAS_D = MODE != kModeVerify;
  constexpr bool HAS_T = MODE != kModeConf;
  const int beta = a.beta_rank > 0 ? a.beta_rank : 0;
  const void* base = HAS_D ? a.draft : a.target;
  int tok_next = 0;
  if (HAS_T) tok_next = __ldg(a.tokens + make_seg<T>(a, s_pref, e_begin, e_end, base, !HAS_D).r);
  for (int64_t e0 = e_begin; e0 < e_end;) {
    const Seg sg = make_seg<T>(a, s_pref, e0, e_end, base, !HAS_D);
    const int len = sg.v1 - sg.v0;
    e0 += len;
    const T* dp = (const T*)a.draft + (size_t)sg.r * (size_t)a.V;
    const T* tp = HAS_T ? (const T*)a.target + ((size_t)sg.b * a.Kt + sg.i) * (size_t)a.V : nullptr;
    Pipe<T> pp;
    pipe_start<T, MODE>(pp, dp, tp, sg.va, sg.vb, lane);
    float c = 0.f, zd = 0.f;
    if (HAS_T) {
      int tok = tok_next;
      if (e0 < e_end) tok_next = __ldg(a.tokens + make_seg<T>(a, s_pref, e0, e_end, base, !HAS_D).r);
      if (tok < 0 || tok >= a.V) {       // out-of-range draft: clamped, reported
        if (lane == 0) atomicOr(a.ws.err, 1u);
        tok = 0;
      }
      c = Elem<T>::load(tp + tok);
      if (SAMPLED) zd = Elem<T>::load(dp + tok);
    }
    SegState ss;
    dlane_init(ss.d);
    tlane_init(ss.t, c, beta);
    ss.c = c;
    ss.zd = zd;
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
    seg_finish<T, MODE, SAMPLED, PH2>(a, ss, sg.ar, sg.r, sg.b, sg.i, len, sp, w, lane, dp, tp);
  }
}

// ---------------------------------------------------------------------------
// second pass: the residual draw and the bonus token (resample kernel)
// ---------------------------------------------------------------------------
//
// The residual draw at a rejected position is a two-level exponential race
// over r_v = max(0, p_v - q_v).  Level 1 races the groups of kGroup
// consecutive entries on their masses R_g = sum of r_v (key E_g / R_g,
// E_g = -log(1-U_g)); level 2 races the entries of the winning group (key
// E_v / r_v).  The group wins with probability R_g / R and the entry within
// it with r_v / R_g, so the token has the law r_v / R of the normalised
// residual.  The bonus token under the sampled rule is the same race with
// r = p; under the PAPER rule it is the verifier row's argmax.
//
// Work is split over warps in units of (queued row, group); a warp walks its
// groups one shared-memory stage at a time (all of a stage's loads in flight
// together, cp.async), GPI groups per iteration, LPG lanes per group with one
// 16-byte vector each.  A group is raced (logarithm and division) only when
// its uniform passes a bound against the warp's best key so far.  Each warp's
// best (key, group) goes to a partial slot with its level-2 winner; the warp
// that completes a row merges the partials.

// r = max(0, p - q), p = e^(zt - Mt) / St, q = e^(zd - Md) / Sd, with every
// operation rounded on its own (p - q formed as p + (-q)), so that the packed
// form below gives the same bits per entry.
struct RowStat {
  float MLt, invSt;    // verifier: max*log2e, 1 / sum
  float MLd, ninvSd;   // drafter: max*log2e, -1 / sum (0: no drafter term)
};

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
  if (vec_ok && v + VEC <= V) return __ldcg(reinterpret_cast<const uint4*>(p + v));
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
  // keys are >= 0 or +inf: their bits order as unsigned integers
  const float km = __uint_as_float(__reduce_min_sync(kFull, __float_as_uint(key)));
  const int vm = __reduce_min_sync(kFull, key == km ? v : kIntMax);
  return km != pos_inf() ? vm : -1;
}

// Units (queued row rr, group g) -> u = rr * ng + g, split over Weff warps.
// When every queued row can have a warp, each row gets wpr warps of its own:
// no warp's units then cross a row end, which would make it stage, race and
// merge two rows one after the other.  Otherwise the units are split evenly
// in order.
struct ResSplit {
  int R, ng, wpr;
  EvenSplit by_row;   // a row's ng groups over its wpr warps
  EvenSplit flat;     // all units over Weff warps
  __device__ ResSplit(int R_, int ng_, int Weff)
      : R(R_), ng(ng_), wpr(R_ <= Weff ? Weff / R_ : 0), by_row(ng_, wpr > 0 ? wpr : 1),
        flat((int64_t)R_ * ng_, Weff) {}
  __device__ int64_t start(int w) const {
    if (wpr == 0) return flat.start(w);
    if (w >= R * wpr) return (int64_t)R * ng;
    const int rr = w / wpr;
    return (int64_t)rr * ng + by_row.start(w - rr * wpr);
  }
  __device__ int owner(int64_t u) const {
    if (wpr == 0) return flat.owner(u);
    const int rr = (int)div_nn(u, ng);
    return rr * wpr + by_row.owner(u - (int64_t)rr * ng);
  }
};

#ifndef CMSD_RES_MIN_BLOCKS
#define CMSD_RES_MIN_BLOCKS 3
#endif
constexpr int kGroupBatch = 128;       // group uniforms one warp draws at once (4 per lane)
constexpr int kResMinGroups = 8;       // fewest groups per warp (small problems: more, shorter warps)
constexpr int kResStageBytes = 8192;   // shared-memory stage per warp (both tensors)
constexpr float kRaceFilter = 0.99999f;  // 1 - 1e-5
constexpr size_t kResSmemBytes = (size_t)kResWarps * kResStageBytes;

__device__ __forceinline__ uint32_t smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

// The groups [gc, ge) of one row (target, and drafter when `two`) into this
// warp's stage, as a series of cp.async groups of kResSubIters race
// iterations each, all in flight together: the race over the first part of
// the stage starts while the rest is still arriving.  Only vectors wholly
// inside the row go by cp.async (the rest is read element by element);
// returns how many, and the number of cp.async groups committed in nsub.
#ifndef CMSD_RES_SUB_ITERS
#define CMSD_RES_SUB_ITERS 2
#endif
constexpr int kResSubIters = CMSD_RES_SUB_ITERS;
template <typename T>
__device__ __forceinline__ int stage_groups(const T* tp, const T* dp, bool two, int gc, int ge, int V, bool vec_ok,
                                            uint32_t st_t, uint32_t st_d, int lane, int& nsub) {
  constexpr int VEC = Elem<T>::kVec;
  constexpr int LPG = kGroup / VEC;
  constexpr int GPI = 32 / LPG;
  constexpr int SG = kResSubIters * GPI;    // groups per cp.async group
  const int v_base = gc * kGroup;
  const int nfull = vec_ok ? min((ge - gc) * LPG, (V - v_base) / VEC) : 0;
  const int ns = (ge - gc + SG - 1) / SG;
  for (int k = 0; k < ns; ++k) {
#pragma unroll
    for (int m = 0; m < kResSubIters; ++m) {
      const int j = (k * kResSubIters + m) * 32 + lane;    // 32 vectors per race iteration
      if (j < nfull) {
        cp_async16(st_t + 16u * (uint32_t)j, tp + v_base + j * VEC);
        if (two) cp_async16(st_d + 16u * (uint32_t)j, dp + v_base + j * VEC);
      }
    }
    cp_async_commit();
  }
  nsub = ns;
  return nfull;
}

// Wait until at most `pending` of this thread's latest cp.async groups are in
// flight, then make the whole warp's completed copies visible to the warp.
__device__ __forceinline__ void stage_wait(int pending) {
  switch (pending) {
    case 0: asm volatile("cp.async.wait_group 0;" ::: "memory"); break;
    case 1: asm volatile("cp.async.wait_group 1;" ::: "memory"); break;
    case 2: asm volatile("cp.async.wait_group 2;" ::: "memory"); break;
    case 3: asm volatile("cp.async.wait_group 3;" ::: "memory"); break;
    case 4: asm volatile("cp.async.wait_group 4;" ::: "memory"); break;
    case 5: asm volatile("cp.async.wait_group 5;" ::: "memory"); break;
    case 6: asm volatile("cp.async.wait_group 6;" ::: "memory"); break;
    default: asm volatile("cp.async.wait_group 7;" ::: "memory"); break;
  }
  __syncwarp();
}

// Vector `sub` of group g (staged chunk starting at group gc), or -inf
// padding past the row end.
template <typename T>
__device__ __forceinline__ uint4 staged_vec(const unsigned char* stage, const T* row, int g, int gc, int ge, int sub,
                                            int nfull, int V) {
  constexpr int VEC = Elem<T>::kVec;
  constexpr int LPG = kGroup / VEC;
  if (g >= ge) return neg_inf_vec<T>();
  const int j = (g - gc) * LPG + sub;
  if (j < nfull) return *reinterpret_cast<const uint4*>(stage + 16 * j);
  return load_logits<T>(row, g * kGroup + sub * VEC, V, false);
}

template <typename T, bool SAMPLED>
__global__ void __launch_bounds__(kResThreads, CMSD_RES_MIN_BLOCKS) resample_kernel(const StreamArgs a) {
  constexpr int VEC = Elem<T>::kVec;
  constexpr int LPG = kGroup / VEC;    // lanes per group
  constexpr int GPI = 32 / LPG;        // groups per warp iteration
  constexpr int CG = kResStageBytes / (2 * kGroup * (int)sizeof(T));   // groups per stage
  static_assert(CG / (kResSubIters * GPI) <= 8, "stage_wait covers at most 8 cp.async groups");
  constexpr int SG = kResSubIters * GPI;            // groups per sub-stage of the sampled race's ring
  constexpr int SV = kResSubIters * 32;             // 16-byte vectors per sub-stage and tensor
  constexpr int NSLOT = CG / SG;                    // sub-stages in the ring
  static_assert(NSLOT >= 2 && NSLOT * SV * 16 == kResStageBytes / 2, "ring layout");
  extern __shared__ __align__(16) unsigned char res_smem[];
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  const unsigned char* stage = res_smem + warp * kResStageBytes;
  const uint32_t st_t = smem_u32(stage), st_d = st_t + kResStageBytes / 2;
  // everything below reads what the streaming kernel wrote: wait until that
  // grid has completed and its memory is visible
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const Workspace& W = a.ws;
  int R = __ldcg(W.rec_count);
  R = R < 0 ? 0 : (R > a.B ? a.B : R);
  const int ng = (a.V + kGroup - 1) / kGroup;
  const int64_t NU = (int64_t)R * ng;
  if (NU > 0) {
    int64_t want = NU / kResMinGroups;
    const int Weff = (int)(want < 1 ? 1 : (want > a.nwarps ? a.nwarps : want));
    const int w = blockIdx.x * kResWarps + warp;
    if (w < Weff) {
      const ResSplit sp(R, ng, Weff);
      int64_t u0 = sp.start(w);
      const int64_t u1 = sp.start(w + 1);
      const uint32_t k0 = seed_lo(a.seed), k1 = seed_hi(a.seed);
      const uint32_t cw_grp = iter_word(a.iteration, kPurposeGroup);
      const uint32_t cw_ent = iter_word(a.iteration, kPurposeResidual);
      const int sub = lane % LPG;
      while (u0 < u1) {
        const int rr = (int)div_nn(u0, ng);
        const int g0 = (int)(u0 - (int64_t)rr * ng);
        const int cnt = (int)min((int64_t)(ng - g0), u1 - u0);
        const int g1 = g0 + cnt;
        const int4 rec = __ldcg(W.rec + rr);
        const int b = rec.x, pos = rec.y, kind = rec.z;
        const int r = b * a.K + pos;                                   // position (stats)
        const T* tp = (const T*)a.target + ((size_t)b * a.Kt + pos) * (size_t)a.V;
        const bool resid_kind = SAMPLED && kind == kSeqResidual;
        const T* dp = resid_kind ? (const T*)a.draft + (size_t)r * (size_t)a.V : tp;
        const bool vec_ok = ((((uintptr_t)tp) | ((uintptr_t)dp)) & 15) == 0;
        float2 ts = make_float2(0.f, 1.f), ds = make_float2(0.f, 1.f);
        if (resid_kind) {
          ts = __ldcg(W.row_tstat + r);
          ds = __ldcg(W.row_dstat + r);
        }
        UnitResult res;
        res.key = pos_inf();
        res.ref = 0.f;
        res.grp = kIntMax;
        res.tok = -1;
        if (!SAMPLED) {
          // PAPER rule, bonus row: the warp's largest logit (lowest index); key = -max
          float best = -pos_inf();
          int bi = kIntMax;
          for (int gc = g0; gc < g1; gc += CG) {
            const int ge = min(g1, gc + CG);
            int nsub = 0;
            const int nfull = stage_groups<T>(tp, dp, false, gc, ge, a.V, vec_ok, st_t, st_d, lane, nsub);
            for (int gi = gc; gi < ge; gi += GPI) {
              const int itr = (gi - gc) / GPI;
              if (itr % kResSubIters == 0) stage_wait(nsub - 1 - itr / kResSubIters);
              const int g = gi + lane / LPG;
              const uint4 qt = staged_vec<T>(stage, tp, g, gc, ge, sub, nfull, a.V);
              const int v = g * kGroup + sub * VEC;
#pragma unroll
              for (int k = 0; k < VEC; ++k) {
                const float z = logit_at<T>(qt, k);
                if (z > best) { best = z; bi = v + k; }
              }
            }
            __syncwarp();
          }
          const float mx = warp_max(best);
          const int im = warp_min_i(best == mx ? bi : kIntMax);
          if (mx != -pos_inf()) {
            res.key = -mx;
            res.grp = im;
            res.tok = im;
          }
        } else {
          RowStat st{0.f, 1.0f, 0.f, 0.f};   // the residual's is formed once the first stage is in
          if (!resid_kind) {
            // bonus race over p: terms relative to the warp's largest logit (a first pass)
            float mx = -pos_inf();
            for (int v = g0 * kGroup + lane * VEC; v < g1 * kGroup && v < a.V; v += 32 * VEC) {
              const uint4 q = load_logits<T>(tp, v, a.V, vec_ok);
#pragma unroll
              for (int k = 0; k < VEC; ++k) mx = fmaxf(mx, logit_at<T>(q, k));
            }
            mx = warp_max(mx);
            res.ref = mx == -pos_inf() ? 0.f : mlog2e(mx);
            st = RowStat{res.ref, 1.0f, 0.f, 0.f};
          }
          float best = pos_inf();              // this lane set's least key
          float thr = pos_inf();               // the warp's least key so far (filter bound)
          int bestg = kIntMax;
          uint4 bqt = neg_inf_vec<T>(), bqd = make_uint4(0, 0, 0, 0);
          int gb = -kGroupBatch;               // first group of the drawn batch
          U4 gw = U4{0u, 0u, 0u, 0u};
          // The groups [g0, g1) stream through the warp's stage as a ring of
          // NSLOT sub-stages of SG groups: sub-stage s + NSLOT - 1 is copied
          // while sub-stage s is raced.  Vector jr of the range (jr = 32 *
          // race iteration + lane) is copied and read by lane jr % 32 alone,
          // so each lane waits only for its own copies.
          const int S = (g1 - g0 + SG - 1) / SG;
          const int vb = g0 * kGroup;
          const int jfull = vec_ok ? min((g1 - g0) * LPG, (a.V - vb) / VEC) : 0;
          auto issue = [&](int sidx) {
            if (sidx < S) {
              const uint32_t sb = 16u * (uint32_t)((sidx % NSLOT) * SV + lane);
#pragma unroll
              for (int m = 0; m < kResSubIters; ++m) {
                const int jr = (sidx * kResSubIters + m) * 32 + lane;
                if (jr < jfull) {
                  cp_async16(st_t + sb + 512u * (uint32_t)m, tp + vb + jr * VEC);
                  if (resid_kind) cp_async16(st_d + sb + 512u * (uint32_t)m, dp + vb + jr * VEC);
                }
              }
            }
            cp_async_commit();              // one group per sub-stage, empty past the range
          };
#pragma unroll
          for (int sidx = 0; sidx < NSLOT - 1; ++sidx) issue(sidx);
          if (resid_kind) st = RowStat{ts.x, 1.0f / ts.y, ds.x, -1.0f / ds.y};
          for (int sidx = 0; sidx < S; ++sidx) {
            issue(sidx + NSLOT - 1);        // into the slot raced one sub-stage ago
            cp_async_wait<NSLOT - 1>();     // this lane's copies of sub-stage sidx are in
            const unsigned char* slot = stage + 16 * ((sidx % NSLOT) * SV + lane);
#pragma unroll
            for (int m = 0; m < kResSubIters; ++m) {
              const int gi = g0 + (sidx * kResSubIters + m) * GPI;
              if (gi >= g1) break;
              const int g = gi + lane / LPG;
              const int jr = (sidx * kResSubIters + m) * 32 + lane;
              uint4 qt = neg_inf_vec<T>(), qd = make_uint4(0, 0, 0, 0);
              if (resid_kind) qd = neg_inf_vec<T>();
              if (g < g1) {
                if (jr < jfull) {
                  qt = *reinterpret_cast<const uint4*>(slot + 512 * m);
                  if (resid_kind) qd = *reinterpret_cast<const uint4*>(slot + 512 * m + kResStageBytes / 2);
                } else {
                  qt = load_logits<T>(tp, vb + jr * VEC, a.V, false);
                  if (resid_kind) qd = load_logits<T>(dp, vb + jr * VEC, a.V, false);
                }
              }
              if (gi + GPI > gb + kGroupBatch) {   // warp-uniform: draw the next 128 group uniforms
                gb = gi & ~3;
                gw = philox4x32_10(U4{(uint32_t)(gb >> 2) + (uint32_t)lane, (uint32_t)b, (uint32_t)pos, cw_grp},
                                   k0, k1);
              }
              float acc = resid_vec<T>(qt, qd, st);
#pragma unroll
              for (int o = 1; o < LPG; o <<= 1) acc += __shfl_xor_sync(kFull, acc, o);
              const int off = min(g - gb, kGroupBatch - 1);
              const int src = off >> 2, sel = off & 3;
              const uint32_t x0 = __shfl_sync(kFull, gw.x, src), x1 = __shfl_sync(kFull, gw.y, src);
              const uint32_t x2 = __shfl_sync(kFull, gw.z, src), x3 = __shfl_sync(kFull, gw.w, src);
              const uint32_t word = sel == 0 ? x0 : sel == 1 ? x1 : sel == 2 ? x2 : x3;
              // E_g >= U_g, so a group with U_g >= thr R_g has a key above the
              // warp's best so far and cannot win (the factor covers the
              // rounding of E and of the product)
              bool improved = false;
              if (g < g1 && acc > 0.f && word_to_unit(word) * kRaceFilter < thr * acc) {
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
          }
          const float kmin = warp_min(best);
          const int gmin = warp_min_i(best == kmin ? bestg : kIntMax);
          if (kmin != pos_inf()) {
            // level 2 on this warp's winning group (its lanes hold it as their best)
            const int own = ((gmin - g0) % GPI) * LPG;
            res.tok = race_group_entries<T>(bqt, bqd, gmin, own, lane, st, (uint32_t)b, (uint32_t)pos, cw_ent,
                                            k0, k1);
            res.key = kmin;
            res.grp = gmin;
          }
        }
        int old = 0;
        if (lane == 0) {
          W.rpart[rr + w] = res;
          old = atom_add_acq_rel(W.res_done + rr, cnt);
        }
        old = __shfl_sync(kFull, old, 0);
        if (old + cnt == ng) {
          // this warp completed row rr: merge the partials of the warps that covered it
          __syncwarp();
          const int wf = sp.owner((int64_t)rr * ng);
          const int wl = sp.owner((int64_t)rr * ng + ng - 1);
          const bool bonus_race = SAMPLED && kind == kSeqBonus;
          float rmax = -pos_inf();
          if (bonus_race) {
            for (int k = wf + lane; k <= wl; k += 32) rmax = fmaxf(rmax, __ldcg(&W.rpart[rr + k].ref));
            rmax = warp_max(rmax);
          }
          float key = pos_inf();
          int gw_ = kIntMax, tw = -1;
          for (int k = wf + lane; k <= wl; k += 32) {
            const int4 x = __ldcg(reinterpret_cast<const int4*>(W.rpart + rr + k));
            float xk = __int_as_float(x.x);
            // bonus race: a warp's key is relative to its own reference: key * 2^(rmax - ref)
            if (bonus_race && xk != pos_inf()) xk *= exp2_diff(rmax, __int_as_float(x.y));
            if (xk < key || (xk == key && x.z < gw_)) {
              key = xk;
              gw_ = x.z;
              tw = x.w;
            }
          }
          const float km = warp_min(key);
          const int gm = warp_min_i(key == km ? gw_ : kIntMax);
          const int tm = warp_min_i((key == km && gw_ == gm && tw >= 0) ? tw : kIntMax);
          if (lane == 0) {
            W.res_done[rr] = 0;
            int out = tm;
            if (gm == kIntMax || tm == kIntMax) out = __ldcg(W.row_targmax + r);   // empty residual: argmax
            a.out_tokens[(size_t)b * a.Ko + pos] = out;
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
      *W.rec_count = 0;
      *W.res_cta_done = 0;
      __threadfence();
    }
  }
}

// ---------------------------------------------------------------------------
// residual draw by group bounds (sampled rule, no bonus row)
// ---------------------------------------------------------------------------
//
// The same two-level race, with the same keys, reading far less.  Since
// r_v = max(0, p_v - q_v) <= p_v <= p(m_g), m_g the largest target logit of
// group g, the group's residual mass has the bound
//   R_g <= Rb_g = kGroup p(m_g) (1 + 2^-16) + 2^-100
// (the factor covers the rounding of the 32-term sum and of ex2, the floor
// entries whose p underflows), and its key E_g / R_g >= U_g / Rb_g because
// E = -log(1 - U) >= U.  A cluster of kCluCtas CTAs takes one sequence's
// rejected row (its record at the sequence's own slot), a share of its groups
// each:
//   stage   the share of the target row is copied to shared memory (cp.async)
//           while the share's uniforms are drawn;
//   bound   m_g and Rb_g of every group of the share, from shared memory;
//   probe   each lane set races its lowest-bound group exactly (the drafter
//           vectors are the only logits read from memory besides the
//           target row); K1, the least of these keys over the cluster, is
//           exchanged through distributed shared memory;
//   race    every group whose bound does not put it above K1 (U_g f > K1 Rb_g
//           fails, f = kRaceFilter) is raced exactly, with the arithmetic and
//           summation order of the race over every group;
//   level 2 the cluster's least (key, group), lowest group on ties, gets the
//           entry race.
// A group left out has a key above K1 by more than the filter's margin (1e-5
// relative, far above the rounding of E, of the sum and of the quotient), so
// it can neither win nor tie: the token is the one the race over every group
// draws.  The drafter row and the exponentials are touched for a few groups
// per row instead of all of them.
#ifndef CMSD_CLU_CTAS
#define CMSD_CLU_CTAS 4
#endif
#ifndef CMSD_CLU_THREADS
#define CMSD_CLU_THREADS 512
#endif
#ifndef CMSD_CLU_MIN_BLOCKS
#define CMSD_CLU_MIN_BLOCKS 2
#endif
constexpr int kCluCtas = CMSD_CLU_CTAS;                  // CTAs per row (one cluster)
constexpr int kCluThreads = CMSD_CLU_THREADS;
constexpr int kCluWarps = kCluThreads / 32;
constexpr int kCluCands = 1024;                          // candidate list; past it the share is raced whole
constexpr size_t kCluSmemMax = 200 * 1024;               // larger shares take the race over every group
constexpr float kGroupBoundScale = 32.0f + 1.0f / 2048.0f;   // kGroup (1 + 2^-16)
constexpr float kGroupBoundFloor = 0x1p-100f;
static_assert(kGroup == 32, "the bound's factor is kGroup (1 + 2^-16)");

// Groups per CTA: a multiple of four, so that a share starts on a block of
// four group uniforms.
__host__ __device__ inline int clu_share(int ng) {
  const int s = (ng + kCluCtas - 1) / kCluCtas;
  return (s + 3) & ~3;
}
// Dynamic shared memory of one CTA: the staged target share, the share's
// uniforms and bounds, the candidate list.
template <typename T>
__host__ __device__ inline size_t clu_smem_bytes(int V) {
  const size_t ngs = (size_t)clu_share((V + kGroup - 1) / kGroup);
  return ngs * kGroup * sizeof(T) + ngs * 2 * sizeof(float) + (size_t)kCluCands * sizeof(int);
}

__device__ __forceinline__ float expo_u(float u) { return -log1pf(-u); }   // expo() of the same word

// The largest logit of a 16-byte vector.
__device__ __forceinline__ float vec_max(uint4 q, const uint16_t*) {
  const uint32_t m = bmax2(bmax2(q.x, q.y), bmax2(q.z, q.w));
  return fmaxf(bf_lo(m), bf_hi(m));
}
__device__ __forceinline__ float vec_max(uint4 q, const float*) {
  return fmaxf(fmaxf(__uint_as_float(q.x), __uint_as_float(q.y)), fmaxf(__uint_as_float(q.z), __uint_as_float(q.w)));
}

// The staged share keeps group g's vectors in 16-byte slots g LPG .. g LPG +
// LPG - 1, vector k in slot g LPG + ((k + rot(g)) mod LPG), rot(g) = g LPG / 8:
// a thread that reads a whole group (one vector per load) and its neighbours
// reading theirs then touch eight different 16-byte bank slots per quarter
// warp.
template <int LPG>
__device__ __forceinline__ int clu_slot(int g, int k) {
  return g * LPG + ((k + ((g * LPG) >> 3)) & (LPG - 1));
}

// The largest logit of staged group g.
__device__ __forceinline__ float group_max(const unsigned char* stage, int g, const uint16_t*) {
  const uint4* q = reinterpret_cast<const uint4*>(stage);
  const uint4 a = q[clu_slot<4>(g, 0)], b = q[clu_slot<4>(g, 1)], c = q[clu_slot<4>(g, 2)], d = q[clu_slot<4>(g, 3)];
  const uint32_t x = bmax2(bmax2(a.x, b.x), bmax2(c.x, d.x));
  const uint32_t y = bmax2(bmax2(a.y, b.y), bmax2(c.y, d.y));
  const uint32_t z = bmax2(bmax2(a.z, b.z), bmax2(c.z, d.z));
  const uint32_t w = bmax2(bmax2(a.w, b.w), bmax2(c.w, d.w));
  const uint32_t m = bmax2(bmax2(x, y), bmax2(z, w));
  return fmaxf(bf_lo(m), bf_hi(m));
}
__device__ __forceinline__ float group_max(const unsigned char* stage, int g, const float*) {
  const uint4* q = reinterpret_cast<const uint4*>(stage);
  float m = -pos_inf();
#pragma unroll
  for (int k = 0; k < 8; ++k) m = fmaxf(m, vec_max(q[clu_slot<8>(g, k)], (const float*)nullptr));
  return m;
}

// Rb_g from the group's largest target logit.
__device__ __forceinline__ float group_bound(float m, const RowStat& st) {
  const float pm = __fmul_rn(ex2(__fmaf_rn(m, kLog2e, -st.MLt)), st.invSt);
  return __fmaf_rn(pm, kGroupBoundScale, kGroupBoundFloor);
}

// (key, group) order: the least key, the lowest group on ties.
__device__ __forceinline__ void key_min(float& k, int& g, float k2, int g2) {
  if (k2 < k || (k2 == k && g2 < g)) {
    k = k2;
    g = g2;
  }
}
// The CTA's least (key, group) in every thread, keys >= 0 or +inf and groups
// >= 0 or kIntMax: the pair ordered as one 64-bit integer (key bits, group),
// a redux.sync minimum per warp and one shared-memory atomicMin per warp.
// *s_best holds ~0 on entry (reset behind a barrier) and is read by every
// thread before the function returns.
__device__ __forceinline__ void key_min_cta(float& k, int& g, unsigned long long* s_best) {
  const uint32_t kb = __reduce_min_sync(kFull, __float_as_uint(k));
  const uint32_t gb = __reduce_min_sync(kFull, __float_as_uint(k) == kb ? (uint32_t)g : 0xFFFFFFFFu);
  if ((threadIdx.x & 31) == 0) atomicMin(s_best, ((unsigned long long)kb << 32) | gb);
  __syncthreads();
  const unsigned long long v = *s_best;
  k = __uint_as_float((uint32_t)(v >> 32));
  g = (int)(uint32_t)v;
}

// The exact key of a group from its vectors (vector `sub` in lane `sub` of
// the lane set; target qt, drafter qd): the sum in the order of the race over
// every group.  +inf when the residual mass is zero or `ok` is false.
template <typename T>
__device__ __forceinline__ float group_key(uint4 qt, uint4 qd, const RowStat& st, float u, bool ok) {
  constexpr int LPG = kGroup / Elem<T>::kVec;
  float acc = resid_vec<T>(qt, qd, st);
#pragma unroll
  for (int o = 1; o < LPG; o <<= 1) acc += __shfl_xor_sync(kFull, acc, o);
  return (ok && acc > 0.f) ? expo_u(u) / acc : pos_inf();
}

// Sequence b's record word, once the streaming kernel's epilogue has released
// it: polled with acquire loads, giving up after one second of globaltimer or
// 2^22 polls, whichever comes first (error bit 2 set, and 0 returned, which
// reads as no record).
__device__ __forceinline__ unsigned poll_record(const unsigned* p, unsigned* err) {
  unsigned long long t0;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t0));
  for (unsigned n = 0;; ++n) {
    unsigned w;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(w) : "l"(p) : "memory");
    if (w & 1u) return w;
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    if (t - t0 > 1000000000ull || n >= (1u << 22)) {
      atomicOr(err, 4u);
      return 0u;
    }
    __nanosleep(32);
  }
}

// The verifier row's argmax (the lowest index of its largest logit), by the
// whole CTA from global memory: the token of a row whose residual is empty.
// *s_am holds 0 on entry (reset behind a barrier).
template <typename T>
__device__ int row_argmax_cta(const T* tp, int V, bool vec_ok, unsigned long long* s_am) {
  constexpr int VEC = Elem<T>::kVec;
  float bm = -pos_inf();
  int bi = kIntMax;
  for (int v = (int)threadIdx.x * VEC; v < V; v += kCluThreads * VEC) {
    const uint4 q = load_logits<T>(tp, v, V, vec_ok);
#pragma unroll
    for (int k = 0; k < VEC; ++k) {
      const float z = logit_at<T>(q, k);
      if (v + k < V && (z > bm || (z == bm && v + k < bi))) {
        bm = z;
        bi = v + k;
      }
    }
  }
  // (value, index) as one 64-bit key: the value's bits in increasing order
  // (-0 taken as +0, so that equal values tie), then the complemented index
  uint32_t ub = __float_as_uint(bm + 0.0f);
  ub = (ub & 0x80000000u) ? ~ub : (ub | 0x80000000u);
  const uint32_t um = __reduce_max_sync(kFull, ub);
  const uint32_t ui = __reduce_max_sync(kFull, ub == um ? ~(uint32_t)bi : 0u);
  if ((threadIdx.x & 31) == 0) atomicMax(s_am, ((unsigned long long)um << 32) | ui);
  __syncthreads();
  return (int)~(uint32_t)(*s_am);
}

template <typename T>
__global__ void __launch_bounds__(kCluThreads, CMSD_CLU_MIN_BLOCKS) resample_bound_kernel(const StreamArgs a) {
  constexpr int VEC = Elem<T>::kVec;
  constexpr int LPG = kGroup / VEC;      // lanes per group
  constexpr int GPI = 32 / LPG;          // lane sets per warp
  constexpr int SETS = kCluWarps * GPI;  // lane sets per CTA
  extern __shared__ __align__(16) unsigned char clu_smem[];
  __shared__ unsigned long long s_best[2];   // key_min_cta of the probes, of the race
  __shared__ int s_n, s_hold;
  __shared__ int s_probe[SETS];          // the group each lane set probed (a group of one of its threads)
  __shared__ uint4 s_qd[SETS * LPG];     // drafter vectors of each lane set's best group
  __shared__ float s_k1[kCluCtas];       // each CTA's least probe key, written by that CTA into every CTA
  __shared__ float s_rk[kCluCtas];       // rank 0: each CTA's (key, group, token)
  __shared__ int s_rg[kCluCtas];
  __shared__ int s_rt[kCluCtas];
  __shared__ unsigned s_word;            // the sequence's record word
  __shared__ int s_fb;                   // rank 0: the row's token, or -1 for the argmax fallback
  __shared__ unsigned long long s_am;    // rank 0: row_argmax_cta's reduction
  cg::cluster_group cl = cg::this_cluster();
  const int cr = (int)cl.block_rank();
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  const int sub = lane % LPG;
  const int set = warp * GPI + lane / LPG;
  const int ng = (a.V + kGroup - 1) / kGroup;
  const int ngs = clu_share(ng);
  unsigned char* stage = clu_smem;
  float* s_u = reinterpret_cast<float*>(clu_smem + (size_t)ngs * kGroup * sizeof(T));
  float* s_rb = s_u + ngs;
  int* s_list = reinterpret_cast<int*>(s_rb + ngs);
  const int gs = cr * ngs;                                   // the share: groups [gs, gs + nloc)
  const int nloc = max(0, min(ng, gs + ngs) - gs);
  const uint32_t k0 = seed_lo(a.seed), k1 = seed_hi(a.seed);
  const uint32_t cw_grp = iter_word(a.iteration, kPurposeGroup);
  const uint32_t cw_ent = iter_word(a.iteration, kPurposeResidual);
  const int ncl = (int)gridDim.x / kCluCtas;
  // No griddepcontrol.wait here: a sequence's draw starts as soon as its
  // epilogue has released the record word (every read below follows that
  // acquire), while the streaming kernel may still be finishing other
  // sequences.  Its CTAs have all started (they trigger this launch at their
  // top), so it completes whatever this kernel does.
  const Workspace& W = a.ws;
  // Two cluster barriers per row: after the probes (K1) and after the
  // results.  A slot written before one barrier is read only between it and
  // the next, so no row overwrites what the previous row still reads.
  for (int rr = (int)blockIdx.x / kCluCtas; rr < a.B; rr += ncl) {   // sequence rr, the same for the cluster
    if (threadIdx.x == 0) s_word = poll_record(rec_word(W, rr), W.err);
    __syncthreads();
    const unsigned word = s_word;
    if ((int)((word >> 1) & 3u) != kSeqResidual) {
      // No residual draw for this sequence in this call: clear the word once
      // every CTA of the cluster has read it.  The same two cluster barriers
      // as a draw, so that CTAs that disagree (one poll timed out) still
      // meet at every barrier.
      cl.sync();
      cl.sync();
      if (cr == 0 && threadIdx.x == 0) *rec_word(W, rr) = 0u;
      continue;
    }
    const int b = rr, pos = (int)(word >> 3);
    const int r = b * a.K + pos;
    const T* tp = (const T*)a.target + (size_t)r * (size_t)a.V;     // no bonus row: Kt == K
    const T* dp = (const T*)a.draft + (size_t)r * (size_t)a.V;
    const bool vec_ok = ((((uintptr_t)tp) | ((uintptr_t)dp)) & 15) == 0;
    if (threadIdx.x == 0) s_best[0] = s_best[1] = ~0ull;   // the last row read them before its barriers
    // stage: the share of the target row (-inf past the row end), while the
    // share's uniforms are drawn and the row statistics load
    const int v0 = gs * kGroup;
    for (int j = threadIdx.x; j < nloc * LPG; j += kCluThreads) {
      const int v = v0 + j * VEC;
      const int sl = clu_slot<LPG>(j / LPG, j % LPG);
      if (vec_ok && v + VEC <= a.V) cp_async16(smem_u32(stage) + 16u * (uint32_t)sl, tp + v);
      else *reinterpret_cast<uint4*>(stage + 16 * sl) = load_logits<T>(tp, v, a.V, false);
    }
    cp_async_commit();
    const float2 ts = __ldcg(W.row_tstat + r), ds = __ldcg(W.row_dstat + r);
    for (int q = threadIdx.x; q < (nloc + 3) / 4; q += kCluThreads) {
      const U4 wd = philox4x32_10(U4{(uint32_t)(gs / 4 + q), (uint32_t)b, (uint32_t)pos, cw_grp}, k0, k1);
      s_u[4 * q + 0] = word_to_unit(wd.x);
      s_u[4 * q + 1] = word_to_unit(wd.y);
      s_u[4 * q + 2] = word_to_unit(wd.z);
      s_u[4 * q + 3] = word_to_unit(wd.w);
    }
    const RowStat st{ts.x, 1.0f / ts.y, ds.x, -1.0f / ds.y};
    cp_async_wait<0>();
    __syncthreads();
    // bound: m_g and Rb_g, one thread per group; each thread keeps its
    // lowest U_g / Rb_g (compared as U_a Rb_b < U_b Rb_a), then each lane set
    // the lowest of its LPG threads'
    float bu = 0.f, brb = 1.f;
    int lg = -1;
#pragma unroll 2
    for (int gl = threadIdx.x; gl < nloc; gl += kCluThreads) {
      const float rb = group_bound(group_max(stage, gl, (const T*)nullptr), st);
      s_rb[gl] = rb;
      const float u = s_u[gl];
      if (lg < 0 || u * brb < bu * rb) {
        bu = u;
        brb = rb;
        lg = gl;
      }
    }
#pragma unroll
    for (int o = 1; o < LPG; o <<= 1) {
      const float u2 = __shfl_xor_sync(kFull, bu, o), rb2 = __shfl_xor_sync(kFull, brb, o);
      const int g2 = __shfl_xor_sync(kFull, lg, o);
      if (g2 >= 0 && (lg < 0 || u2 * brb < bu * rb2 || (u2 * brb == bu * rb2 && g2 < lg))) {
        bu = u2;
        brb = rb2;
        lg = g2;
      }
    }
    // probe: the lane set's lowest-bound group, exactly
    float sk;                              // the lane set's best (key, group), its drafter vectors in s_qd
    int sg;
    {
      uint4 qt = neg_inf_vec<T>(), qd = neg_inf_vec<T>();
      if (lg >= 0) {
        qt = *reinterpret_cast<const uint4*>(stage + 16 * clu_slot<LPG>(lg, sub));
        qd = load_logits<T>(dp, (gs + lg) * kGroup + sub * VEC, a.V, vec_ok);
      }
      sk = group_key<T>(qt, qd, st, lg >= 0 ? s_u[lg] : 0.f, lg >= 0);
      sg = sk != pos_inf() ? gs + lg : kIntMax;
      s_qd[set * LPG + sub] = qd;
      if (sub == 0) s_probe[set] = lg;
    }
    float K1 = sk;
    int g1 = sg;
    key_min_cta(K1, g1, &s_best[0]);
    // K1: the least probe key of the cluster, an upper bound on the winner's key
    if (threadIdx.x < kCluCtas) *cl.map_shared_rank(&s_k1[cr], (int)threadIdx.x) = K1;
    if (threadIdx.x == 0) s_n = 0;
    cl.sync();
#pragma unroll
    for (int c = 0; c < kCluCtas; ++c) K1 = fminf(K1, s_k1[c]);
    // race: the groups of the share that the bound leaves at or below K1 and
    // that no lane set has probed (s_rb is complete: the barriers above)
    for (int gl = threadIdx.x; gl < nloc; gl += kCluThreads) {
      if (!(s_u[gl] * kRaceFilter > K1 * s_rb[gl]) && s_probe[(gl % kCluThreads) / LPG] != gl) {
        const int i = atomicAdd(&s_n, 1);
        if (i < kCluCands) s_list[i] = gl;
      }
    }
    __syncthreads();
    const int nc = s_n;
    const bool whole = nc > kCluCands;
    const int items = whole ? nloc : nc;
    for (int i0 = 0; i0 < items; i0 += SETS) {               // warp-uniform trip count
      const int i = i0 + set;
      const int gl = i < items ? (whole ? i : s_list[i]) : -1;
      uint4 qt = neg_inf_vec<T>(), qd = neg_inf_vec<T>();
      if (gl >= 0) {
        qt = *reinterpret_cast<const uint4*>(stage + 16 * clu_slot<LPG>(gl, sub));
        qd = load_logits<T>(dp, (gs + gl) * kGroup + sub * VEC, a.V, vec_ok);
      }
      const float key = group_key<T>(qt, qd, st, gl >= 0 ? s_u[gl] : 0.f, gl >= 0);
      if (key != pos_inf() && (key < sk || (key == sk && gs + gl < sg))) {   // the whole lane set agrees
        sk = key;
        sg = gs + gl;
        s_qd[set * LPG + sub] = qd;
      }
    }
    // the CTA's least (key, group), the lane set holding it, and its level-2
    // winner, pushed to rank 0 of the cluster
    float ck = sk;
    int cgrp = sg;
    if (threadIdx.x == 0) s_hold = 0;
    key_min_cta(ck, cgrp, &s_best[1]);
    if (sub == 0 && cgrp != kIntMax && sk == ck && sg == cgrp) s_hold = set;   // holders share one vector set
    __syncthreads();
    if (warp == 0) {
      int tok = -1;
      if (cgrp != kIntMax) {
        const int h = s_hold;
        const uint4 qt = *reinterpret_cast<const uint4*>(stage + 16 * clu_slot<LPG>(cgrp - gs, sub));
        const uint4 qd = s_qd[h * LPG + sub];
        tok = race_group_entries<T>(qt, qd, cgrp, 0, lane, st, (uint32_t)b, (uint32_t)pos, cw_ent, k0, k1);
      }
      if (lane == 0) {
        *cl.map_shared_rank(&s_rk[cr], 0) = ck;
        *cl.map_shared_rank(&s_rg[cr], 0) = cgrp;
        *cl.map_shared_rank(&s_rt[cr], 0) = tok;
      }
    }
    cl.sync();                             // every CTA's result is in rank 0
    if (cr == 0) {
      if (threadIdx.x == 0) {
        float k = pos_inf();
        int g = kIntMax, tok = -1;
#pragma unroll 1
        for (int c = 0; c < kCluCtas; ++c) {
          const float kc = s_rk[c];
          const int gc = s_rg[c];
          if (kc < k || (kc == k && gc < g)) {
            k = kc;
            g = gc;
            tok = s_rt[c];
          }
        }
        s_fb = (g == kIntMax || tok < 0) ? -1 : tok;
        s_am = 0ull;
      }
      __syncthreads();
      int tok = s_fb;
      if (tok < 0) tok = row_argmax_cta<T>(tp, a.V, vec_ok, &s_am);   // empty residual: the argmax
      if (threadIdx.x == 0) {
        a.out_tokens[(size_t)b * a.Ko + pos] = tok;
        *rec_word(W, rr) = 0u;             // every CTA of the cluster has read it (the barrier above)
      }
    }
  }
  // this grid completes only after the streaming grid (whatever comes next on
  // the stream then sees both)
  asm volatile("griddepcontrol.wait;" ::: "memory");
}

// ---------------------------------------------------------------------------
// the kernel
// ---------------------------------------------------------------------------

template <typename T, int MODE, bool SAMPLED, bool PH2>
__global__ void __launch_bounds__(kStreamThreads, 1) stream_kernel(const StreamArgs a) {
  constexpr bool HAS_D = MODE != kModeVerify;
  constexpr bool HAS_T = MODE != kModeConf;
  constexpr int VEC = Elem<T>::kVec;
  extern __shared__ __align__(128) unsigned char smem[];
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  const int w = blockIdx.x * kStreamWarps + warp;
  const Workspace& W = a.ws;
  const bool ragged = a.k_row != nullptr;
  int* s_pref = reinterpret_cast<int*>(smem);
  // the resample kernel (launched as a programmatic dependent) may be
  // scheduled now; it waits for this grid's completion before reading anything
  if (PH2) asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

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
        if (HAS_D && a.k_next) a.k_next[b] = a.k_fixed > 0 ? a.k_fixed : a.k_min;
        if (HAS_T) {
          a.n_accept[b] = 0;
          for (int i = 0; i < a.Ko; ++i) a.out_tokens[(size_t)b * a.Ko + i] = -1;
          if (a.accept)
            for (int i = 0; i < a.K; ++i) a.accept[(size_t)b * a.K + i] = 0;
          if (PH2) publish(a, b, a.bonus ? kSeqBonus : kSeqNone, 0);
        }
      }
    }
  }

  if (nrows > 0) {
    const StreamSplit sp(nrows, a.V, VEC, a.nwarps, stream_min_len(a.V));
    if (w < sp.W) {
      const int64_t e_begin = sp.start(w);
      const int64_t e_end = sp.start(w + 1);
      if (e_begin < e_end) walk_slice<T, MODE, SAMPLED, PH2>(a, s_pref, e_begin, e_end, sp, w, lane);
    }
  }
}

// Dynamic shared memory is at most the k_row prefix of kMaxRaggedB sequences;
// the attribute is set once per kernel and device.
constexpr size_t kMaxStreamSmem = ((size_t)(kMaxRaggedB + 1) * sizeof(int) + 127) / 128 * 128;

template <typename K>
cudaError_t smem_attr_once(K kernel, unsigned long long* done_mask) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const unsigned long long bit = 1ull << (dev & 63);
  if (__atomic_load_n(done_mask, __ATOMIC_ACQUIRE) & bit) return cudaSuccess;
  e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kMaxStreamSmem);
  if (e == cudaSuccess) __atomic_fetch_or(done_mask, bit, __ATOMIC_ACQ_REL);
  return e;
}

template <typename T, int MODE, bool SAMPLED, bool PH2>
cudaError_t launch_one(const StreamArgs& a, int grid, size_t smem, cudaStream_t s) {
  static unsigned long long done = 0ull;
  cudaError_t e = smem_attr_once(stream_kernel<T, MODE, SAMPLED, PH2>, &done);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3(kStreamThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  return cudaLaunchKernelEx(&cfg, stream_kernel<T, MODE, SAMPLED, PH2>, a);
}

template <typename T, int MODE, bool SAMPLED, bool PH2>
cudaError_t occupancy_one(size_t smem, int* nb) {
  static unsigned long long done = 0ull;
  cudaError_t e = smem_attr_once(stream_kernel<T, MODE, SAMPLED, PH2>, &done);
  if (e != cudaSuccess) return e;
  return cudaOccupancyMaxActiveBlocksPerMultiprocessor(nb, stream_kernel<T, MODE, SAMPLED, PH2>,
                                                       kStreamThreads, smem);
}

// Launched as a programmatic dependent of the streaming kernel just before it
// on the same stream: its CTAs may be scheduled as the streaming kernel's CTAs
// retire, and griddepcontrol.wait at its top orders it after that grid.
template <typename T, bool SAMPLED>
cudaError_t launch_resample_one(const StreamArgs& a, int grid, cudaStream_t s) {
  static unsigned long long done = 0ull;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const unsigned long long bit = 1ull << (dev & 63);
  if (!(__atomic_load_n(&done, __ATOMIC_ACQUIRE) & bit)) {
    e = cudaFuncSetAttribute(resample_kernel<T, SAMPLED>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)kResSmemBytes);
    if (e != cudaSuccess) return e;
    __atomic_fetch_or(&done, bit, __ATOMIC_ACQ_REL);
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3(kResThreads);
  cfg.dynamicSmemBytes = kResSmemBytes;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, resample_kernel<T, SAMPLED>, a);
}

// The residual draw by group bounds: `clusters` clusters of kCluCtas CTAs,
// launched the same way (the row loop covers any number of queued rows).
template <typename T>
cudaError_t launch_resample_bound_t(const StreamArgs& a, int clusters, cudaStream_t s) {
  static unsigned long long done = 0ull;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const unsigned long long bit = 1ull << (dev & 63);
  if (!(__atomic_load_n(&done, __ATOMIC_ACQUIRE) & bit)) {
    e = cudaFuncSetAttribute(resample_bound_kernel<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kCluSmemMax);
    if (e != cudaSuccess) return e;
    __atomic_fetch_or(&done, bit, __ATOMIC_ACQ_REL);
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(clusters * kCluCtas));
  cfg.blockDim = dim3(kCluThreads);
  cfg.dynamicSmemBytes = clu_smem_bytes<T>(a.V);
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = kCluCtas;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, resample_bound_kernel<T>, a);
}

// Whether the residual draw by group bounds takes rows of V entries on the
// current device: the share fits kCluSmemMax, and a cluster of kCluCtas CTAs
// with that much shared memory can be resident (answer cached per device and
// size).  Otherwise resample_kernel draws the residual.
template <typename T>
bool resample_bound_fits_t(int V) {
  const size_t smem = clu_smem_bytes<T>(V);
  if (smem > kCluSmemMax) return false;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return false;
  static std::mutex mu;
  static std::map<std::pair<int, size_t>, bool> cache;
  std::lock_guard<std::mutex> lk(mu);
  const auto key = std::make_pair(dev, smem);
  const auto it = cache.find(key);
  if (it != cache.end()) return it->second;
  bool ok = false;
  if (cudaFuncSetAttribute(resample_bound_kernel<T>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)kCluSmemMax) == cudaSuccess) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(kCluCtas);
    cfg.blockDim = dim3(kCluThreads);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = kCluCtas;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    ok = cudaOccupancyMaxActiveClusters(&n, resample_bound_kernel<T>, &cfg) == cudaSuccess && n > 0;
  }
  if (!ok) (void)cudaGetLastError();   // a refused query leaves no error behind for the caller
  cache.emplace(key, ok);
  return ok;
}

template <typename T>
cudaError_t launch_resample_t(bool sampled, const StreamArgs& a, int grid, cudaStream_t s) {
  return sampled ? launch_resample_one<T, true>(a, grid, s) : launch_resample_one<T, false>(a, grid, s);
}

template <typename T>
cudaError_t occupancy_resample_t(bool sampled, int* nb) {
  cudaError_t e = sampled ? cudaFuncSetAttribute(resample_kernel<T, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                 (int)kResSmemBytes)
                          : cudaFuncSetAttribute(resample_kernel<T, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                 (int)kResSmemBytes);
  if (e != cudaSuccess) return e;
  return sampled ? cudaOccupancyMaxActiveBlocksPerMultiprocessor(nb, resample_kernel<T, true>, kResThreads,
                                                                 kResSmemBytes)
                 : cudaOccupancyMaxActiveBlocksPerMultiprocessor(nb, resample_kernel<T, false>, kResThreads,
                                                                 kResSmemBytes);
}

// The kernel variants: confidence only; verify and fused, each under the
// PAPER rule without a second pass, the PAPER rule with the bonus row, and
// the sampled rule (always a second pass).
#define CMSD_DISPATCH(FN, ...)                                                              \
  do {                                                                                      \
    if (mode == kModeConf) return FN<T, kModeConf, false, false>(__VA_ARGS__);              \
    if (mode == kModeVerify) {                                                              \
      if (sampled) return FN<T, kModeVerify, true, true>(__VA_ARGS__);                      \
      if (second) return FN<T, kModeVerify, false, true>(__VA_ARGS__);                      \
      return FN<T, kModeVerify, false, false>(__VA_ARGS__);                                 \
    }                                                                                       \
    if (sampled) return FN<T, kModeFused, true, true>(__VA_ARGS__);                         \
    if (second) return FN<T, kModeFused, false, true>(__VA_ARGS__);                         \
    return FN<T, kModeFused, false, false>(__VA_ARGS__);                                    \
  } while (0)

template <typename T>
cudaError_t launch_stream_t(int mode, bool sampled, bool second, const StreamArgs& a, int grid, size_t smem,
                            cudaStream_t s) {
  CMSD_DISPATCH(launch_one, a, grid, smem, s);
}

template <typename T>
cudaError_t occupancy_stream_t(int mode, bool sampled, bool second, size_t smem, int* nb) {
  CMSD_DISPATCH(occupancy_one, smem, nb);
}
#undef CMSD_DISPATCH

}  // namespace cmsd
