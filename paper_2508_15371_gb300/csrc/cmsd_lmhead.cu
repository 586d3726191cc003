// The drafter's LM head fused with its confidence signals (include/cmsd.h,
// cmsd_lmhead_confidence).
//
// The paper's estimator sits on the drafter's output logits (Sec. I), the
// product z = h W^T of the drafter's last hidden state with its LM-head
// weight, and reads from each logit row the entropy, logit margin and softmax
// margin of Sec. III.B(1).  Here the product runs on the 5th-generation
// tensor cores (tcgen05.mma, bf16 in, fp32 accumulators in tensor memory) and
// each finished tile of 128 vocabulary entries x 64 hidden rows is folded, in
// the GEMM's epilogue, into per-row running statistics: running maximum and
// its first index, second largest logit, and compensated sums of e^(z - ref)
// and e^(z - ref)(z - ref) log2 e against a lazily moved exponent reference
// (the same arithmetic as the logits pass).  The logits never reach HBM
// unless the caller asks for them.  A second small kernel merges the per-CTA
// statistics of each row and computes H, margin, C and the log-sum-exp with
// the logits pass's row arithmetic.
//
// Layout: hidden [R][d] and weight [V][d] row-major bf16 (the usual
// [out][in] layout of a linear layer's weight), d a multiple of 64.  Each CTA
// owns a contiguous run of the vocabulary for one block of 64 hidden rows and
// streams its weight rows once through a ring of shared-memory stages filled
// by 2D tensor-memory-access (TMA) loads: per stage one box of 64 hidden
// dimensions x 128 weight rows (the MMA's A) and one of 64 x 64 hidden rows
// (its B), both with the 128-byte swizzle that the MMA's shared-memory
// descriptors name; rows past R or V arrive as zeros.  The hidden block is
// re-read from L2 for every tile.
#include <cuda.h>

#include <mutex>

#include "cmsd_stream_impl.cuh"

namespace cmsd {
namespace {

constexpr int kMergeRowsPerCta = 8;                 // one warp per row

// ---- shared-memory barriers and 2D TMA loads -----------------------------------
__device__ __forceinline__ unsigned long long lh_ns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
constexpr unsigned long long kLhWaitLimitNs = 1000000000ull;   // the launch takes well under a millisecond
__device__ __forceinline__ void mbar_init(uint32_t bar, unsigned count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
// arrive once and expect tx bytes of asynchronous copies in this phase
__device__ __forceinline__ void mbar_arrive_tx(uint32_t bar, uint32_t tx) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(tx) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}
// true once the phase with this parity has completed, false after kLhWaitLimitNs
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity) {
  if (mbar_try_wait(bar, parity)) return true;
  const unsigned long long t0 = lh_ns();
  for (;;) {
    for (int k = 0; k < 32; ++k)
      if (mbar_try_wait(bar, parity)) return true;
    if (lh_ns() - t0 > kLhWaitLimitNs) return false;
  }
}
// box of the 2D tensor map at (x, y) (x: innermost, in elements) into shared
// memory at dst, completing `bar` by transaction count
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int x, int y, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::
          "r"(dst), "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
      : "memory");
}

// The vocabulary run of CTA `cta` of a row block: nct near-equal runs of
// 8 entries ([v0, v1), v1 <= V).
__device__ __forceinline__ void cta_run(int V, int nct, int cta, int& v0, int& v1) {
  const int n8 = (V + 7) / 8;
  const int q = n8 / nct, rem = n8 - q * nct;
  v0 = (cta * q + (cta < rem ? cta : rem)) * 8;
  const int e = ((cta + 1) * q + (cta + 1 < rem ? cta + 1 : rem)) * 8;
  v1 = e < V ? e : V;
}

// Fold 32 consecutive logits (vocabulary entries v0 .. v0+31, those at or
// past vend masked) into a thread's running drafter statistics.
__device__ __forceinline__ void fold32(DLane& st, const float* z_src, int v0, int vend) {
  float z[32];
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    const float4 q = *reinterpret_cast<const float4*>(z_src + 4 * k);
    z[4 * k] = q.x; z[4 * k + 1] = q.y; z[4 * k + 2] = q.z; z[4 * k + 3] = q.w;
  }
#pragma unroll
  for (int k = 0; k < 32; ++k)
    if (v0 + k >= vend) z[k] = -pos_inf();
  // maxima: top-2 and the first index of the running maximum (entries come
  // in increasing index order, so a strict increase keeps the lowest index)
#pragma unroll
  for (int k = 0; k < 32; ++k) {
    st.f2 = fmaxf(st.f2, fminf(st.f1, z[k]));
    st.f1 = fmaxf(st.f1, z[k]);
    const bool up = z[k] > st.m;
    st.pos = up ? v0 + k : st.pos;
    st.m = up ? z[k] : st.m;
  }
  st.posw = 1;
  // one reference check, then the exponentials, summed among themselves
  const float me = d_mexp(st);
  if (me > st.ref + kRefSlack) d_reref(st, me);
  const float nc = neg_clamp();
  const u64 L = dup2(kLog2e);
  u64 ss = 0ull, ts = 0ull;
#pragma unroll
  for (int k = 0; k < 16; ++k) {
    const u64 x = fma2(pack2(fmaxf(z[2 * k], nc), fmaxf(z[2 * k + 1], nc)), L, st.negrL);
    const u64 e = ex2_2(x);
    ss = add2(ss, e);
    ts = fma2(e, x, ts);
  }
  kahan(st.s, st.cs, lo32f(ss) + hi32f(ss));
  kahan(st.t, st.ct, lo32f(ts) + hi32f(ts));
}

// ===========================================================================
// tcgen05 variant: the product on the 5th-generation tensor cores
// ===========================================================================
//
// One CTA of 192 threads per SM:
//   warp 0      lane 0 issues the TMA loads of each stage (weight box 64 x 128
//               rows = the MMA's A, hidden box 64 x 64 rows = its B);
//   warp 1      allocates TMEM (two 64-column fp32 accumulators), and lane 0
//               issues tcgen05.mma (M = 128 vocabulary entries, N = 64 hidden
//               rows, K = 16 per instruction) and the commits;
//   warps 2..5  the epilogue: warp w reads TMEM lanes 32 (w mod 4) .. (one
//               vocabulary entry per thread, 64 logits: one per hidden row),
//               transposes the tile through shared memory and folds it into
//               the per-row statistics (each thread: one hidden row, one half
//               of the 128 entries).
// Barriers: full[s] / empty[s] per stage (TMA -> MMA -> TMA), tfull[b] /
// tempty[b] per accumulator (MMA -> epilogue -> MMA).  Every wait is bounded;
// TMEM is released after the last commit and the last load have completed.
constexpr int kTcM = 128;                           // vocabulary entries per tile (MMA M)
constexpr int kTcAStage = kTcM * 128;               // 16 KB: 128 rows x 64 bf16
constexpr int kTcThreads = 192;
constexpr int kTcCPitch = kTcM + 4;                 // floats per row of the transposed 64-row chunk

// Shapes for a block of N hidden rows (the MMA's N: 64, 128 or 256).  The
// accumulators take 2N TMEM columns; the epilogue walks them in chunks of 64
// columns (hidden rows); the stage count fills the shared memory.
template <int N>
struct TcShape {
  static_assert(N == 64 || N == 128 || N == 256, "block rows");
  static constexpr int kStages = N == 256 ? 4 : (N == 128 ? 5 : 6);
  static constexpr int kBStage = N * 128;
  static constexpr int kCols = 2 * N;
  static constexpr int kChunks = N / 64;
  static constexpr size_t kStageBytes = (size_t)kStages * (kTcAStage + kBStage);
  static constexpr size_t kCBytes = (size_t)64 * kTcCPitch * 4;
  static constexpr size_t kSmem = 1024 + kStageBytes + kCBytes + 8 * (2 * kStages + 4) + 16;
  // instruction descriptor, kind::f16: fp32 accumulator, bf16 A and B, both
  // K-major, N >> 3 at bit 17, M >> 4 at bit 24
  static constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(N >> 3) << 17) |
                                     ((uint32_t)(kTcM >> 4) << 24);
  static_assert(kSmem <= 227 * 1024, "shared memory");
};

// Shared-memory matrix descriptor of a K-major tile with 128-byte rows and the
// 128-byte swizzle: start address, leading offset (unused for this layout),
// stride between 8-row groups = 1024 bytes, descriptor version 1, layout
// SWIZZLE_128B.
__device__ __forceinline__ uint64_t umma_desc_sw128(uint32_t saddr) {
  return (uint64_t)((saddr & 0x3FFFFu) >> 4) | ((uint64_t)1 << 16) | ((uint64_t)(1024 >> 4) << 32) |
         ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}

__device__ __forceinline__ void tc_mma(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                       uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void tc_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
// 32 lanes x 64 columns of fp32 from TMEM: thread i gets lane (taddr lane + i), columns c .. c + 63
__device__ __forceinline__ void tc_ld64(uint32_t taddr, float (&v)[64]) {
  uint32_t r[64];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x64.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32,%33,%34,%35,%36,%37,%38,%39,"
      "%40,%41,%42,%43,%44,%45,%46,%47,%48,%49,%50,%51,%52,%53,%54,%55,%56,%57,%58,%59,%60,%61,%62,%63}, [%64];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31]),
        "=r"(r[32]), "=r"(r[33]), "=r"(r[34]), "=r"(r[35]), "=r"(r[36]), "=r"(r[37]), "=r"(r[38]), "=r"(r[39]),
        "=r"(r[40]), "=r"(r[41]), "=r"(r[42]), "=r"(r[43]), "=r"(r[44]), "=r"(r[45]), "=r"(r[46]), "=r"(r[47]),
        "=r"(r[48]), "=r"(r[49]), "=r"(r[50]), "=r"(r[51]), "=r"(r[52]), "=r"(r[53]), "=r"(r[54]), "=r"(r[55]),
        "=r"(r[56]), "=r"(r[57]), "=r"(r[58]), "=r"(r[59]), "=r"(r[60]), "=r"(r[61]), "=r"(r[62]), "=r"(r[63])
      : "r"(taddr)
      : "memory");
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int k = 0; k < 64; ++k) v[k] = __uint_as_float(r[k]);
}
// named barrier among the 128 epilogue threads (barrier 0 is __syncthreads)
__device__ __forceinline__ void epi_bar() { asm volatile("bar.sync 1, 128;" ::: "memory"); }

template <int N>
__global__ void __launch_bounds__(kTcThreads, 1) lmhead_tc_kernel(const LmHeadArgs h,
                                                                 const __grid_constant__ CUtensorMap tmap_h,
                                                                 const __grid_constant__ CUtensorMap tmap_w) {
  using S = TcShape<N>;
  constexpr int kStages = S::kStages;
  extern __shared__ __align__(1024) unsigned char tc_smem_raw[];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int rb = blockIdx.x / h.nct, cta = blockIdx.x - rb * h.nct;
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  int v0, v1;
  cta_run(h.V, h.nct, cta, v0, v1);
  const int ntiles = v1 > v0 ? (v1 - v0 + kTcM - 1) / kTcM : 0;
  const int nkc = h.d / 64;
  const int G = ntiles * nkc;
  const int row0 = rb * N;

  const uint32_t raw = smem_u32(tc_smem_raw);
  const uint32_t pad = ((raw + 1023u) & ~1023u) - raw;
  unsigned char* sm = tc_smem_raw + pad;
  const uint32_t sA = raw + pad, sB = sA + kStages * kTcAStage;
  float* sC = reinterpret_cast<float*>(sm + S::kStageBytes);
  const uint32_t bars = smem_u32(sm + S::kStageBytes + S::kCBytes);
  const uint32_t full = bars, empty = bars + 8 * kStages;
  const uint32_t tfull = bars + 16 * kStages, tempty = tfull + 16;
  uint32_t* s_taddr = reinterpret_cast<uint32_t*>(sm + S::kStageBytes + S::kCBytes + 8 * (2 * kStages + 4));
  if (tid == 0) {
    for (int k = 0; k < kStages; ++k) {
      mbar_init(full + 8 * k, 1);
      mbar_init(empty + 8 * k, 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(tfull + 8 * b, 1);
      mbar_init(tempty + 8 * b, 128);
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(s_taddr)),
                 "r"(S::kCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tbase = *s_taddr;
  bool ok = true;

  if (warp == 0) {
    // ---- producer ----------------------------------------------------------
    if (lane == 0) {
      for (int g = 0; g < G; ++g) {
        const int slot = g % kStages;
        if (g >= kStages && ok) ok = mbar_wait(empty + 8 * slot, (uint32_t)((g / kStages - 1) & 1));
        const int t = g / nkc, kc = g - t * nkc;
        mbar_arrive_tx(full + 8 * slot, kTcAStage + S::kBStage);
        tma_load_2d(sA + slot * kTcAStage, &tmap_w, kc * 64, v0 + t * kTcM, full + 8 * slot);
        tma_load_2d(sB + slot * S::kBStage, &tmap_h, kc * 64, row0, full + 8 * slot);
      }
    }
  } else if (warp == 1) {
    // ---- MMA issuer --------------------------------------------------------
    if (lane == 0) {
      for (int t = 0; t < ntiles; ++t) {
        const int b = t & 1;
        if (t >= 2 && ok) ok = mbar_wait(tempty + 8 * b, (uint32_t)((t / 2 - 1) & 1));
        tc_fence_after();
        const uint32_t d = tbase + (uint32_t)(b * N);
        for (int kc = 0; kc < nkc; ++kc) {
          const int g = t * nkc + kc, slot = g % kStages;
          if (ok) ok = mbar_wait(full + 8 * slot, (uint32_t)((g / kStages) & 1));
          tc_fence_after();
          const uint64_t ad = umma_desc_sw128(sA + slot * kTcAStage);
          const uint64_t bd = umma_desc_sw128(sB + slot * S::kBStage);
#pragma unroll
          for (int ks = 0; ks < 4; ++ks)          // K = 16 per instruction: 32 bytes along the row
            tc_mma(d, ad + (uint64_t)(2 * ks), bd + (uint64_t)(2 * ks), S::kIdesc, (kc | ks) != 0);
          tc_commit(empty + 8 * slot);             // the stage may be refilled once these MMAs are done
        }
        tc_commit(tfull + 8 * b);                  // the accumulator is complete
      }
    }
    __syncwarp();
  } else {
    // ---- epilogue: warps 2..5 ------------------------------------------------
    const int e = tid - 64;                        // 0 .. 127
    const int q = warp & 3;                        // TMEM lane quarter this warp may read
    const int m = q * 32 + lane;                   // the vocabulary entry (TMEM lane) this thread reads
    const int jrow = e >> 1, half = e & 1;         // within each 64-row chunk: the row and half-tile it folds
    DLane st[S::kChunks];
#pragma unroll
    for (int c = 0; c < S::kChunks; ++c) dlane_init(st[c]);
    for (int t = 0; t < ntiles; ++t) {
      const int b = t & 1;
      if (ok) ok = mbar_wait(tfull + 8 * b, (uint32_t)((t / 2) & 1));
      tc_fence_after();
#pragma unroll
      for (int c = 0; c < S::kChunks; ++c) {
        float v[64];
        tc_ld64(tbase + ((uint32_t)(q * 32) << 16) + (uint32_t)(b * N + 64 * c), v);
        if (c == S::kChunks - 1) {
          tc_fence_before();
          mbar_arrive(tempty + 8 * b);             // this lane of the accumulator has been read
        }
        // transpose: row j of the chunk holds hidden row 64 c + j's logits over the 128 entries
#pragma unroll
        for (int j = 0; j < 64; ++j) sC[j * kTcCPitch + m] = v[j];
        epi_bar();
        const int vq = v0 + t * kTcM + half * 64;
        const float* zs = sC + jrow * kTcCPitch + half * 64;
        fold32(st[c], zs, vq, v1);
        fold32(st[c], zs + 32, vq + 32, v1);
        const int grow = row0 + 64 * c + jrow;
        if (h.logits && grow < h.R) {
          float* dst = h.logits + (size_t)grow * h.V;
          for (int k = 0; k < 64 && vq + k < v1; ++k) dst[vq + k] = zs[k];
        }
        epi_bar();                                 // the chunk buffer is rewritten next
      }
    }
#pragma unroll
    for (int c = 0; c < S::kChunks; ++c) {
      float s, t2;
      d_final(st[c], s, t2);
      DRed x{d_mexp(st[c]), s, t2, st[c].f2, st[c].pos};
      DRed y;
      y.m = __shfl_xor_sync(kFull, x.m, 1);
      y.s = __shfl_xor_sync(kFull, x.s, 1);
      y.t2 = __shfl_xor_sync(kFull, x.t2, 1);
      y.top2 = __shfl_xor_sync(kFull, x.top2, 1);
      y.idx = __shfl_xor_sync(kFull, x.idx, 1);
      fold_d(x, y);
      if (half == 0) {
        Partial p;
        p.d_m = x.m; p.d_s = x.s; p.d_t2 = x.t2; p.d_top2 = x.top2; p.d_idx = x.idx;
        p.t_m = 0.f; p.t_s = 0.f; p.t_idx = 0; p.t_cnt = 0;
        p.pad[0] = p.pad[1] = p.pad[2] = 0;
        h.part[((size_t)rb * h.nct + cta) * N + 64 * c + jrow] = p;
      }
    }
  }
  if (!ok) atomicOr(h.err, 4u);
  // teardown: the MMA issuer's last commit covers every MMA of the CTA; then
  // every thread is past its last TMEM access and TMEM is released
  if (warp == 1 && lane == 0 && ntiles > 0) {
    const int t = ntiles - 1;
    if (!mbar_wait(tfull + 8 * (t & 1), (uint32_t)((t / 2) & 1))) atomicOr(h.err, 4u);
  }
  if (warp == 0 && lane == 0) {                    // no TMA box still in flight into this CTA
    for (int g = (G > kStages ? G - kStages : 0); g < G; ++g)
      if (!mbar_wait(full + 8 * (g % kStages), (uint32_t)((g / kStages) & 1))) atomicOr(h.err, 4u);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tbase), "r"(S::kCols) : "memory");
}

// One warp per hidden row: fold the row's per-CTA partials, then the row's
// signals and confidence (the logits pass's row arithmetic).
__global__ void __launch_bounds__(32 * kMergeRowsPerCta) lmhead_merge_kernel(const LmHeadArgs h, const StreamArgs a) {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int lane = threadIdx.x & 31;
  const int r = blockIdx.x * kMergeRowsPerCta + (threadIdx.x >> 5);
  if (r >= h.R) return;                            // whole warps
  const int rb = r / h.nb, row = r - rb * h.nb;
  const Partial* base = h.part + (size_t)rb * h.nct * h.nb + row;
  DRed m = dred_empty();
  constexpr int kBatch = 8;                        // partials in flight per lane
  for (int k0 = lane; k0 < h.nct; k0 += 32 * kBatch) {
    float4 x0[kBatch], x1[kBatch];
#pragma unroll
    for (int j = 0; j < kBatch; ++j) {
      const int k = k0 + 32 * j;
      if (k < h.nct) {
        const float4* src = reinterpret_cast<const float4*>(base + (size_t)k * h.nb);
        x0[j] = __ldcg(src);
        x1[j] = __ldcg(src + 1);
      }
    }
#pragma unroll
    for (int j = 0; j < kBatch; ++j)
      if (k0 + 32 * j < h.nct) fold_d(m, DRed{x0[j].x, x0[j].y, x0[j].z, x0[j].w, __float_as_int(x1[j].x)});
  }
  const DRed dr = reduce_d(m);
  bool acc;
  unsigned long long cfx;
  row_results<float, kModeConf, false>(a, r, 0, 0, dr, tred_empty(), 0.f, 0.f, lane, acc, cfx);
}

}  // namespace

// Hidden rows per block: the least of 64, 128, 256 that holds R (more rows
// than 256 take several blocks, each reading the weight once).
int lmhead_block_rows(int R) { return R <= 64 ? 64 : (R <= 128 ? 128 : 256); }

int lmhead_ctas_per_block(int sms, int R, int V) {
  const int nb = lmhead_block_rows(R);
  const int nrb = (R + nb - 1) / nb;
  int nct = sms / (nrb > 0 ? nrb : 1);
  const int n8 = (V + 7) / 8;
  if (nct > n8) nct = n8;
  return nct < 1 ? 1 : nct;
}

namespace {
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static bool tried = false;
  static std::mutex mu;
  std::lock_guard<std::mutex> lk(mu);
  if (!tried) {
    tried = true;
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = (EncodeTiledFn)p;
  }
  return fn;
}
// a [rows][d] bf16 matrix read in boxes of 64 x box_rows, 128-byte swizzle,
// out-of-range rows read as zeros
bool encode_rows(CUtensorMap* m, const void* base, int d, int rows, int box_rows) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  const cuuint64_t dims[2] = {(cuuint64_t)d, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)d * 2};
  const cuuint32_t box[2] = {64u, (cuuint32_t)box_rows};
  const cuuint32_t estr[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}
}  // namespace

template <int N>
cudaError_t launch_tc(const LmHeadArgs& h, cudaStream_t s) {
  static unsigned long long done = 0ull;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  CUtensorMap tmap_h, tmap_w;
  if (!encode_rows(&tmap_h, h.hidden, h.d, h.R, N) || !encode_rows(&tmap_w, h.weight, h.d, h.V, kTcM))
    return cudaErrorInvalidValue;
  const unsigned long long bit = 1ull << (dev & 63);
  if (!(__atomic_load_n(&done, __ATOMIC_ACQUIRE) & bit)) {
    e = cudaFuncSetAttribute(lmhead_tc_kernel<N>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)TcShape<N>::kSmem);
    if (e != cudaSuccess) return e;
    __atomic_fetch_or(&done, bit, __ATOMIC_ACQ_REL);
  }
  const int nrb = (h.R + N - 1) / N;
  lmhead_tc_kernel<N><<<nrb * h.nct, kTcThreads, TcShape<N>::kSmem, s>>>(h, tmap_h, tmap_w);
  return cudaGetLastError();
}

cudaError_t launch_lmhead(const LmHeadArgs& h, const StreamArgs& a, cudaStream_t s) {
  if (h.nb != lmhead_block_rows(h.R)) return cudaErrorInvalidValue;
  cudaError_t e = h.nb == 64 ? launch_tc<64>(h, s) : (h.nb == 128 ? launch_tc<128>(h, s) : launch_tc<256>(h, s));
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)((h.R + kMergeRowsPerCta - 1) / kMergeRowsPerCta));
  cfg.blockDim = dim3(32 * kMergeRowsPerCta);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, lmhead_merge_kernel, h, a);
}

}  // namespace cmsd
