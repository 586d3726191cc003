// The drafter's LM head fused with its confidence signals (include/cmsd.h,
// cmsd_lmhead_confidence).
//
// The paper's estimator sits on the drafter's output logits (Sec. I), the
// product z = h W^T of the drafter's last hidden state with its LM-head
// weight, and reads from each logit row the entropy, logit margin and softmax
// margin of Sec. III.B(1).  Here the product runs on the tensor cores
// (mma.sync m16n8k16, bf16 in, fp32 accumulation; 8 warps, each 64 rows x 32
// vocabulary entries) and each finished 64 x 256 tile of logits is folded, in
// the GEMM's epilogue, into per-row running
// statistics: running maximum and its first index, second largest logit, and
// compensated sums of e^(z - ref) and e^(z - ref)(z - ref) log2 e against a
// lazily moved exponent reference (the same arithmetic as the logits pass).
// The logits never reach HBM unless the caller asks for them.  A second small
// kernel merges the per-CTA statistics of each row and computes H, margin, C
// and the log-sum-exp with the logits pass's row arithmetic.
//
// Layout: hidden [R][d] and weight [V][d] row-major bf16 (the usual
// [out][in] layout of a linear layer's weight), d a multiple of 64.  Each CTA
// owns a contiguous run of the vocabulary for one block of 64 hidden rows and
// streams its weight rows once through a ring of shared-memory stages filled
// by 2D tensor-memory-access (TMA) loads: per stage one box of 64 hidden
// dimensions x 64 hidden rows and one of 64 x 256 weight rows, with the
// 128-byte swizzle (16-byte chunk c of row r lands at chunk c ^ (r mod 8)), so
// that ldmatrix reads are free of bank conflicts; rows past R or V arrive as
// zeros.  The hidden block is re-read from L2 for every tile.  (cp.async
// loads of the same stages held the weight stream near 3.7 TB/s.)
#include <cuda.h>

#include <mutex>

#include "cmsd_stream_impl.cuh"

namespace cmsd {
namespace {

#ifndef CMSD_LH_WARPS
#define CMSD_LH_WARPS 8
#endif
#ifndef CMSD_LH_WARP_COLS
#define CMSD_LH_WARP_COLS 32
#endif
#ifndef CMSD_LH_STAGES
#define CMSD_LH_STAGES 3
#endif
constexpr int kLhWarps = CMSD_LH_WARPS;
constexpr int kLhWarpCols = CMSD_LH_WARP_COLS;      // vocabulary entries per warp and tile (multiple of 16)
constexpr int kLhNT = kLhWarpCols / 8;              // n8 tiles per warp
constexpr int kLhThreads = 32 * kLhWarps;
constexpr int kLhCols = kLhWarps * kLhWarpCols;     // vocabulary entries per tile
#ifndef CMSD_LH_DEPTH
#define CMSD_LH_DEPTH 64
#endif
constexpr int kLhDepth = CMSD_LH_DEPTH;             // hidden dimensions per stage (a multiple of 64)
constexpr int kLhChunks = kLhDepth / 8;             // 16-byte chunks per row of a stage
constexpr int kLhKs = kLhDepth / 16;                // k16 steps per stage
constexpr int kLhStages = CMSD_LH_STAGES;
constexpr int kLhAStage = kLhRows * kLhDepth * 2;   // 8 KB
constexpr int kLhBStage = kLhCols * kLhDepth * 2;
constexpr int kLhCPitch = kLhCols + 4;              // floats per row of the epilogue tile
constexpr int kLhRowThreads = kLhThreads / kLhRows; // threads that fold one row of a tile
constexpr int kLhFold = kLhCols / kLhRowThreads;    // logits each of them folds per tile
constexpr size_t kLhStageBytes = (size_t)kLhStages * (kLhAStage + kLhBStage);
constexpr size_t kLhSmem = 1024 + kLhStageBytes + (size_t)kLhRows * kLhCPitch * 4 + 8 * kLhStages;
static_assert(kLhWarpCols % 16 == 0 && kLhFold % 32 == 0 && kLhThreads % kLhRows == 0, "tile shape");
static_assert((kLhRows * kLhChunks) % kLhThreads == 0 && (kLhCols * kLhChunks) % kLhThreads == 0, "stage copy split");
static_assert(kLhDepth == 64, "one TMA box (128 bytes, the swizzle span) per row and stage");
static_assert(kLhCols <= 256, "TMA box height");
static_assert(kLhSmem <= 227 * 1024, "shared memory");
#ifndef CMSD_LH_CTAS_PER_SM
#define CMSD_LH_CTAS_PER_SM 1
#endif
constexpr int kLhCtasPerSm = CMSD_LH_CTAS_PER_SM;
constexpr int kMergeRowsPerCta = 8;                 // one warp per row

// Byte offset of 16-byte chunk `ch` of row `row` in a stage whose rows are
// 2 kLhDepth bytes: chunks are XOR-swizzled by the row's low 3 bits, so the 8
// rows an ldmatrix phase reads fall on 8 different bank groups.
__device__ __forceinline__ uint32_t swz(int row, int ch) {
  return (uint32_t)(row * (2 * kLhDepth) + ((ch ^ (row & 7)) << 4));
}

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

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t (&r)[4]) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}

// c += a b for one 16x8 tile, a 16x16 (row-major fragments), b 16x8 (column fragments)
__device__ __forceinline__ void mma_bf16(float (&c)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
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

__global__ void __launch_bounds__(kLhThreads, kLhCtasPerSm) lmhead_gemm_kernel(const LmHeadArgs h,
                                                                    const __grid_constant__ CUtensorMap tmap_h,
                                                                    const __grid_constant__ CUtensorMap tmap_w) {
  extern __shared__ __align__(1024) unsigned char lh_smem_raw[];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int rb = blockIdx.x / h.nct, cta = blockIdx.x - rb * h.nct;
  // the merge kernel may be scheduled now; it waits for this grid before reading
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  int v0, v1;
  cta_run(h.V, h.nct, cta, v0, v1);
  const int ntiles = v1 > v0 ? (v1 - v0 + kLhCols - 1) / kLhCols : 0;
  const int nkc = h.d / kLhDepth;
  const int G = ntiles * nkc;                      // stages of this CTA
  const int row0 = rb * kLhRows;
  // the swizzled TMA boxes want 1024-byte aligned destinations
  const uint32_t raw = smem_u32(lh_smem_raw);
  const uint32_t pad = ((raw + 1023u) & ~1023u) - raw;
  unsigned char* lh_smem = lh_smem_raw + pad;
  const uint32_t sA = raw + pad, sB = sA + kLhStages * kLhAStage;
  float* sC = reinterpret_cast<float*>(lh_smem + kLhStageBytes);
  const uint32_t sBar = smem_u32(lh_smem + kLhStageBytes + (size_t)kLhRows * kLhCPitch * 4);
  if (tid == 0) {
#pragma unroll
    for (int k = 0; k < kLhStages; ++k) mbar_init(sBar + 8 * k, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  bool ok_waits = true;

  // stage g: hidden dimensions [64 kc, 64 kc + 64) of tile t = g / nkc; one
  // thread arms the stage's barrier and issues both boxes
  auto load = [&](int g) {
    const int t = g / nkc, kc = g - t * nkc;
    const int slot = g % kLhStages;
    const uint32_t bar = sBar + 8 * slot;
    mbar_arrive_tx(bar, kLhAStage + kLhBStage);
    tma_load_2d(sA + slot * kLhAStage, &tmap_h, kc * kLhDepth, row0, bar);
    tma_load_2d(sB + slot * kLhBStage, &tmap_w, kc * kLhDepth, v0 + t * kLhCols, bar);
  };

  DLane st;
  dlane_init(st);
  float acc[4][kLhNT][4];
#pragma unroll
  for (int mt = 0; mt < 4; ++mt)
#pragma unroll
    for (int nt = 0; nt < kLhNT; ++nt)
#pragma unroll
      for (int k = 0; k < 4; ++k) acc[mt][nt][k] = 0.f;

  if (tid == 0) {
#pragma unroll
    for (int s = 0; s < kLhStages - 1; ++s)
      if (s < G) load(s);
  }
  const int j8 = lane >> 3, r8 = lane & 7;
  for (int g = 0; g < G; ++g) {
    __syncthreads();                               // every warp is done with stage g - 1 ...
    if (tid == 0 && g + kLhStages - 1 < G) load(g + kLhStages - 1);   // ... so its slot is refilled
    const int slot = g % kLhStages;
    if (ok_waits) ok_waits = mbar_wait(sBar + 8 * slot, (uint32_t)((g / kLhStages) & 1));
    const uint32_t a_st = sA + slot * kLhAStage, b_st = sB + slot * kLhBStage;
    // fragments double-buffered: k16 step ks + 1 is read from shared memory
    // while step ks multiplies
    uint32_t af[2][4][4], bf[2][kLhNT / 2][4];
    auto frags = [&](int ks, int buf) {
#pragma unroll
      for (int mt = 0; mt < 4; ++mt)
        ldsm_x4(a_st + swz(mt * 16 + (j8 & 1) * 8 + r8, ks * 2 + (j8 >> 1)), af[buf][mt]);
#pragma unroll
      for (int np = 0; np < kLhNT / 2; ++np)      // two n8 tiles per ldmatrix
        ldsm_x4(b_st + swz(warp * kLhWarpCols + np * 16 + (j8 >> 1) * 8 + r8, ks * 2 + (j8 & 1)), bf[buf][np]);
    };
    frags(0, 0);
#pragma unroll
    for (int ks = 0; ks < kLhKs; ++ks) {
      if (ks + 1 < kLhKs) frags(ks + 1, (ks + 1) & 1);
#pragma unroll
      for (int mt = 0; mt < 4; ++mt)
#pragma unroll
        for (int np = 0; np < kLhNT / 2; ++np) {
          mma_bf16(acc[mt][2 * np], af[ks & 1][mt], bf[ks & 1][np][0], bf[ks & 1][np][1]);
          mma_bf16(acc[mt][2 * np + 1], af[ks & 1][mt], bf[ks & 1][np][2], bf[ks & 1][np][3]);
        }
    }
    if ((g + 1) % nkc == 0) {
      // tile t complete: accumulators -> shared tile -> each thread folds
      // kLhFold logits of one row (row tid / kLhRowThreads)
      const int t = g / nkc;
      const int gq = lane >> 2, tq = lane & 3;
#pragma unroll
      for (int mt = 0; mt < 4; ++mt)
#pragma unroll
        for (int nt = 0; nt < kLhNT; ++nt) {
          const int r = mt * 16 + gq, c = warp * kLhWarpCols + nt * 8 + 2 * tq;
          *reinterpret_cast<float2*>(sC + r * kLhCPitch + c) = make_float2(acc[mt][nt][0], acc[mt][nt][1]);
          *reinterpret_cast<float2*>(sC + (r + 8) * kLhCPitch + c) = make_float2(acc[mt][nt][2], acc[mt][nt][3]);
#pragma unroll
          for (int k = 0; k < 4; ++k) acc[mt][nt][k] = 0.f;
        }
      __syncthreads();
      const int row = tid / kLhRowThreads, qt = tid % kLhRowThreads;
      const int vq = v0 + t * kLhCols + qt * kLhFold;
      const float* zs = sC + row * kLhCPitch + qt * kLhFold;
#pragma unroll 1
      for (int c = 0; c < kLhFold; c += 32) fold32(st, zs + c, vq + c, v1);
      if (h.logits && row0 + row < h.R) {
        float* dst = h.logits + (size_t)(row0 + row) * h.V;
        for (int k = 0; k < kLhFold && vq + k < v1; ++k) dst[vq + k] = zs[k];
      }
      // the tile is rewritten only after the next tile's stages, each of
      // which starts with a barrier
    }
  }
  if (!ok_waits) atomicOr(h.err, 4u);
  // before the CTA exits, no box may still be in flight into its shared memory
  if (tid == 0) {
    for (int g = (G > kLhStages ? G - kLhStages : 0); g < G; ++g)
      if (!mbar_wait(sBar + 8 * (g % kLhStages), (uint32_t)((g / kLhStages) & 1))) atomicOr(h.err, 4u);
  }

  // the row's kLhRowThreads runs (adjacent lanes), then one partial per (row, CTA)
  float s, t2;
  d_final(st, s, t2);
  DRed x{d_mexp(st), s, t2, st.f2, st.pos};
#pragma unroll
  for (int o = 1; o < kLhRowThreads; o <<= 1) {
    DRed y;
    y.m = __shfl_xor_sync(kFull, x.m, o);
    y.s = __shfl_xor_sync(kFull, x.s, o);
    y.t2 = __shfl_xor_sync(kFull, x.t2, o);
    y.top2 = __shfl_xor_sync(kFull, x.top2, o);
    y.idx = __shfl_xor_sync(kFull, x.idx, o);
    fold_d(x, y);
  }
  if (tid % kLhRowThreads == 0) {
    Partial p;
    p.d_m = x.m; p.d_s = x.s; p.d_t2 = x.t2; p.d_top2 = x.top2; p.d_idx = x.idx;
    p.t_m = 0.f; p.t_s = 0.f; p.t_idx = 0; p.t_cnt = 0;
    p.pad[0] = p.pad[1] = p.pad[2] = 0;
    h.part[((size_t)rb * h.nct + cta) * kLhRows + tid / kLhRowThreads] = p;
  }
}

// One warp per hidden row: fold the row's per-CTA partials, then the row's
// signals and confidence (the logits pass's row arithmetic).
__global__ void __launch_bounds__(32 * kMergeRowsPerCta) lmhead_merge_kernel(const LmHeadArgs h, const StreamArgs a) {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int lane = threadIdx.x & 31;
  const int r = blockIdx.x * kMergeRowsPerCta + (threadIdx.x >> 5);
  if (r >= h.R) return;                            // whole warps
  const int rb = r / kLhRows, row = r - rb * kLhRows;
  const Partial* base = h.part + (size_t)rb * h.nct * kLhRows + row;
  DRed m = dred_empty();
  constexpr int kBatch = 8;                        // partials in flight per lane
  for (int k0 = lane; k0 < h.nct; k0 += 32 * kBatch) {
    float4 x0[kBatch], x1[kBatch];
#pragma unroll
    for (int j = 0; j < kBatch; ++j) {
      const int k = k0 + 32 * j;
      if (k < h.nct) {
        const float4* src = reinterpret_cast<const float4*>(base + (size_t)k * kLhRows);
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

int lmhead_ctas_per_block(int sms, int R, int V) {
  const int nrb = (R + kLhRows - 1) / kLhRows;
  int nct = sms * kLhCtasPerSm / (nrb > 0 ? nrb : 1);
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
  const cuuint32_t box[2] = {(cuuint32_t)kLhDepth, (cuuint32_t)box_rows};
  const cuuint32_t estr[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}
}  // namespace

cudaError_t launch_lmhead(const LmHeadArgs& h, const StreamArgs& a, cudaStream_t s) {
  static unsigned long long done = 0ull;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  CUtensorMap tmap_h, tmap_w;
  if (!encode_rows(&tmap_h, h.hidden, h.d, h.R, kLhRows) || !encode_rows(&tmap_w, h.weight, h.d, h.V, kLhCols))
    return cudaErrorInvalidValue;
  const unsigned long long bit = 1ull << (dev & 63);
  if (!(__atomic_load_n(&done, __ATOMIC_ACQUIRE) & bit)) {
    e = cudaFuncSetAttribute(lmhead_gemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kLhSmem);
    if (e != cudaSuccess) return e;
    __atomic_fetch_or(&done, bit, __ATOMIC_ACQ_REL);
  }
  const int nrb = (h.R + kLhRows - 1) / kLhRows;
  lmhead_gemm_kernel<<<nrb * h.nct, kLhThreads, kLhSmem, s>>>(h, tmap_h, tmap_w);
  e = cudaGetLastError();
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
