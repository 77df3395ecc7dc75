// Adapter drift (Eq. 8) on the tensor cores.
//
// Per (layer, module) item, the weight-space change of the unscaled LoRA update factors as
//   B1 A1 - B0 A0 = [B1 - B0 | B0] [A1 ; A1 - A0],
// so ||B1 A1 - B0 A0||_F^2 = tr(GB GA) with the 2r x 2r Grams GB = Bt^T Bt over the output rows
// and GA = At At^T over the input columns; every Gram entry already scales with the change, so
// nothing cancels. The parameter-space change ||A1 - A0||^2 + ||B1 - B0||^2 is the trace of the
// two difference blocks.
//
// Both Grams are contractions over a long dimension (the output rows of B, the input columns of
// A: 512..18944 at the Qwen2.5 shapes) and run here as bf16 mma.sync products with fp32
// accumulation. The difference of two bf16 factors is exact in fp32 but not in bf16, so each
// difference enters as a bf16 pair hi + lo (hi = bf16(d), lo = bf16(d - hi)); every product of
// two bf16 values is exact in fp32, so the Grams carry the fp32-accumulated value of the exact
// differences. Per long-dimension row the feature vector is [hi(d) | lo(d) | base] with
// d = B1 - B0, base = B0 for the B side and d = A1 - A0, base = A1 for the A side, padded to
// RP = max(r, 8) features per part (zeros), and the kernel accumulates the block-upper triangle
// of its Gram (16 x 16 blocks).
//
// Work split: the long dimension of every (item, side) segment is cut into 256-row steps; the
// steps of all segments are laid end to end and a persistent grid of G CTAs takes equal
// consecutive ranges of them (stream-K). A CTA stages each step's rows of both versions with
// cp.async (two steps in flight while one is multiplied, no registers held), builds the
// hi/lo/base fragments in registers from ldmatrix loads (transposed for the B side, whose rows
// are [r] wide), and its 8 warps each accumulate two 16-row slices. When its range leaves a segment (or ends) the CTA sums
// its warps in a fixed order and writes one partial Gram to slot (b + seg), unique because a
// CTA's segments follow the previous CTA's. The final kernel sums each segment's slots in CTA
// order and forms tr(GB GA) and the parameter distance in fp64. The result does not depend on
// timing: same inputs, same bits.
#include "common.cuh"
#include "kernels.h"

namespace crf {

namespace {

constexpr int kDtThreads = 256;
constexpr int kDtRows = 256;   // long-dimension rows per step: 8 warps x 2 slices x 16
constexpr int kDtSlices = kDtRows / 128;  // 16-row slices per warp and step
constexpr int kDtStages = 3;   // two steps in flight while one is multiplied
constexpr int kDtCtasPerSm = 3;
constexpr int kDtMaxItems = 224;
constexpr int kDtMaxSegs = 2 * kDtMaxItems;
constexpr int kDtAStride = kDtRows * 2 + 16;  // bytes per A row in a stage (+16: no bank conflicts)

struct DriftTcArgs {
  DriftItem items[kDtMaxItems];
  int seg_step0[kDtMaxSegs + 1];  // first step of segment s = 2 * item + side; [n_segs] = total
  int n_items, n_segs, total_steps, grid, rank;
};

template <int R>
struct DtShape {
  static constexpr int RP = R < 8 ? 8 : R;                      // features per part (zero padded)
  // bytes per B row in a stage: 32 for RP = 16, its two 16-byte halves swapped in rows 4-7 of
  // every 8 (b_unit), so the transposed ldmatrix of 8 consecutive rows meets 8 distinct bank groups
  static constexpr int kBStride = RP == 16 ? 32 : 16;
  static constexpr int kBVersion = kDtRows * kBStride;          // one version of the B side
  static constexpr int kAVersion = RP * kDtAStride;             // one version of the A side
  static constexpr int kStage = 2 * (kBVersion > kAVersion ? kBVersion : kAVersion);
  static constexpr int kBlocks = RP == 16 ? 3 : 2;              // 16-feature blocks of [hi|lo|base]
  // block pairs (I <= J) accumulated: the block-upper triangle, except lo x lo for RP = 16 (its
  // entries are below 2^-18 of hi x hi, far under the drift tolerance)
  static constexpr int kPairs = RP == 16 ? 5 : 3;
  static constexpr int kSlotFloats = kPairs * 256;
  // copies per step and version: B side in chunks of min(16, 2R) bytes per row; A side in 16-byte
  // chunks of R rows
  static constexpr int kBChunkBytes = 2 * R < 16 ? 2 * R : 16;
  static constexpr int kBChunksPerRow = 2 * R / kBChunkBytes;
  static constexpr int kBCopies = 2 * kDtRows * kBChunksPerRow;
  static constexpr int kACopies = 2 * R * (kDtRows / 8);
  static constexpr int kBPerThread = (kBCopies + kDtThreads - 1) / kDtThreads;
  static constexpr int kAPerThread = (kACopies + kDtThreads - 1) / kDtThreads;
};

// (I, J) of accumulated pair p, and the pair of (I, J) (-1: not accumulated, reads as zero)
template <int RP>
__host__ __device__ constexpr int pair_I(int p) { return RP == 16 ? (p < 3 ? 0 : (p == 3 ? 1 : 2)) : (p < 2 ? 0 : 1); }
template <int RP>
__host__ __device__ constexpr int pair_J(int p) { return RP == 16 ? (p < 3 ? p : 2) : (p < 2 ? p : 1); }
template <int RP>
__host__ __device__ constexpr int pair_of(int I, int J) {
  return RP == 16 ? (I == 0 ? J : (I == 1 ? (J == 2 ? 3 : -1) : 4)) : (I == 0 ? J : 2);
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, bool valid) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(valid ? 16 : 0)
               : "memory");
}
__device__ __forceinline__ void cp_async8(uint32_t dst, const void* src, bool valid) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 8, %2;" ::"r"(dst), "l"(src), "r"(valid ? 8 : 0)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

__device__ __forceinline__ void ldsm_x2(uint32_t addr, uint32_t& r0, uint32_t& r1) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x2.shared.b16 {%0, %1}, [%2];" : "=r"(r0), "=r"(r1) : "r"(addr));
}
__device__ __forceinline__ void ldsm_x2_t(uint32_t addr, uint32_t& r0, uint32_t& r1) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x2.trans.shared.b16 {%0, %1}, [%2];" : "=r"(r0), "=r"(r1) : "r"(addr));
}

__device__ __forceinline__ uint32_t bf2_sub(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("sub.rn.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}
__device__ __forceinline__ uint32_t bf2_add(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("add.rn.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}

// hi = bf16(a - b) and lo = (a - b) - hi, exactly, for two bf16 pairs: Knuth's TwoSum of a and -b
// in bf16 arithmetic with round-to-nearest (the rounding error of a sum is itself representable,
// and these six operations recover it without a wider format).
__device__ __forceinline__ void split_diff(uint32_t a, uint32_t b, uint32_t& hi, uint32_t& lo) {
  hi = bf2_sub(a, b);
  const uint32_t bv = bf2_sub(hi, a);   // the part of -b that hi holds
  const uint32_t av = bf2_sub(hi, bv);  // the part of a that hi holds
  lo = bf2_sub(bf2_sub(a, av), bf2_add(b, bv));
}

// Byte offset of 16-byte unit `ch` of B row `row` in a stage (rank 16: the XOR swizzle above).
template <int RP>
__device__ __forceinline__ int b_unit(int row, int ch) {
  return RP == 16 ? ((ch ^ ((row >> 2) & 1)) << 4) : (ch << 4);
}

// The item a run of steps belongs to, cached while the run stays in one segment.
struct SegCache {
  int seg = -1, side = 0, len = 0, step0 = 0, next0 = 0;
  const __nv_bfloat16 *p1 = nullptr, *p0 = nullptr;  // version 1 / version 0 of this side

  __device__ __forceinline__ void at(const DriftTcArgs& a, int x) {
    if (seg >= 0 && x < next0) return;
    int s = seg < 0 ? 0 : seg;
    while (s + 1 < a.n_segs && x >= a.seg_step0[s + 1]) ++s;
    seg = s;
    side = s & 1;
    const DriftItem& it = a.items[s >> 1];
    len = side == 0 ? it.out_dim : it.in_dim;
    step0 = a.seg_step0[s];
    next0 = a.seg_step0[s + 1];
    p1 = side == 0 ? it.B1 : it.A1;
    p0 = side == 0 ? it.B0 : it.A0;
  }
};

// Issue the copies of step x (version 1 then version 0) into a stage. Copy i of the step goes
// to thread i % 256: for the B side version i / (rows * chunks per row), then row and chunk; for
// the A side version, rank row and 16-byte chunk.
template <int R>
__device__ __forceinline__ void load_step(const SegCache& sc, int x, uint32_t stage) {
  using S = DtShape<R>;
  const int tid = threadIdx.x;
  const int row0 = (x - sc.step0) * kDtRows;
  if (sc.side == 0) {
    const size_t blk = static_cast<size_t>(row0) * R;
#pragma unroll
    for (int u = 0; u < S::kBPerThread; ++u) {
      const int i = tid + u * kDtThreads;
      if (S::kBCopies % kDtThreads != 0 && i >= S::kBCopies) continue;
      const int v = i / (kDtRows * S::kBChunksPerRow), rem = i % (kDtRows * S::kBChunksPerRow);
      const int row = rem / S::kBChunksPerRow, ch = rem % S::kBChunksPerRow;
      const bool ok = row0 + row < sc.len;
      const __nv_bfloat16* src =
          (v == 0 ? sc.p1 : sc.p0) + (ok ? blk + row * R + ch * (S::kBChunkBytes / 2) : 0);
      const uint32_t dst = stage + v * S::kBVersion + row * S::kBStride + b_unit<S::RP>(row, ch);
      if constexpr (S::kBChunkBytes == 16)
        cp_async16(dst, src, ok);
      else
        cp_async8(dst, src, ok);
    }
  } else {
#pragma unroll
    for (int u = 0; u < S::kAPerThread; ++u) {
      const int i = tid + u * kDtThreads;
      if (S::kACopies % kDtThreads != 0 && i >= S::kACopies) continue;
      const int v = i / (R * (kDtRows / 8)), rem = i % (R * (kDtRows / 8));
      const int k = rem / (kDtRows / 8), ch = rem % (kDtRows / 8);
      const int c = row0 + ch * 8;
      const bool ok = c < sc.len;  // the input width is a multiple of 8: a chunk is in or out
      const __nv_bfloat16* src = (v == 0 ? sc.p1 : sc.p0) + (ok ? static_cast<size_t>(k) * sc.len + c : 0);
      cp_async16(stage + v * S::kAVersion + k * kDtAStride + ch * 16, src, ok);
    }
  }
}

// This warp's 16-row slice of a staged step into its Gram accumulators.
template <int R>
__device__ __forceinline__ void mma_slice(int side, uint32_t stage, int row0,
                                          float (&acc)[DtShape<R>::kPairs][2][4]) {
  using S = DtShape<R>;
  constexpr int RP = S::RP;
  const int lane = threadIdx.x & 31;
  const int m = lane >> 3, i = lane & 7;
  uint32_t f1[4], f0[4];  // fragments of version 1 and version 0: {m0, m1, m2, m3} (RP = 8: m0, m2)
  if (side == 0) {
    // X[o][f] rows: matrix m covers rows k0 + (m >> 1) * 8 .. and features (m & 1) * 8 ..
    if constexpr (RP == 16) {
      const int row = row0 + (m >> 1) * 8 + i;
      const uint32_t off = row * S::kBStride + b_unit<RP>(row, m & 1);
      ldsm_x4_t(stage + off, f1[0], f1[1], f1[2], f1[3]);
      ldsm_x4_t(stage + S::kBVersion + off, f0[0], f0[1], f0[2], f0[3]);
    } else {
      const uint32_t off = (row0 + (m & 1) * 8 + i) * S::kBStride;
      ldsm_x2_t(stage + off, f1[0], f1[2]);
      ldsm_x2_t(stage + S::kBVersion + off, f0[0], f0[2]);
    }
  } else {
    // Xt[f][c] rows: matrix m covers features (m & 1) * 8 .. and columns k0 + (m >> 1) * 8 ..
    if constexpr (RP == 16) {
      const uint32_t off = ((m & 1) * 8 + i) * kDtAStride + (row0 + (m >> 1) * 8) * 2;
      ldsm_x4(stage + off, f1[0], f1[1], f1[2], f1[3]);
      ldsm_x4(stage + S::kAVersion + off, f0[0], f0[1], f0[2], f0[3]);
    } else {
      const uint32_t off = i * kDtAStride + (row0 + (m & 1) * 8) * 2;
      ldsm_x2(stage + off, f1[0], f1[2]);
      ldsm_x2(stage + S::kAVersion + off, f0[0], f0[2]);
    }
  }
  // base: B0 on the B side, A1 on the A side
  uint32_t blk[S::kBlocks][4];
  if constexpr (RP == 16) {
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      split_diff(f1[r], f0[r], blk[0][r], blk[1][r]);
      blk[2][r] = side == 0 ? f0[r] : f1[r];
    }
  } else {
    // block 0 = [hi (8 features) | lo (8)], block 1 = [base (8) | zeros]
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int r = 2 * h;
      split_diff(f1[r], f0[r], blk[0][r], blk[0][r + 1]);
      blk[1][r] = side == 0 ? f0[r] : f1[r];
      blk[1][r + 1] = 0u;
    }
  }
#pragma unroll
  for (int p = 0; p < S::kPairs; ++p) {
    const int I = pair_I<RP>(p), J = pair_J<RP>(p);
    mma16816(acc[p][0], blk[I], blk[J][0], blk[J][2]);
    mma16816(acc[p][1], blk[I], blk[J][1], blk[J][3]);
  }
}

// This warp's slices of a staged step.
template <int R>
__device__ __forceinline__ void mma_step(int side, uint32_t stage, float (&acc)[DtShape<R>::kPairs][2][4]) {
  const int warp = threadIdx.x >> 5;
#pragma unroll
  for (int sl = 0; sl < kDtSlices; ++sl) mma_slice<R>(side, stage, (warp * kDtSlices + sl) * 16, acc);
}

template <int R>
__global__ void __launch_bounds__(kDtThreads, kDtCtasPerSm)
    drift_tc_kernel(const __grid_constant__ DriftTcArgs a, float* __restrict__ slots) {
  using S = DtShape<R>;
  extern __shared__ __align__(128) uint8_t dt_smem[];
  float* red = reinterpret_cast<float*>(dt_smem + kDtStages * S::kStage);  // [kPairs * 8][32]
  const uint32_t stage0 = smem_u32(dt_smem);
  const int b = blockIdx.x;
  const int x0 = static_cast<int>((static_cast<long long>(b) * a.total_steps) / a.grid);
  const int x1 = static_cast<int>((static_cast<long long>(b + 1) * a.total_steps) / a.grid);
  if (x0 >= x1) return;
  // zero the stages once: the copies of a rank-4 adapter leave part of each row untouched
  for (int i = threadIdx.x; i < kDtStages * S::kStage / 16; i += kDtThreads)
    reinterpret_cast<uint4*>(dt_smem)[i] = make_uint4(0u, 0u, 0u, 0u);
  __syncthreads();

  float acc[S::kPairs][2][4];
#pragma unroll
  for (int p = 0; p < S::kPairs; ++p)
#pragma unroll
    for (int h = 0; h < 2; ++h)
#pragma unroll
      for (int v = 0; v < 4; ++v) acc[p][h][v] = 0.f;

  SegCache lc, sc;  // the next step to load, the step multiplied
  int lx = x0;
  auto issue = [&]() {
    if (lx < x1) {
      lc.at(a, lx);
      load_step<R>(lc, lx, stage0 + ((lx - x0) % kDtStages) * S::kStage);
    }
    cp_async_commit();  // empty groups keep the count uniform
    ++lx;
  };
  for (int k = 0; k < kDtStages - 1; ++k) issue();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int x = x0; x < x1; ++x) {
    cp_async_wait<kDtStages - 2>();  // this thread's copies of step x have landed
    __syncthreads();                 // everyone's have, and step x - 1's stage is free again
    issue();                         // step x + kDtStages - 1 into that stage
    sc.at(a, x);
    mma_step<R>(sc.side, stage0 + ((x - x0) % kDtStages) * S::kStage, acc);
    if (x + 1 == x1 || x + 1 >= sc.next0) {
      // the warps' partial Grams summed in warp order, then written as one slot
      for (int w = 0; w < kDtThreads / 32; ++w) {
        if (warp == w) {
#pragma unroll
          for (int p = 0; p < S::kPairs; ++p)
#pragma unroll
            for (int h = 0; h < 2; ++h)
#pragma unroll
              for (int v = 0; v < 4; ++v) {
                float* r = red + (p * 8 + h * 4 + v) * 32 + lane;
                *r = (w == 0 ? 0.f : *r) + acc[p][h][v];
              }
        }
        __syncthreads();
      }
      float* out = slots + static_cast<size_t>(b + sc.seg) * S::kSlotFloats;
      for (int e = threadIdx.x; e < S::kSlotFloats; e += kDtThreads) {
        const int p = e >> 8, rr = (e >> 4) & 15, cc = e & 15;
        const int ln = (rr & 7) * 4 + ((cc & 7) >> 1);
        const int v = (rr >> 3) * 2 + (cc & 1);
        out[e] = red[(p * 8 + (cc >> 3) * 4 + v) * 32 + ln];
      }
#pragma unroll
      for (int p = 0; p < S::kPairs; ++p)
#pragma unroll
        for (int h = 0; h < 2; ++h)
#pragma unroll
          for (int v = 0; v < 4; ++v) acc[p][h][v] = 0.f;
      __syncthreads();  // `red` is read before the next flush overwrites it
    }
  }
  cp_async_wait<0>();
}

// One block per item: the segment's slots summed in CTA order, GB and GA assembled from the
// [hi | lo | base] Grams (fp32: sums of at most four entries), then tr(GB GA) and the parameter
// distance in fp64.
template <int R>
__global__ void __launch_bounds__(256) drift_tc_final_kernel(const __grid_constant__ DriftTcArgs a,
                                                             const float* __restrict__ slots,
                                                             float* __restrict__ out_sq) {
  using S = DtShape<R>;
  constexpr int RP = S::RP;
  constexpr int r2 = 2 * R;
  __shared__ float g[2][S::kSlotFloats];
  __shared__ float gb[r2][r2 + 1], ga[r2][r2 + 1];
  __shared__ double red[2][8];
  const int item = blockIdx.x;
  // slots b_lo .. b_hi of each side's segment, summed in CTA order; every load of one slot
  // offset (both sides, all of a thread's entries) is issued before any of them is added
  constexpr int kPer = (S::kSlotFloats + 255) / 256;
  int b_lo[2], n_slot[2];
  for (int side = 0; side < 2; ++side) {
    const int seg = 2 * item + side;
    const long long s0 = a.seg_step0[seg], s1 = a.seg_step0[seg + 1] - 1;
    b_lo[side] = static_cast<int>(((s0 + 1) * a.grid - 1) / a.total_steps);
    n_slot[side] = static_cast<int>(((s1 + 1) * a.grid - 1) / a.total_steps) - b_lo[side] + 1;
  }
  float v[2][kPer];
#pragma unroll
  for (int side = 0; side < 2; ++side)
#pragma unroll
    for (int u = 0; u < kPer; ++u) v[side][u] = 0.f;
  const int n_max = n_slot[0] > n_slot[1] ? n_slot[0] : n_slot[1];
  for (int k = 0; k < n_max; ++k) {
    float x[2][kPer];
#pragma unroll
    for (int side = 0; side < 2; ++side) {
      const float* p = slots + static_cast<size_t>(b_lo[side] + k + 2 * item + side) * S::kSlotFloats;
#pragma unroll
      for (int u = 0; u < kPer; ++u) {
        const int e = threadIdx.x + 256 * u;
        x[side][u] = (k < n_slot[side] && e < S::kSlotFloats) ? p[e] : 0.f;
      }
    }
#pragma unroll
    for (int side = 0; side < 2; ++side)
#pragma unroll
      for (int u = 0; u < kPer; ++u)
        if (k < n_slot[side]) v[side][u] += x[side][u];
  }
#pragma unroll
  for (int side = 0; side < 2; ++side)
#pragma unroll
    for (int u = 0; u < kPer; ++u) {
      const int e = threadIdx.x + 256 * u;
      if (e < S::kSlotFloats) g[side][e] = v[side][u];
    }
  __syncthreads();
  // entry (f1, f2) of a side's symmetric feature Gram from its accumulated block pairs
  auto G = [&](int side, int f1, int f2) -> float {
    int I = f1 >> 4, J = f2 >> 4;
    if (I > J) {
      const int t = f1;
      f1 = f2;
      f2 = t;
      I = f1 >> 4;
      J = f2 >> 4;
    }
    const int p = pair_of<RP>(I, J);
    return p < 0 ? 0.f : g[side][p * 256 + (f1 & 15) * 16 + (f2 & 15)];
  };
  // <d_i, d_j>, <d_i, base_j>, <base_i, base_j> with d = hi + lo; features hi_i = i,
  // lo_i = RP + i, base_i = 2 RP + i
  auto dd = [&](int s, int i, int j) {
    return G(s, i, j) + G(s, i, RP + j) + G(s, RP + i, j) + G(s, RP + i, RP + j);
  };
  auto db = [&](int s, int i, int j) { return G(s, i, 2 * RP + j) + G(s, RP + i, 2 * RP + j); };
  auto bb = [&](int s, int i, int j) { return G(s, 2 * RP + i, 2 * RP + j); };
  for (int idx = threadIdx.x; idx < r2 * r2; idx += 256) {
    const int p = idx / r2, q = idx % r2;
    // GB over [B1 - B0 | B0]; GA over [A1 ; A1 - A0]: base first on the A side
    gb[p][q] = p < R ? (q < R ? dd(0, p, q) : db(0, p, q - R)) : (q < R ? db(0, q, p - R) : bb(0, p - R, q - R));
    ga[p][q] = p < R ? (q < R ? bb(1, p, q) : db(1, q - R, p)) : (q < R ? db(1, p - R, q) : dd(1, p - R, q - R));
  }
  __syncthreads();
  double t = 0.0, par = 0.0;
  for (int idx = threadIdx.x; idx < r2 * r2; idx += 256) {
    const int p = idx / r2, q = idx % r2;
    t += static_cast<double>(gb[p][q]) * static_cast<double>(ga[p][q]);  // both symmetric
  }
  if (threadIdx.x < R)
    par = static_cast<double>(gb[threadIdx.x][threadIdx.x]) + static_cast<double>(ga[R + threadIdx.x][R + threadIdx.x]);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    t += __shfl_xor_sync(0xffffffffu, t, o);
    par += __shfl_xor_sync(0xffffffffu, par, o);
  }
  if ((threadIdx.x & 31) == 0) {
    red[0][threadIdx.x >> 5] = t;
    red[1][threadIdx.x >> 5] = par;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    double tt = 0.0, pp = 0.0;
    for (int w = 0; w < 8; ++w) {
      tt += red[0][w];
      pp += red[1][w];
    }
    out_sq[a.items[item].out_index * 2 + 0] = static_cast<float>(tt);
    out_sq[a.items[item].out_index * 2 + 1] = static_cast<float>(pp);
  }
}

template <int R>
cudaError_t launch_rank(const DriftTcArgs& a, float* slots, float* out_sq, cudaStream_t stream) {
  using S = DtShape<R>;
  constexpr int smem = kDtStages * S::kStage + 32 * S::kPairs * 8 * 4;
  static PerDevice once;
  int dev = 0;
  if (once.pending(&dev)) {
    const cudaError_t e =
        cudaFuncSetAttribute(drift_tc_kernel<R>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    once.done(dev);
  }
  drift_tc_kernel<R><<<a.grid, kDtThreads, smem, stream>>>(a, slots);
  drift_tc_final_kernel<R><<<a.n_items, 256, 0, stream>>>(a, slots, out_sq);
  return cudaGetLastError();
}

int slot_floats(int rank) { return rank == 16 ? DtShape<16>::kSlotFloats : DtShape<8>::kSlotFloats; }

}  // namespace

size_t drift_workspace_bytes(int num_sms, int rank, int n_items) {
  const int items = n_items < kDtMaxItems ? n_items : kDtMaxItems;
  const size_t slots = static_cast<size_t>(kDtCtasPerSm) * num_sms + 2 * static_cast<size_t>(items);
  return slots * slot_floats(rank) * sizeof(float);
}

int drift_launches(int n_items) { return 2 * ((n_items + kDtMaxItems - 1) / kDtMaxItems); }

cudaError_t launch_drift(const DriftItem* items, int n_items, int rank, float* slots, int num_sms,
                         float* out_sq, cudaStream_t stream) {
  if (rank != 4 && rank != 8 && rank != 16) return cudaErrorInvalidValue;
  for (int base = 0; base < n_items; base += kDtMaxItems) {
    DriftTcArgs a;
    a.n_items = n_items - base < kDtMaxItems ? n_items - base : kDtMaxItems;
    a.n_segs = 2 * a.n_items;
    a.rank = rank;
    int steps = 0;
    for (int i = 0; i < a.n_items; ++i) {
      a.items[i] = items[base + i];
      for (int side = 0; side < 2; ++side) {
        a.seg_step0[2 * i + side] = steps;
        const int len = side == 0 ? a.items[i].out_dim : a.items[i].in_dim;
        steps += (len + kDtRows - 1) / kDtRows;
      }
    }
    a.seg_step0[a.n_segs] = steps;
    a.total_steps = steps;
    const int want = kDtCtasPerSm * num_sms;
    a.grid = steps < want ? steps : want;
    if (a.grid < 1) continue;
    const cudaError_t e = rank == 16 ? launch_rank<16>(a, slots, out_sq, stream)
                          : rank == 8 ? launch_rank<8>(a, slots, out_sq, stream)
                                      : launch_rank<4>(a, slots, out_sq, stream);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace crf
