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
// RP = max(r, 8) features per part, and the kernel accumulates the block-upper triangle of its
// Gram (16 x 16 blocks).
//
// Data movement: the long dimension of every (item, side) segment is cut into steps of 256
// fragment rows; the steps of all segments are laid end to end and a persistent grid of G CTAs
// takes equal consecutive ranges of them (stream-K). A step is a few contiguous runs of memory:
// the B side's rows, r values wide, are one run per version; the A side's columns are one run
// per version and rank row. A producer warp copies them with 1-D bulk copies (cp.async.bulk)
// that complete on the stage's full mbarrier, up to three steps ahead of the 8 consumer warps,
// which release each stage on its empty mbarrier once they have multiplied it. A
// segment's last, shorter step has the rest of its stage zeroed first. Rank 4 packs two B rows
// into one 16-byte fragment row (features [row 2j | row 2j + 1]); the combine folds the two
// halves of that Gram. Fragments come from ldmatrix loads (transposed for the B side), hi/lo/base
// are built in registers, and each warp accumulates two 16-row slices per step. When its range
// leaves a segment (or ends) the CTA sums its warps in a fixed tree and writes one partial Gram
// to slot (b + seg), unique because a CTA's segments follow the previous CTA's. A combine kernel,
// dependent-launched so that its launch overlaps the Gram kernel's last CTAs, sums each item's
// slots in CTA order and forms tr(GB GA) and the parameter distance in fp64. The result does not
// depend on timing: same inputs, same bits.
#include "common.cuh"
#include "kernels.h"

namespace crf {

namespace {

constexpr int kDtConsumers = 256;         // 8 consumer warps multiply the staged steps
constexpr int kDtThreads = kDtConsumers + 32;  // + 1 producer warp issues the copies
constexpr int kDtRows = 256;              // fragment rows per step: 8 warps x 2 slices x 16
constexpr int kDtSlices = kDtRows / 128;  // 16-row slices per warp and step
constexpr int kDtStages = 3;              // two steps in flight while one is multiplied
constexpr int kDtCtasPerSm = 3;
constexpr int kDtMaxItems = 224;
constexpr int kDtMaxSegs = 2 * kDtMaxItems;
constexpr int kDtAStride = kDtRows * 2 + 16;  // bytes per A row in a stage (+16: no bank conflicts)

struct DriftTcArgs {
  DriftItem items[kDtMaxItems];
  int seg_step0[kDtMaxSegs + 1];  // first step of segment s = 2 * item + side; [n_segs] = total
  int n_items, n_segs, total_steps, grid;
  int n_out;      // (layer, module) entries of out_sq (pairs of floats)
  int zero_mask;  // modules whose entries CTA 0 clears (0: none)
};

template <int R>
struct DtShape {
  static constexpr int RP = R < 8 ? 8 : R;              // features per part (zero padded)
  static constexpr int kPack = RP / R;                  // B rows per fragment row (rank 4: 2)
  static constexpr int kBRowBytes = 2 * RP;             // bytes per fragment row on the B side
  static constexpr int kBFactorRows = kDtRows * kPack;  // B rows per step
  static constexpr int kBVersion = kDtRows * kBRowBytes;
  static constexpr int kAVersion = RP * kDtAStride;
  static constexpr int kVersion = kBVersion > kAVersion ? kBVersion : kAVersion;
  static constexpr int kStage = 2 * kVersion;
  static constexpr int kBlocks = RP == 16 ? 3 : 2;      // 16-feature blocks of [hi|lo|base]
  // block pairs (I <= J) accumulated: the block-upper triangle, except lo x lo for RP = 16 (its
  // entries are below 2^-18 of hi x hi, far under the drift tolerance)
  static constexpr int kPairs = RP == 16 ? 5 : 3;
  static constexpr int kSlotFloats = kPairs * 256;
  static constexpr int kRedFloats = kPairs * 8 * 32;  // one warp's accumulators
  // the combine's scratch: both sides' summed slots, 2 x 8 doubles
  static constexpr int kCombineBytes = 2 * kSlotFloats * 4 + 128;
  static constexpr int kScratch = 4 * kRedFloats * 4;  // the warp-sum tree's first round
  // stages, the tree's scratch, a full and an empty mbarrier per stage, the abort flag
  static constexpr int kSmem = kDtStages * kStage + kScratch + kDtStages * 16 + 16;
};

// (I, J): the 16-feature blocks of accumulated pair p
template <int RP>
__host__ __device__ constexpr int pair_I(int p) { return RP == 16 ? (p < 3 ? 0 : (p == 3 ? 1 : 2)) : (p < 2 ? 0 : 1); }
template <int RP>
__host__ __device__ constexpr int pair_J(int p) { return RP == 16 ? (p < 3 ? p : 2) : (p < 2 ? p : 1); }

// 1-D bulk copy global -> this CTA's shared memory, completing `bytes` on mbarrier `bar`. Both
// addresses 16-byte aligned, `bytes` a positive multiple of 16.
__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
      "l"(src), "r"(bytes), "r"(bar)
      : "memory");
}

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

// D += A B for one m16n8k16 bf16 tile with fp32 accumulation. Not volatile: it only reads and
// writes registers, so the compiler may interleave the MMAs of the two slices a warp multiplies.
__device__ __forceinline__ void mma_bf16(float (&c)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7},"
      " {%8, %9}, {%0, %1, %2, %3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
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

// The segment of step x, searched forward from segment s (segments are visited in order).
__device__ __forceinline__ int seg_of(const DriftTcArgs& a, int s, int x) {
  while (s + 1 < a.n_segs && x >= a.seg_step0[s + 1]) ++s;
  return s;
}

// What the producer needs of the segment it loads, read from the arguments once per segment.
struct ProdSeg {
  int seg = -1, side = 0, len = 0, step0 = 0, next0 = 0;
  const __nv_bfloat16 *p1 = nullptr, *p0 = nullptr;  // version 1 / version 0 of this side

  __device__ __forceinline__ void at(const DriftTcArgs& a, int x) {
    if (seg >= 0 && x < next0) return;
    seg = seg_of(a, seg < 0 ? 0 : seg, x);
    side = seg & 1;
    const DriftItem& it = a.items[seg >> 1];
    len = side == 0 ? it.out_dim : it.in_dim;
    step0 = a.seg_step0[seg];
    next0 = a.seg_step0[seg + 1];
    p1 = side == 0 ? it.B1 : it.A1;
    p0 = side == 0 ? it.B0 : it.A0;
  }
};

// 16-byte cp.async global -> shared, zero-filled when !valid (no bytes read).
__device__ __forceinline__ void cp_async16_zfill(uint32_t dst, const void* src, bool valid) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(valid ? 16 : 0)
               : "memory");
}

__device__ __forceinline__ void st_shared_zero16(uint32_t addr) {
  asm volatile("st.shared.v4.u32 [%0], {%1, %1, %1, %1};" ::"r"(addr), "r"(0u) : "memory");
}

// Producer warp, every lane: the copies of step x into stage `st`, completing on `bar` (32 arrivals a
// phase). B side: rows [r0, r0 + rows) of both versions, one bulk copy each (lane 0's arrival
// expects their bytes; each lane's arrival releases its own zero stores of a shorter last step).
// A side: columns [c0, c0 + cols) of every rank row of both versions, by cp.async. Rows and
// columns come in multiples of 8 (the host checks every width), so every run is a multiple of
// 16 bytes and starts 16-byte aligned.
template <int R>
__device__ __forceinline__ void issue_step(const ProdSeg& ps, int x, uint32_t st, uint64_t* bar) {
  using S = DtShape<R>;
  const int lane = threadIdx.x & 31;
  const int j = x - ps.step0;
  const uint32_t bar_a = smem_u32(bar);
  const int len = ps.len;
  if (ps.side == 0) {
    const int r0 = j * S::kBFactorRows;
    const int rows = len - r0 < S::kBFactorRows ? len - r0 : S::kBFactorRows;
    const uint32_t bytes = static_cast<uint32_t>(rows) * R * 2;
    if (bytes < static_cast<uint32_t>(S::kBVersion)) {
      for (uint32_t o = bytes + lane * 16; o < static_cast<uint32_t>(S::kBVersion); o += 32 * 16) {
        st_shared_zero16(st + o);
        st_shared_zero16(st + S::kVersion + o);
      }
    }
    __syncwarp();
    if (lane == 0)
      mbar_arrive_expect_tx(bar, 2 * bytes);
    else
      mbar_arrive(bar);
    if (lane < 2)
      bulk_g2s(st + lane * S::kVersion, (lane == 0 ? ps.p1 : ps.p0) + static_cast<size_t>(r0) * R, bytes, bar_a);
  } else {
    // A side: lane l copies 16-byte chunk l of every rank row and version (one 512-byte run of
    // a row per instruction); chunks past the step's columns are zero-filled. Each lane's arrival
    // fires when its own copies have landed.
    const int c0 = j * kDtRows;
    const int cols = len - c0 < kDtRows ? len - c0 : kDtRows;
    const bool in = lane * 8 < cols;  // columns come in multiples of 8: a chunk is in or out
    const uint32_t dst = st + lane * 16;
    const __nv_bfloat16* src1 = ps.p1 + c0 + (in ? lane * 8 : 0);
    const __nv_bfloat16* src0 = ps.p0 + c0 + (in ? lane * 8 : 0);
#pragma unroll 4
    for (int f = 0; f < R; ++f) {
      cp_async16_zfill(dst + f * kDtAStride, src1 + static_cast<size_t>(f) * len, in);
      cp_async16_zfill(dst + S::kVersion + f * kDtAStride, src0 + static_cast<size_t>(f) * len, in);
    }
    asm volatile("cp.async.mbarrier.arrive.noinc.shared::cta.b64 [%0];" ::"r"(bar_a) : "memory");
  }
}

// This warp's fragments of one 16-row slice of a staged step, both versions:
// {m0, m1, m2, m3} (RP = 8: m0, m2).
template <int R, int SIDE>
__device__ __forceinline__ void load_frags(uint32_t st, int row0, uint32_t (&f1)[4], uint32_t (&f0)[4]) {
  using S = DtShape<R>;
  constexpr int RP = S::RP;
  const int lane = threadIdx.x & 31;
  const int m = lane >> 3, i = lane & 7;
  if constexpr (SIDE == 0) {
    // X[o][f] rows: matrix m covers rows row0 + (m >> 1) * 8 .. and features (m & 1) * 8 ..
    if constexpr (RP == 16) {
      const uint32_t off = (row0 + (m >> 1) * 8 + i) * S::kBRowBytes + (m & 1) * 16;
      ldsm_x4_t(st + off, f1[0], f1[1], f1[2], f1[3]);
      ldsm_x4_t(st + S::kVersion + off, f0[0], f0[1], f0[2], f0[3]);
    } else {
      const uint32_t off = (row0 + (m & 1) * 8 + i) * S::kBRowBytes;
      ldsm_x2_t(st + off, f1[0], f1[2]);
      ldsm_x2_t(st + S::kVersion + off, f0[0], f0[2]);
    }
  } else {
    // Xt[f][c] rows: matrix m covers features (m & 1) * 8 .. and columns row0 + (m >> 1) * 8 ..
    if constexpr (RP == 16) {
      const uint32_t off = ((m & 1) * 8 + i) * kDtAStride + (row0 + (m >> 1) * 8) * 2;
      ldsm_x4(st + off, f1[0], f1[1], f1[2], f1[3]);
      ldsm_x4(st + S::kVersion + off, f0[0], f0[1], f0[2], f0[3]);
    } else {
      const uint32_t off = i * kDtAStride + (row0 + (m & 1) * 8) * 2;
      ldsm_x2(st + off, f1[0], f1[2]);
      ldsm_x2(st + S::kVersion + off, f0[0], f0[2]);
      if constexpr (R < RP) {
        // lane holds feature lane / 4: rank rows R.. of the stage are not this adapter's
        if (lane >= 4 * R) f1[0] = f1[2] = f0[0] = f0[2] = 0u;
      }
    }
  }
}

// One slice's fragments into the Gram accumulators: [hi | lo | base] built in registers
// (base: B0 on the B side, A1 on the A side), then the accumulated block pairs.
template <int R, int SIDE>
__device__ __forceinline__ void mma_frags(const uint32_t (&f1)[4], const uint32_t (&f0)[4],
                                          float (&acc)[DtShape<R>::kPairs][2][4]) {
  using S = DtShape<R>;
  constexpr int RP = S::RP;
  uint32_t blk[S::kBlocks][4];
  if constexpr (RP == 16) {
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      split_diff(f1[r], f0[r], blk[0][r], blk[1][r]);
      blk[2][r] = SIDE == 0 ? f0[r] : f1[r];
    }
  } else {
    // block 0 = [hi (8 features) | lo (8)], block 1 = [base (8) | zeros]
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int r = 2 * h;
      split_diff(f1[r], f0[r], blk[0][r], blk[0][r + 1]);
      blk[1][r] = SIDE == 0 ? f0[r] : f1[r];
      blk[1][r + 1] = 0u;
    }
  }
#pragma unroll
  for (int p = 0; p < S::kPairs; ++p) {
    const int I = pair_I<RP>(p), J = pair_J<RP>(p);
    mma_bf16(acc[p][0], blk[I], blk[J][0], blk[J][2]);
    mma_bf16(acc[p][1], blk[I], blk[J][1], blk[J][3]);
  }
}

// Named barrier over the 8 consumer warps (the producer warp runs its own loop).
__device__ __forceinline__ void consumers_sync() {
  asm volatile("bar.sync 1, %0;" ::"n"(kDtConsumers) : "memory");
}

// Consumers: steps [x, end) of one segment of side SIDE. Each waits for its stage, multiplies
// it and releases it to the producer (one arrival per warp). False (x left at the failed step)
// when a wait times out.
template <int R, int SIDE>
__device__ __forceinline__ bool run_steps(int& x, int end, int& stage, uint32_t& phase, uint64_t* full,
                                          uint64_t* empty, uint32_t stage0, volatile int* abort_flag,
                                          int* status, float (&acc)[DtShape<R>::kPairs][2][4]) {
  using S = DtShape<R>;
  const int warp = threadIdx.x >> 5;
  for (; x < end; ++x) {
    if (!mbar_wait(full + stage, phase, abort_flag, status)) return false;
    const uint32_t st = stage0 + stage * S::kStage;
    // both slices' fragments into registers, then the stage goes back to the producer before
    // they are multiplied
    uint32_t f1[kDtSlices][4], f0[kDtSlices][4];
#pragma unroll
    for (int sl = 0; sl < kDtSlices; ++sl) load_frags<R, SIDE>(st, (warp * kDtSlices + sl) * 16, f1[sl], f0[sl]);
    __syncwarp();
    if ((threadIdx.x & 31) == 0) mbar_arrive(empty + stage);
#pragma unroll
    for (int sl = 0; sl < kDtSlices; ++sl) mma_frags<R, SIDE>(f1[sl], f0[sl], acc);
    if (++stage == kDtStages) {
      stage = 0;
      phase ^= 1u;
    }
  }
  return true;
}

// Producer warp: steps [x0, x1) into the stages in turn, each once the consumers have released
// the stage's previous step; then it waits until they have released the last ones. On a timeout
// (its own or the consumers') it waits, within the same limit, for the copies it has issued, so
// none is in flight when the CTA's shared memory goes.
template <int R>
__device__ __forceinline__ void produce(const DriftTcArgs& a, int x0, int x1, uint64_t* full,
                                        uint64_t* empty, uint32_t stage0, volatile int* abort_flag,
                                        int* status) {
  using S = DtShape<R>;
  ProdSeg ps;
  int ls = 0, issued = 0;
  bool ok = true;
  for (int lx = x0; lx < x1; ++lx) {
    const int i = lx - x0;
    if (i >= kDtStages && !mbar_wait(empty + ls, static_cast<uint32_t>((i / kDtStages - 1) & 1), abort_flag, status)) {
      ok = false;
      break;
    }
    ps.at(a, lx);
    issue_step<R>(ps, lx, stage0 + ls * S::kStage, full + ls);
    ++issued;
    if (++ls == kDtStages) ls = 0;
  }
  for (int i = issued > kDtStages ? issued - kDtStages : 0; ok && i < issued; ++i)
    ok = mbar_wait(empty + i % kDtStages, static_cast<uint32_t>((i / kDtStages) & 1), abort_flag, status);
  if (ok) return;
  if ((threadIdx.x & 31) == 0) {
    // the last use of every stage: step issued - 1 - k sits in stage (issued - 1 - k) % S
    const unsigned long long t0 = globaltimer_ns();
    for (int k = 0; k < kDtStages && k < issued; ++k) {
      const int i = issued - 1 - k;
      while (!mbar_try_wait(full + i % kDtStages, static_cast<uint32_t>((i / kDtStages) & 1)) &&
             globaltimer_ns() - t0 < kWaitLimitNs) {
      }
    }
  }
}

// Slots [b_lo, b_lo + n_slot) of segment `seg`: the CTAs whose step ranges meet it.
__device__ __forceinline__ void seg_slots(const DriftTcArgs& a, int seg, int& b_lo, int& n_slot) {
  const long long s0 = a.seg_step0[seg], s1 = a.seg_step0[seg + 1] - 1;
  b_lo = static_cast<int>(((s0 + 1) * a.grid - 1) / a.total_steps);
  n_slot = static_cast<int>(((s1 + 1) * a.grid - 1) / a.total_steps) - b_lo + 1;
}

// Entries of one side's difference/base Grams from its accumulated block pairs `gs`
// ([pair][16][16]): features hi_i, lo_i (d = hi + lo) and base_i.
//   DD(i, j) = <d_i, d_j>,  DB(i, j) = <d_i, base_j>,  BB(i, j) = <base_i, base_j>.
// RP = 16: blocks hi | lo | base, pairs (hi,hi) (hi,lo) (hi,base) (lo,base) (base,base), lo x lo
// not accumulated. RP = 8: blocks [hi | lo] | [base | 0], pairs (0,0) (0,1) (1,1).
template <int RP>
struct SideGram {
  const float* gs;
  __device__ __forceinline__ float P(int k, int r, int c) const { return gs[k * 256 + r * 16 + c]; }
  __device__ __forceinline__ float DD(int i, int j) const {
    if constexpr (RP == 16) return P(0, i, j) + P(1, i, j) + P(1, j, i);
    else return P(0, i, j) + P(0, i, 8 + j) + P(0, 8 + i, j) + P(0, 8 + i, 8 + j);
  }
  __device__ __forceinline__ float DB(int i, int j) const {
    if constexpr (RP == 16) return P(2, i, j) + P(3, i, j);
    else return P(1, i, j) + P(1, 8 + i, j);
  }
  __device__ __forceinline__ float BB(int i, int j) const { return RP == 16 ? P(4, i, j) : P(2, i, j); }
};

// One item, by 256 threads: both segments' slots summed in CTA order, then
//   tr(GB GA) = sum_ij DD_B(i,j) BB_A(i,j) + BB_B(i,j) DD_A(i,j) + 2 DB_B(i,j) DB_A(j,i)
// (GB = [[DD_B, DB_B], [DB_B^T, BB_B]] over [B1 - B0 | B0]; GA = [[BB_A, DB_A^T], [DB_A, DD_A]]
// over [A1 ; A1 - A0]) and the parameter distance sum_i DD_B(i,i) + DD_A(i,i): one (i, j) term
// per thread in fp64 from fp32 Gram entries, reduced in a fixed order, written to the item's
// out_sq pair. Rank 4 adds the B side's two packed halves (fragment features i and i + 4).
// `buf` is shared scratch of kCombineBytes. The slots come from other CTAs: read through L2.
template <int R>
__device__ void combine_item(const DriftTcArgs& a, int item, const float* __restrict__ slots,
                             float* __restrict__ out_sq, uint8_t* buf) {
  using S = DtShape<R>;
  constexpr int RP = S::RP;
  float (*g)[S::kSlotFloats] = reinterpret_cast<float (*)[S::kSlotFloats]>(buf);
  double (*red)[8] = reinterpret_cast<double (*)[8]>(buf + S::kCombineBytes - 128);
  // every load of up to eight slot offsets (both sides, all of a thread's entries) is issued
  // before any of them is added; the adds keep CTA order
  constexpr int kPer = (S::kSlotFloats + kDtConsumers - 1) / kDtConsumers;
  constexpr int kBatch = 8;
  int b_lo[2], n_slot[2];
  for (int side = 0; side < 2; ++side) seg_slots(a, 2 * item + side, b_lo[side], n_slot[side]);
  float v[2][kPer];
#pragma unroll
  for (int side = 0; side < 2; ++side)
#pragma unroll
    for (int u = 0; u < kPer; ++u) v[side][u] = 0.f;
  const int n_max = n_slot[0] > n_slot[1] ? n_slot[0] : n_slot[1];
  for (int k0 = 0; k0 < n_max; k0 += kBatch) {
    float x[kBatch][2][kPer];
#pragma unroll
    for (int kk = 0; kk < kBatch; ++kk)
#pragma unroll
      for (int side = 0; side < 2; ++side) {
        const int k = k0 + kk;
        const float* p = slots + static_cast<size_t>(b_lo[side] + k + 2 * item + side) * S::kSlotFloats;
#pragma unroll
        for (int u = 0; u < kPer; ++u) {
          const int e = threadIdx.x + kDtConsumers * u;
          x[kk][side][u] = (k < n_slot[side] && e < S::kSlotFloats) ? __ldcg(p + e) : 0.f;
        }
      }
#pragma unroll
    for (int kk = 0; kk < kBatch; ++kk)
#pragma unroll
      for (int side = 0; side < 2; ++side)
#pragma unroll
        for (int u = 0; u < kPer; ++u)
          if (k0 + kk < n_slot[side]) v[side][u] += x[kk][side][u];
  }
#pragma unroll
  for (int side = 0; side < 2; ++side)
#pragma unroll
    for (int u = 0; u < kPer; ++u) {
      const int e = threadIdx.x + kDtConsumers * u;
      if (e < S::kSlotFloats) g[side][e] = v[side][u];
    }
  consumers_sync();
  const SideGram<RP> gB{g[0]}, gA{g[1]};
  double t = 0.0, par = 0.0;
  if (threadIdx.x < R * R) {
    const int i = threadIdx.x / R, j = threadIdx.x % R;
    float dd0 = gB.DD(i, j), db0 = gB.DB(i, j), bb0 = gB.BB(i, j);
    if constexpr (R < RP) {
      dd0 += gB.DD(i + R, j + R);
      db0 += gB.DB(i + R, j + R);
      bb0 += gB.BB(i + R, j + R);
    }
    const float dd1 = gA.DD(i, j), db1t = gA.DB(j, i), bb1 = gA.BB(i, j);
    t = static_cast<double>(dd0) * bb1 + static_cast<double>(bb0) * dd1 + 2.0 * (static_cast<double>(db0) * db1t);
    if (i == j) par = static_cast<double>(dd0) + static_cast<double>(dd1);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    t += __shfl_xor_sync(0xffffffffu, t, o);
    par += __shfl_xor_sync(0xffffffffu, par, o);
  }
  if ((threadIdx.x & 31) == 0) {
    red[0][threadIdx.x >> 5] = t;
    red[1][threadIdx.x >> 5] = par;
  }
  consumers_sync();
  if (threadIdx.x == 0) {
    double tt = 0.0, pp = 0.0;
    for (int w = 0; w < kDtConsumers / 32; ++w) {
      tt += red[0][w];
      pp += red[1][w];
    }
    out_sq[a.items[item].out_index * 2 + 0] = static_cast<float>(tt);
    out_sq[a.items[item].out_index * 2 + 1] = static_cast<float>(pp);
  }
}

template <int R>
__global__ void __launch_bounds__(kDtThreads, kDtCtasPerSm)
    drift_tc_kernel(const __grid_constant__ DriftTcArgs a, float* __restrict__ slots, int* status) {
  using S = DtShape<R>;
  extern __shared__ __align__(128) uint8_t dt_smem[];
  uint8_t* scratch = dt_smem + kDtStages * S::kStage;
  float* red = reinterpret_cast<float*>(scratch);  // [4][kPairs * 8][32]: warp partials
  uint64_t* full = reinterpret_cast<uint64_t*>(scratch + S::kScratch);
  uint64_t* empty = full + kDtStages;
  volatile int* abort_flag = reinterpret_cast<volatile int*>(empty + kDtStages);
  const uint32_t stage0 = smem_u32(dt_smem);
  // the combine kernel may become resident as this grid's CTAs retire; it waits for the grid
  griddep_launch_dependents();
  const int b = blockIdx.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int x0 = static_cast<int>((static_cast<long long>(b) * a.total_steps) / a.grid);
  const int x1 = static_cast<int>((static_cast<long long>(b + 1) * a.total_steps) / a.grid);
  if (x0 >= x1) return;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kDtStages; ++s) {
      mbar_init(full + s, 32);                  // the producer warp's lanes
      mbar_init(empty + s, kDtConsumers / 32);  // one lane per consumer warp
    }
    *abort_flag = 0;
    fence_barrier_init();
  }
  __syncthreads();
  if (warp == kDtConsumers / 32) {
    produce<R>(a, x0, x1, full, empty, stage0, abort_flag, status);
    return;
  }

  float acc[S::kPairs][2][4];
#pragma unroll
  for (int q = 0; q < S::kPairs; ++q)
#pragma unroll
    for (int h = 0; h < 2; ++h)
#pragma unroll
      for (int v = 0; v < 4; ++v) acc[q][h][v] = 0.f;

  int x = x0, seg = seg_of(a, 0, x0), stage = 0;  // the step, segment and stage being multiplied
  uint32_t phase = 0;
  while (x < x1) {
    seg = seg_of(a, seg, x);
    const int next0 = a.seg_step0[seg + 1];
    const int end = x1 < next0 ? x1 : next0;
    const bool ok = (seg & 1) == 0
                        ? run_steps<R, 0>(x, end, stage, phase, full, empty, stage0, abort_flag, status, acc)
                        : run_steps<R, 1>(x, end, stage, phase, full, empty, stage0, abort_flag, status, acc);
    // the producer drains the copies in flight; a warp that got past a wait another warp gave
    // up on stops here too, before the flush's barriers
    if (!ok || *abort_flag) return;
    // the warps' partial Grams summed in a fixed tree ((w0 + w4) + (w2 + w6)) + ((w1 + w5) +
    // (w3 + w7)), then written as one slot
#pragma unroll 1
    for (int h = kDtConsumers / 64; h >= 1; h >>= 1) {
      if (warp >= h && warp < 2 * h) {
#pragma unroll
        for (int q = 0; q < S::kPairs; ++q)
#pragma unroll
          for (int hh = 0; hh < 2; ++hh)
#pragma unroll
            for (int v = 0; v < 4; ++v) red[((warp - h) * S::kPairs * 8 + q * 8 + hh * 4 + v) * 32 + lane] = acc[q][hh][v];
      }
      consumers_sync();
      if (warp < h) {
#pragma unroll
        for (int q = 0; q < S::kPairs; ++q)
#pragma unroll
          for (int hh = 0; hh < 2; ++hh)
#pragma unroll
            for (int v = 0; v < 4; ++v) acc[q][hh][v] += red[(warp * S::kPairs * 8 + q * 8 + hh * 4 + v) * 32 + lane];
      }
      consumers_sync();
    }
    if (warp == 0) {
#pragma unroll
      for (int q = 0; q < S::kPairs; ++q)
#pragma unroll
        for (int hh = 0; hh < 2; ++hh)
#pragma unroll
          for (int v = 0; v < 4; ++v) red[(q * 8 + hh * 4 + v) * 32 + lane] = acc[q][hh][v];
    }
    consumers_sync();
    float* out = slots + static_cast<size_t>(b + seg) * S::kSlotFloats;
    for (int e = threadIdx.x; e < S::kSlotFloats; e += kDtConsumers) {
      const int q = e >> 8, rr = (e >> 4) & 15, cc = e & 15;
      const int ln = (rr & 7) * 4 + ((cc & 7) >> 1);
      const int v = (rr >> 3) * 2 + (cc & 1);
      out[e] = red[(q * 8 + (cc >> 3) * 4 + v) * 32 + ln];
    }
#pragma unroll
    for (int q = 0; q < S::kPairs; ++q)
#pragma unroll
      for (int hh = 0; hh < 2; ++hh)
#pragma unroll
        for (int v = 0; v < 4; ++v) acc[q][hh][v] = 0.f;
    consumers_sync();  // `red` is read before the next flush overwrites it
  }
}

// One 256-thread block per item, dependent-launched after the Gram kernel: it waits for that
// grid, then combines the item's slots. Block 0 also clears the entries of modules without an
// adapter.
template <int R>
__global__ void __launch_bounds__(kDtConsumers) drift_tc_final_kernel(const __grid_constant__ DriftTcArgs a,
                                                                      const float* __restrict__ slots,
                                                                      float* __restrict__ out_sq) {
  using S = DtShape<R>;
  __shared__ __align__(16) uint8_t buf[S::kCombineBytes];
  griddep_wait();
  if (blockIdx.x == 0 && a.zero_mask)
    for (int e = threadIdx.x; e < a.n_out; e += kDtConsumers)
      if ((a.zero_mask >> (e % 7)) & 1) {
        out_sq[2 * e] = 0.f;
        out_sq[2 * e + 1] = 0.f;
      }
  combine_item<R>(a, blockIdx.x, slots, out_sq, buf);
}

template <int R>
cudaError_t launch_rank(const DriftTcArgs& a, float* slots, float* out_sq, int* status, cudaStream_t stream) {
  using S = DtShape<R>;
  static PerDevice once;
  int dev = 0;
  if (once.pending(&dev)) {
    const cudaError_t e =
        cudaFuncSetAttribute(drift_tc_kernel<R>, cudaFuncAttributeMaxDynamicSharedMemorySize, S::kSmem);
    if (e != cudaSuccess) return e;
    once.done(dev);
  }
  // the Gram kernel is not dependent-launched: it overwrites the slots that the combine kernel
  // of an earlier call on this stream reads
  drift_tc_kernel<R><<<a.grid, kDtThreads, S::kSmem, stream>>>(a, slots, status);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  PdlScope pdl;
  return launch_kernel(drift_tc_final_kernel<R>, dim3(a.n_items), dim3(kDtConsumers), 0, stream, a,
                       static_cast<const float*>(slots), out_sq);
}

int slot_floats(int rank) { return rank == 16 ? DtShape<16>::kSlotFloats : DtShape<8>::kSlotFloats; }

}  // namespace

size_t drift_workspace_bytes(int num_sms, int rank, int n_items) {
  const int items = n_items < kDtMaxItems ? n_items : kDtMaxItems;
  const size_t slots = static_cast<size_t>(kDtCtasPerSm) * num_sms + 2 * static_cast<size_t>(items);
  return slots * slot_floats(rank) * sizeof(float);
}

int drift_launches(int n_items) { return 2 * ((n_items + kDtMaxItems - 1) / kDtMaxItems); }

cudaError_t launch_drift(const DriftItem* items, int n_items, int rank, int n_out, int adapted_mask,
                         void* workspace, int num_sms, float* out_sq, int* status, cudaStream_t stream) {
  if (rank != 4 && rank != 8 && rank != 16) return cudaErrorInvalidValue;
  float* slots = static_cast<float*>(workspace);
  const int b_rows = rank == 4 ? DtShape<4>::kBFactorRows : kDtRows;  // B rows per step
  for (int base = 0; base < n_items; base += kDtMaxItems) {
    DriftTcArgs a;
    a.n_items = n_items - base < kDtMaxItems ? n_items - base : kDtMaxItems;
    a.n_segs = 2 * a.n_items;
    a.n_out = n_out;
    a.zero_mask = base == 0 ? (~adapted_mask & 0x7f) : 0;
    int steps = 0;
    for (int i = 0; i < a.n_items; ++i) {
      a.items[i] = items[base + i];
      for (int side = 0; side < 2; ++side) {
        a.seg_step0[2 * i + side] = steps;
        const int len = side == 0 ? a.items[i].out_dim : a.items[i].in_dim;
        const int per = side == 0 ? b_rows : kDtRows;
        steps += (len + per - 1) / per;
      }
    }
    a.seg_step0[a.n_segs] = steps;
    a.total_steps = steps;
    const int want = kDtCtasPerSm * num_sms;
    a.grid = steps < want ? steps : want;
    if (a.grid < 1) continue;
    const cudaError_t e = rank == 16 ? launch_rank<16>(a, slots, out_sq, status, stream)
                          : rank == 8 ? launch_rank<8>(a, slots, out_sq, status, stream)
                                      : launch_rank<4>(a, slots, out_sq, status, stream);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace crf
