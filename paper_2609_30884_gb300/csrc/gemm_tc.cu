// Persistent tcgen05 GEMM for sm_103a with the unmerged LoRA product and fused epilogues.
//
//   D[256 x 256] = A[256 x K] * B[256 x K]^T  (+ XA[256 x 64] * BL^T)
//
// A cluster of two CTAs on one TPC works on a 256 x 256 tile with cta_group::2 MMAs. Each CTA
// stages its own 128 rows of A and its own half of the B rows, so the operand bytes each SM
// pulls through L2 per FLOP are two thirds of the single-CTA 128 x 256 tile's. The even CTA
// issues the MMAs; both CTAs hold 128 accumulator lanes in their own TMEM and drain them through
// the same epilogue.
//
// Per CTA: warp 0 loads operands into a STAGES-deep shared-memory ring (TMA, issued by one lane),
// warp 1 owns TMEM (two accumulators, so the epilogue of tile i overlaps the main loop of tile
// i+1) and, in the MMA-issuing CTA, issues tcgen05.mma from one thread; warps 2..5 drain the
// accumulator (one TMEM lane = one output row per thread) through the fused epilogue. Operands
// are bf16, K-major, staged with 128-byte swizzle; accumulation is fp32 in TMEM.
//
// The adapter term (alpha/r) (x A^T) B^T of every adapted projection (Eq. S3, W = W0 + (alpha/r)
// B A kept unmerged) is computed in the same launch, on the operand tiles already staged:
//  - the first output tile of each 256-row block (its XA tile) also accumulates x A^T for the
//    GEMM's adapted modules (N = 16 per module, B operand = the LoRA A rows, staged beside the W
//    rows) into the other accumulator's first columns, which the epilogue of the previous tile has
//    drained by then. Its epilogue warps store that product, scaled, as a bf16 pair [hi | lo] per
//    module (16 + 16 columns of the XA buffer) and count themselves done in the row block's ready
//    word;
//  - every output tile of an adapted module adds one 64-wide K block: A side = the XA columns of
//    its row block (the XA tile writes them into its own stage; the others copy them once the
//    ready word shows both CTAs done), B side = BX, the module's B rows twice over ([B | B],
//    against [hi | lo]) under the K steps of its slot and zeros under the other slot, so one K
//    block serves two stacked modules and the two halves of a pair alike. The RMSNorm launch
//    before the layer's projections builds the BX rows.
// XA tiles run first, one per unit, ahead of the other tiles of their row block, so those rarely
// wait; the wait is bounded like every other. x is read once: the XA product needs no pass of its
// own.
#include "common.cuh"
#include "kernels.h"

#include <algorithm>
#include <cstdio>
#include <cstdlib>
#include <cstring>

namespace crf {

namespace {

constexpr int BM = 128;
constexpr int BK = 64;
constexpr int kRasterGroup = 8;
constexpr int kThreads = 192;

struct GemmArgs {
  CUtensorMap tmA;
  CUtensorMap tmB[3];
  CUtensorMap tmXA;
  CUtensorMap tmLA[3];  // LoRA A of XA slot j: the B operand of the XA product
  CUtensorMap tmBX[3];  // BX rows of map index i: the B side of the LoRA K block
  int M, K, num_kb;
  int ngroups, nseg;
  int group_tiles[3];
  int group_cols[3];
  int ext_on[3];      // per group: tile has the LoRA K block
  int ext_steps[3];   // per group: K = 16 steps of that block that carry data
  int xa_base[3];     // per group: first XA column of that block
  int row_tiles, total_n, total_tiles;
  int n_slots;        // adapted modules (XA slots); 0: no XA product
  int xa_n;           // N of the XA product: 16 per slot, two CTA halves of 16 x slots_per_cta
  int xa_lead;        // XA tiles placed before every other tile (the rest follow their row block)
  int rank;
  __nv_bfloat16* xa;
  int* xa_flags;
  int epi;
  float scale;
  __nv_bfloat16* out;
  int ldo;
  const __nv_bfloat16* resid;
  int ld_resid;
  const __nv_bfloat16* bias[3];
  const float2* rope;
  int head_dim, n_kv_heads;
  __nv_bfloat16* qbuf;
  int ldq;
  __nv_bfloat16* kpages;
  __nv_bfloat16* vpages;
  ReqTable req;
  int* status;
  const int* abort;
};

struct Tile {
  int m_blk, g, n_loc;
  bool xa;  // the row block's first output tile, which also forms its XA product
};

// Output tiles run in bands of kRasterGroup column tiles over every row block (the band's B
// rows stay in L2). With an adapter, band 0 is reordered so that each row block's first tile
// (its XA tile) runs ahead of the block's other band-0 tiles: the first `lead` XA tiles, then
// per row block m the XA tile of m + lead followed by m's other band-0 tiles (lead = all row
// blocks puts every XA tile first).
__device__ __forceinline__ Tile decode_tile(int t, const GemmArgs& a) {
  Tile r;
  r.xa = false;
  if (a.n_slots > 0) {
    const int w0 = min(kRasterGroup, a.total_n);
    const int lead = min(a.xa_lead, a.row_tiles);
    const int g1 = a.row_tiles - lead;  // row blocks whose other tiles follow an XA tile
    if (t < lead) {
      t = t * w0;  // the plain order's index of tile (t, 0)
    } else if (t - lead < g1 * w0) {
      const int u = t - lead;
      const int m = u / w0, i = u - m * w0;
      t = i == 0 ? (m + lead) * w0 : m * w0 + i;
    } else if (t - lead - g1 * w0 < lead * (w0 - 1)) {
      const int v = t - lead - g1 * w0;
      const int m = g1 + v / (w0 - 1);
      t = m * w0 + 1 + v % (w0 - 1);
    }  // else: the later bands keep their plain index
  }
  const int band_tiles = a.row_tiles * kRasterGroup;
  const int band = t / band_tiles;
  const int idx = t - band * band_tiles;
  const int n0 = band * kRasterGroup;
  const int width = min(kRasterGroup, a.total_n - n0);
  r.m_blk = idx / width;
  int n = n0 + (idx - r.m_blk * width);
  r.xa = a.n_slots > 0 && n == 0;
  int g = 0;
  while (g < a.ngroups - 1 && n >= a.group_tiles[g]) {
    n -= a.group_tiles[g];
    ++g;
  }
  r.g = g;
  r.n_loc = n;
  return r;
}

__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32"
      " {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
}

__device__ __forceinline__ void store16_bf16(__nv_bfloat16* dst, const float (&v)[16]) {
  uint4 w0, w1;
  w0.x = pack_bf16(v[0], v[1]);
  w0.y = pack_bf16(v[2], v[3]);
  w0.z = pack_bf16(v[4], v[5]);
  w0.w = pack_bf16(v[6], v[7]);
  w1.x = pack_bf16(v[8], v[9]);
  w1.y = pack_bf16(v[10], v[11]);
  w1.z = pack_bf16(v[12], v[13]);
  w1.w = pack_bf16(v[14], v[15]);
  reinterpret_cast<uint4*>(dst)[0] = w0;
  reinterpret_cast<uint4*>(dst)[1] = w1;
}

// Store the first `n` (<= 16) values; n == 16 takes the vector path.
__device__ __forceinline__ void store_bf16_n(__nv_bfloat16* dst, const float (&v)[16], int n) {
  if (n >= 16) {
    store16_bf16(dst, v);
  } else {
#pragma unroll
    for (int j = 0; j < 16; ++j)
      if (j < n) dst[j] = __float2bfloat16_rn(v[j]);
  }
}

__device__ __forceinline__ void load16_bf16(const __nv_bfloat16* src, float (&v)[16]) {
  const uint4 w0 = reinterpret_cast<const uint4*>(src)[0];
  const uint4 w1 = reinterpret_cast<const uint4*>(src)[1];
  const uint32_t w[8] = {w0.x, w0.y, w0.z, w0.w, w1.x, w1.y, w1.z, w1.w};
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    v[2 * j] = bf16_lo(w[j]);
    v[2 * j + 1] = bf16_hi(w[j]);
  }
}

// Find the request and position of batched row `row`; returns false if none.
__device__ __forceinline__ bool row_lookup(const ReqTable& rt, int row, int& pos,
                                           const int32_t*& pt) {
  for (int i = 0; i < rt.n; ++i) {
    const int r0 = rt.row0[i];
    if (row >= r0 && row < r0 + rt.len[i]) {
      pos = row - r0;
      pt = rt.page_table[i];
      return true;
    }
  }
  return false;
}

template <int BN, int EPI>
__device__ __forceinline__ void epilogue_tile(const GemmArgs& a, const Tile& tl, uint32_t tacc,
                                              int row) {
  const bool row_ok = row < a.M;
  uint32_t r0[16], r1[16];
  float v[16], w[16];

  if constexpr (EPI == kEpiResid) {
    const int col0 = tl.n_loc * BN;
    const int ncols = a.group_cols[tl.g];
    // residual chunk c + 16 is requested while chunk c is drained: its load latency overlaps
    auto load_resid = [&](int col, float (&dst)[16]) {
      const int n = min(16, ncols - col);
      if (n >= 16) {
        load16_bf16(a.resid + (size_t)row * a.ld_resid + col, dst);
      } else {
#pragma unroll
        for (int j = 0; j < 16; ++j)
          dst[j] = j < n ? __bfloat162float(a.resid[(size_t)row * a.ld_resid + col + j]) : 0.f;
      }
    };
    float wn[16];
    if (row_ok && col0 < ncols) load_resid(col0, w);
#pragma unroll 1
    for (int c = 0; c < BN; c += 16) {
      tmem_ld16(tacc + c, r0);
      const bool more = row_ok && c + 16 < BN && col0 + c + 16 < ncols;
      if (more) load_resid(col0 + c + 16, wn);
      tmem_ld_wait();
      const int col = col0 + c;
      if (!row_ok || col >= ncols) continue;
#pragma unroll
      for (int j = 0; j < 16; ++j) v[j] = w[j] + __uint_as_float(r0[j]);
      store_bf16_n(a.out + (size_t)row * a.ldo + col, v, min(16, ncols - col));
      if (more) {
#pragma unroll
        for (int j = 0; j < 16; ++j) w[j] = wn[j];
      }
    }
    return;
  }

  if constexpr (EPI == kEpiSwiGLU) {
    constexpr int HALF = BN / 2;
    const int f0 = tl.n_loc * HALF;
    const int ffn = a.group_cols[0];
#pragma unroll 1
    for (int c = 0; c < HALF; c += 16) {
      tmem_ld16(tacc + c, r0);
      tmem_ld16(tacc + HALF + c, r1);
      tmem_ld_wait();
      const int col = f0 + c;
      if (!row_ok || col >= ffn) continue;
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        const float gt = __uint_as_float(r0[j]);
        const float up = __uint_as_float(r1[j]);
        v[j] = gt / (1.0f + __expf(-gt)) * up;
      }
      store_bf16_n(a.out + (size_t)row * a.ldo + col, v, min(16, ffn - col));
    }
    return;
  }

  if constexpr (EPI == kEpiQkv) {
    // kEpiQkv: group 0 = q, 1 = k, 2 = v; tiles are head-aligned (BN % head_dim == 0).
    const int d = a.head_dim;
    const int half = d >> 1;
    int pos = 0;
    const int32_t* pt = nullptr;
    const bool have = row_ok && row_lookup(a.req, row, pos, pt);
    const int g = tl.g;
    const __nv_bfloat16* bias = a.bias[g];
    __nv_bfloat16* dst_row = nullptr;
    size_t head_stride = 0;
    if (have) {
      if (g == 0) {
        dst_row = a.qbuf + (size_t)row * a.ldq;
        head_stride = d;
      } else {
        const int page = checked_page(pt[pos / kPage], a.req.num_pages, a.status);
        __nv_bfloat16* base = (g == 1) ? a.kpages : a.vpages;
        dst_row = base + ((size_t)page * a.n_kv_heads * kPage + (pos % kPage)) * d;
        head_stride = (size_t)kPage * d;
      }
    }
    // Chunks of 16 rotation pairs outermost: a chunk's cos/sin (one row of the angle table,
    // shared by every head of the tile) is loaded once, and the next chunk's is requested
    // while this one is applied, so the table's load latency overlaps the TMEM drain.
    const bool rot = have && g < 2;
    const float4* rope4 = reinterpret_cast<const float4*>(a.rope + (size_t)pos * half);
    float4 cs[8], csn[8];
    if (rot) {
  #pragma unroll
      for (int k = 0; k < 8; ++k) cs[k] = rope4[k];
    }
  #pragma unroll 1
    for (int i0 = 0; i0 < half; i0 += 16) {
      const bool more = rot && i0 + 16 < half;
      if (more) {
  #pragma unroll
        for (int k = 0; k < 8; ++k) csn[k] = rope4[(i0 + 16) / 2 + k];
      }
  #pragma unroll 1
      for (int hh = 0; hh < BN / d; ++hh) {
        const int head = (tl.n_loc * BN) / d + hh;
        const int gcol = head * d;
        tmem_ld16(tacc + hh * d + i0, r0);
        tmem_ld16(tacc + hh * d + half + i0, r1);
        tmem_ld_wait();
        if (!have || gcol >= a.group_cols[g]) continue;
  #pragma unroll
        for (int j = 0; j < 16; ++j) {
          v[j] = __uint_as_float(r0[j]);
          w[j] = __uint_as_float(r1[j]);
        }
        if (bias) {
          float b0[16], b1[16];
          load16_bf16(bias + gcol + i0, b0);
          load16_bf16(bias + gcol + half + i0, b1);
  #pragma unroll
          for (int j = 0; j < 16; ++j) {
            v[j] += b0[j];
            w[j] += b1[j];
          }
        }
        if (g < 2) {
  #pragma unroll
          for (int j = 0; j < 16; ++j) {
            const float c = (j & 1) ? cs[j >> 1].z : cs[j >> 1].x;
            const float sn = (j & 1) ? cs[j >> 1].w : cs[j >> 1].y;
            const float x1 = v[j], x2 = w[j];
            v[j] = x1 * c - x2 * sn;
            w[j] = x2 * c + x1 * sn;
          }
        }
        __nv_bfloat16* dst = dst_row + head * head_stride;
        store16_bf16(dst + i0, v);
        store16_bf16(dst + half + i0, w);
      }
      if (more) {
  #pragma unroll
        for (int k = 0; k < 8; ++k) cs[k] = csn[k];
      }
    }
  }
}

// Bounded wait until *flag >= target (acquire at GPU scope). Gives up like mbar_wait.
__device__ __forceinline__ bool flag_wait(const int* flag, int target, volatile int* abort_flag, int* status) {
  unsigned long long t0 = 0;
  for (uint32_t it = 0;; ++it) {
    int v;
    asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(flag) : "memory");
    if (v >= target) return true;
    if (*abort_flag) return false;
    if ((it & 15u) == 0) {
      const unsigned long long now = globaltimer_ns();
      if (t0 == 0) {
        t0 = now;
      } else if (now - t0 > kWaitLimitNs) {
        *abort_flag = 1;
        if (status) atomicOr(status, kStatusTimeout);
        return false;
      }
    }
    __nanosleep(128);
  }
}

__device__ __forceinline__ void fence_proxy_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}

// Stage layout: the A tile (this CTA's 128 rows x 64), the B tile (its 128 rows x 64) and, for XA
// tiles, the LoRA A rows of its half of the XA product (up to 32 rows x 64); 128-byte swizzle.
constexpr int kABytes = BM * BK * 2;
constexpr int kBBytes = 128 * BK * 2;
constexpr int kLaBytes = 32 * BK * 2;
constexpr int kStageBytes = kABytes + kBBytes + kLaBytes;
constexpr int kPair = 2;

// Producer ring position (stage, phase) and whether every wait so far succeeded.
struct Ring {
  int stage;
  uint32_t phase;
  int ok;
};

template <int STAGES>
__device__ __forceinline__ void ring_next(Ring& r) {
  if (++r.stage == STAGES) {
    r.stage = 0;
    r.phase ^= 1;
  }
}

// B rows of an output tile staged by CTA `rank`: its share of the tile (plain) or its segment of
// the stacked tile; with the map index of the first of them.
template <int BN>
__device__ __forceinline__ void tile_b_rows(const GemmArgs& a, const Tile& tl, uint32_t rank, int& g0, int& nb,
                                            int& yb, int& b_step) {
  const int nseg = a.nseg;
  const int seg_rows = BN / nseg;
  const int per = nseg / kPair;
  g0 = nseg == 1 ? tl.g : tl.g + static_cast<int>(rank) * per;
  nb = nseg == 1 ? 1 : per;
  yb = nseg == 1 ? tl.n_loc * BN + static_cast<int>(rank) * (BN / kPair) : tl.n_loc * seg_rows;
  b_step = nseg == 1 ? 0 : seg_rows * BK * 2;
}

// Copies of an XA tile: per K block the tile's x and W rows, as for any output tile, and the LoRA
// A rows of this CTA's half of the XA product (16 rows per XA slot; CTA r takes slots
// [r * spc, r * spc + spc)). Its LoRA stage, if it has one, gets the BX rows only: the epilogue
// warps write the A side from the XA product.
template <int BN, int STAGES>
__device__ __noinline__ Ring load_xa_tile(const GemmArgs& a, const Tile& tl, int m0, uint32_t rank, bool leader,
                                          uint8_t* smem, uint64_t* full_bar, uint64_t* empty_bar,
                                          int* armed_parity, volatile int* abort_flag, Ring ring) {
  int g0, nb, yb, b_step;
  tile_b_rows<BN>(a, tl, rank, g0, nb, yb, b_step);
  const int spc = a.xa_n / (16 * kPair);
  const int s0 = static_cast<int>(rank) * spc, s1 = min(a.n_slots, s0 + spc);
  const uint32_t bytes = kPair * (kABytes + kBBytes) + a.n_slots * 16 * BK * 2;
  for (int kb = 0; kb < a.num_kb; ++kb) {
    if (!mbar_wait(&empty_bar[ring.stage], ring.phase ^ 1, abort_flag, a.status)) {
      ring.ok = 0;
      return ring;
    }
    uint8_t* sa = smem + ring.stage * kStageBytes;
    uint8_t* sb = sa + kABytes;
    uint8_t* sl = sb + kBBytes;
    if (leader) {
      mbar_arrive_expect_tx(&full_bar[ring.stage], bytes);
      armed_parity[ring.stage] = ring.phase;
    }
    const uint32_t bar = mapa_shared(&full_bar[ring.stage], 0);
    tma_load_2d_pair(sa, &a.tmA, bar, kb * BK, m0);
    for (int j = 0; j < nb; ++j) tma_load_2d_pair(sb + j * b_step, &a.tmB[g0 + j], bar, kb * BK, yb);
    for (int j = s0; j < s1; ++j) tma_load_2d_pair(sl + (j - s0) * 16 * BK * 2, &a.tmLA[j], bar, kb * BK, 0);
    ring_next<STAGES>(ring);
  }
  if (a.ext_on[tl.g]) {
    if (!mbar_wait(&empty_bar[ring.stage], ring.phase ^ 1, abort_flag, a.status)) {
      ring.ok = 0;
      return ring;
    }
    uint8_t* sb = smem + ring.stage * kStageBytes + kABytes;
    if (leader) {
      mbar_arrive_expect_tx(&full_bar[ring.stage], kPair * kBBytes);
      armed_parity[ring.stage] = ring.phase;
    }
    const uint32_t bar = mapa_shared(&full_bar[ring.stage], 0);
    for (int j = 0; j < nb; ++j) tma_load_2d_pair(sb + j * b_step, &a.tmBX[g0 + j], bar, 0, yb);
    ring_next<STAGES>(ring);
  }
  return ring;
}

// The LoRA stage of any other output tile: once the stage is free, wait (unless seen already)
// until both CTAs of the row block's XA tile have stored its XA rows, and copy those rows (the A
// side of the K block) and the tile's BX rows (the B side).
template <int BN, int STAGES>
__device__ __noinline__ Ring load_lora_stage(const GemmArgs& a, const Tile& tl, int m0, uint32_t rank, bool xa_ready,
                                             bool leader, uint8_t* smem, uint64_t* full_bar, uint64_t* empty_bar,
                                             int* armed_parity, volatile int* abort_flag, Ring ring) {
  if (!mbar_wait(&empty_bar[ring.stage], ring.phase ^ 1, abort_flag, a.status)) {
    ring.ok = 0;
    return ring;
  }
  if (!xa_ready && !flag_wait(a.xa_flags + tl.m_blk, 4 * kPair, abort_flag, a.status)) {
    ring.ok = 0;
    return ring;
  }
  fence_proxy_async_global();  // the TMA copy below reads what the XA tile's stores wrote
  int g0, nb, yb, b_step;
  tile_b_rows<BN>(a, tl, rank, g0, nb, yb, b_step);
  uint8_t* sa = smem + ring.stage * kStageBytes;
  if (leader) {
    mbar_arrive_expect_tx(&full_bar[ring.stage], kPair * (kABytes + kBBytes));
    armed_parity[ring.stage] = ring.phase;
  }
  const uint32_t bar = mapa_shared(&full_bar[ring.stage], 0);
  tma_load_2d_pair(sa, &a.tmXA, bar, a.xa_base[tl.g], m0);
  for (int j = 0; j < nb; ++j) tma_load_2d_pair(sa + kABytes + j * b_step, &a.tmBX[g0 + j], bar, 0, yb);
  ring_next<STAGES>(ring);
  return ring;
}

// MMAs of an XA tile: per K block the tile's product into d_tmem and the XA product x A^T into
// the other accumulator's first xa_n columns (x_tmem); then xa_full for the epilogue warps, which
// drain the XA product (xa_done, having written it into the tile's LoRA stage) before the LoRA
// stage, or the next tile, may use those columns.
template <int BN, int STAGES>
__device__ __noinline__ Ring mma_xa_tile(const GemmArgs& a, const Tile& tl, uint32_t d_tmem, uint32_t x_tmem,
                                         uint32_t idesc, uint32_t idesc_xa, uint8_t* smem, uint64_t* full_bar,
                                         uint64_t* empty_bar, uint64_t* xa_full, uint64_t* xa_done,
                                         uint32_t xa_parity, volatile int* abort_flag, Ring ring) {
  for (int kb = 0; kb < a.num_kb; ++kb) {
    if (!mbar_wait(&full_bar[ring.stage], ring.phase, abort_flag, a.status)) {
      ring.ok = 0;
      return ring;
    }
    tc_fence_after();
    const uint32_t sa = smem_u32(smem + ring.stage * kStageBytes);
    const uint64_t ad = smem_desc(sa, 16, 1024, kSwizzle128B);
    const uint64_t bd = smem_desc(sa + kABytes, 16, 1024, kSwizzle128B);
    const uint64_t ld = smem_desc(sa + kABytes + kBBytes, 16, 1024, kSwizzle128B);
#pragma unroll
    for (int k = 0; k < BK / 16; ++k) {
      const uint32_t acc = (kb > 0 || k > 0) ? 1u : 0u;
      mma_bf16_ss_pair(d_tmem, ad + 2 * k, bd + 2 * k, idesc, acc);
      mma_bf16_ss_pair(x_tmem, ad + 2 * k, ld + 2 * k, idesc_xa, acc);
    }
    mma_commit_pair(&empty_bar[ring.stage], 0x3);
    ring_next<STAGES>(ring);
  }
  mma_commit_pair(xa_full, 0x3);
  if (!mbar_wait<true>(xa_done, xa_parity, abort_flag, a.status)) {
    ring.ok = 0;
    return ring;
  }
  tc_fence_after();
  if (a.ext_on[tl.g]) {
    // BX copies landed; the A side (the XA product) came with xa_done
    if (!mbar_wait(&full_bar[ring.stage], ring.phase, abort_flag, a.status)) {
      ring.ok = 0;
      return ring;
    }
    tc_fence_after();
    const uint32_t sa = smem_u32(smem + ring.stage * kStageBytes);
    const uint64_t ad = smem_desc(sa, 16, 1024, kSwizzle128B);
    const uint64_t bd = smem_desc(sa + kABytes, 16, 1024, kSwizzle128B);
    for (int k = 0; k < a.ext_steps[tl.g]; ++k) mma_bf16_ss_pair(d_tmem, ad + 2 * k, bd + 2 * k, idesc, 1u);
    mma_commit_pair(&empty_bar[ring.stage], 0x3);
    ring_next<STAGES>(ring);
  }
  return ring;
}

// XA tile, after its main loop: slot j of the XA product (columns 16j .. 16j + 15 of x_tmem) is
// x A_j^T for this thread's row. Scaled by alpha / r it is stored as hi = bf16(v) at XA columns
// 32j.. and lo = bf16(v - hi) at 32j + 16.. (the pair carries about 16 mantissa bits): to the XA
// buffer for the row block's other tiles, and into the tile's own LoRA stage `st` (A side, the 64
// columns from xa_base) when it has one. Then xa_done for the MMAs and the row block's ready word.
template <int BN>
__device__ __noinline__ bool drain_xa(const GemmArgs& a, const Tile& tl, uint32_t x_tmem, int row, int row_in_cta,
                                      int st, int lane, uint8_t* smem, uint64_t* xa_full, uint64_t* xa_done,
                                      uint32_t xa_parity, volatile int* abort_flag) {
  if (!__all_sync(0xffffffffu, mbar_wait(xa_full, xa_parity, abort_flag, a.status))) return false;
  tc_fence_after();
  const bool ext = a.ext_on[tl.g] != 0;
  const int xb = a.xa_base[tl.g];
  uint8_t* arow = smem + st * kStageBytes + row_in_cta * 128;
  uint32_t r0[16];
  float v[16], w[16];
#pragma unroll 1
  for (int j = 0; j < a.n_slots; ++j) {
    tmem_ld16(x_tmem + 16 * j, r0);
    tmem_ld_wait();
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      v[i] = __uint_as_float(r0[i]) * a.scale;
      w[i] = v[i] - __bfloat162float(__float2bfloat16_rn(v[i]));
    }
    if (row < a.M) {
      store16_bf16(a.xa + (size_t)row * kXaCols + 32 * j, v);
      store16_bf16(a.xa + (size_t)row * kXaCols + 32 * j + 16, w);
    }
    const int c0 = (32 * j - xb) / 8;  // 16-byte unit of hi within the stage's 64 columns
    if (ext && 32 * j >= xb && 32 * j < xb + BK) {
      uint4 q[4];
      q[0] = make_uint4(pack_bf16(v[0], v[1]), pack_bf16(v[2], v[3]), pack_bf16(v[4], v[5]), pack_bf16(v[6], v[7]));
      q[1] = make_uint4(pack_bf16(v[8], v[9]), pack_bf16(v[10], v[11]), pack_bf16(v[12], v[13]),
                        pack_bf16(v[14], v[15]));
      q[2] = make_uint4(pack_bf16(w[0], w[1]), pack_bf16(w[2], w[3]), pack_bf16(w[4], w[5]), pack_bf16(w[6], w[7]));
      q[3] = make_uint4(pack_bf16(w[8], w[9]), pack_bf16(w[10], w[11]), pack_bf16(w[12], w[13]),
                        pack_bf16(w[14], w[15]));
#pragma unroll
      for (int u = 0; u < 4; ++u)
        *reinterpret_cast<uint4*>(arow + (((c0 + u) ^ (row_in_cta & 7)) << 4)) = q[u];
    }
  }
  // TMEM columns read (tcgen05.wait::ld above); XA rows visible to the tensor core of this CTA
  // (shared) and to the other tiles' copies (global, GPU scope)
  tc_fence_before();
  fence_proxy_async_smem();
  __threadfence();
  fence_proxy_async_global();
  __syncwarp();
  if (lane == 0) {
    mbar_arrive_cluster(mapa_shared(xa_done, 0));
    atomicAdd(a.xa_flags + tl.m_blk, 1);
  }
  return true;
}

template <int BN, int STAGES, int EPI>
__global__ void __launch_bounds__(kThreads, 1) gemm_tc_kernel(const __grid_constant__ GemmArgs a) {
  static_assert(BN == 256 && kBBytes == (BN / kPair) * BK * 2, "CTA-pair tiles of 256 columns");
  constexpr uint32_t TMEM_COLS = 2 * BN;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  __shared__ __align__(8) uint64_t full_bar[STAGES];
  __shared__ __align__(8) uint64_t empty_bar[STAGES];
  __shared__ __align__(8) uint64_t tfull_bar[2];
  __shared__ __align__(8) uint64_t tempty_bar[2];
  __shared__ __align__(8) uint64_t drain_bar;
  __shared__ __align__(8) uint64_t xa_full;         // an XA tile's MMAs done (MMA commit)
  __shared__ __align__(8) uint64_t xa_done;         // its XA product drained (each epilogue warp of both CTAs)
  __shared__ uint32_t tmem_base_sh;
  __shared__ volatile int abort_flag;
  // a rejected call: every CTA of every cluster sees the same word and leaves before any set-up
  if (call_aborted(a.abort)) return;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const bool leader = rank == 0;
  const int unit = blockIdx.x / kPair;
  const int n_units = gridDim.x / kPair;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&tfull_bar[i], 1);
      mbar_init(&tempty_bar[i], 4 * kPair);
    }
    mbar_init(&drain_bar, 1);
    mbar_init(&xa_full, 1);
    mbar_init(&xa_done, 4 * kPair);
    abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&a.tmA);
    for (int i = 0; i < 3; ++i) tma_prefetch_desc(&a.tmB[i]);
    if (a.n_slots > 0) {
      tma_prefetch_desc(&a.tmXA);
      for (int i = 0; i < a.n_slots; ++i) tma_prefetch_desc(&a.tmLA[i]);
      for (int i = 0; i < 3; ++i) tma_prefetch_desc(&a.tmBX[i]);
    }
  }
  if (warp == 1) {
    tmem_alloc_pair(&tmem_base_sh, TMEM_COLS);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  cluster_sync();
  tc_fence_after();
  const uint32_t tmem_base = tmem_base_sh;

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer (every CTA)
    // The per-stage loop of the output tiles stays minimal (one thread, on the critical path of
    // every stage); XA tiles and the LoRA stage go through out-of-line helpers.
    if (lane == 0) {
      Ring ring{0, 0u, 1};
      int armed_parity[STAGES];
      for (int s = 0; s < STAGES; ++s) armed_parity[s] = -1;
      for (int t = unit; t < a.total_tiles && ring.ok; t += n_units) {
        const Tile tl = decode_tile(t, a);
        const int m0 = tl.m_blk * (BM * kPair) + static_cast<int>(rank) * BM;
        if (tl.xa) {
          ring = load_xa_tile<BN, STAGES>(a, tl, m0, rank, leader, smem, full_bar, empty_bar, armed_parity,
                                          &abort_flag, ring);
          continue;
        }
        int g0, nb, yb, b_step;
        tile_b_rows<BN>(a, tl, rank, g0, nb, yb, b_step);
        // Whether the row block's XA rows are stored, asked (acquire) while the stages already
        // copied still feed the MMAs; only a tile whose XA tile has not finished by then waits at
        // its LoRA stage.
        int xa_ready = 0;
        if (a.ext_on[tl.g]) {
          asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(xa_ready) : "l"(a.xa_flags + tl.m_blk) : "memory");
          xa_ready = xa_ready >= 4 * kPair;
        }
        int stage = ring.stage;
        uint32_t phase = ring.phase;
        for (int kb = 0; kb < a.num_kb; ++kb) {
          if (!mbar_wait(&empty_bar[stage], phase ^ 1, &abort_flag, a.status)) {
            ring.ok = 0;
            break;
          }
          uint8_t* sa = smem + stage * kStageBytes;
          uint8_t* sb = sa + kABytes;
          // the MMA-issuing CTA's full barrier counts the bytes of both CTAs
          if (leader) {
            mbar_arrive_expect_tx(&full_bar[stage], kPair * (kABytes + kBBytes));
            armed_parity[stage] = phase;
          }
          const CUtensorMap* mB = &a.tmB[g0];
          const uint32_t bar = mapa_shared(&full_bar[stage], 0);
          tma_load_2d_pair(sa, &a.tmA, bar, kb * BK, m0);
          for (int j = 0; j < nb; ++j) tma_load_2d_pair(sb + j * b_step, mB + j, bar, kb * BK, yb);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
        ring.stage = stage;
        ring.phase = phase;
        if (ring.ok && a.ext_on[tl.g])
          ring = load_lora_stage<BN, STAGES>(a, tl, m0, rank, xa_ready != 0, leader, smem, full_bar, empty_bar,
                                             armed_parity, &abort_flag, ring);
      }
      if (!ring.ok) {
        if (leader) {
          // Let every copy already issued land before the CTA can exit.
          for (int s = 0; s < STAGES; ++s)
            if (armed_parity[s] >= 0) {
              volatile int never = 0;
              mbar_wait(&full_bar[s], static_cast<uint32_t>(armed_parity[s]), &never, nullptr);
            }
        } else {
          // The peer's copies complete on the other CTA's barriers: give them time to land.
          const unsigned long long t0 = globaltimer_ns();
          while (globaltimer_ns() - t0 < 200000ull) {
          }
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer (even CTA)
    if (lane == 0 && leader) {
      Ring ring{0, 0u, 1};
      int it = 0;
      bool issued = false;
      const uint32_t idesc = idesc_bf16_f32(BM * kPair, BN);
      const uint32_t idesc_xa = idesc_bf16_f32(BM * kPair, a.n_slots > 0 ? a.xa_n : 32);
      uint32_t xa_it = 0;      // XA tiles so far (phase of xa_done)
      for (int t = unit; t < a.total_tiles && ring.ok; t += n_units, ++it) {
        const Tile tl = decode_tile(t, a);
        const int acc = it & 1;
        const uint32_t acc_phase = (it >> 1) & 1;
        if (!mbar_wait<true>(&tempty_bar[acc], acc_phase ^ 1, &abort_flag, a.status)) {
          ring.ok = 0;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * BN;
        if (tl.xa) {
          // the XA product takes the other accumulator's first columns: its previous tile's
          // epilogue must have drained them
          if (!mbar_wait<true>(&tempty_bar[acc ^ 1], (((it + 1) >> 1) & 1) ^ 1, &abort_flag, a.status)) {
            ring.ok = 0;
            break;
          }
          tc_fence_after();
          ring = mma_xa_tile<BN, STAGES>(a, tl, d_tmem, tmem_base + (acc ^ 1) * BN, idesc, idesc_xa, smem, full_bar,
                                         empty_bar, &xa_full, &xa_done, xa_it & 1u, &abort_flag, ring);
          ++xa_it;
          issued = true;
          if (!ring.ok) break;
          mma_commit_pair(&tfull_bar[acc], 0x3);
          continue;
        }
        int stage = ring.stage;
        uint32_t phase = ring.phase;
        for (int kb = 0; kb < a.num_kb; ++kb) {
          if (!mbar_wait(&full_bar[stage], phase, &abort_flag, a.status)) {
            ring.ok = 0;
            break;
          }
          tc_fence_after();
          const uint32_t sa = smem_u32(smem + stage * kStageBytes);
          const uint64_t ad = smem_desc(sa, 16, 1024, kSwizzle128B);
          const uint64_t bd = smem_desc(sa + kABytes, 16, 1024, kSwizzle128B);
          // K = 16 steps advance 32 bytes = 2 units of the descriptor's start-address field
#pragma unroll
          for (int k = 0; k < BK / 16; ++k)
            mma_bf16_ss_pair(d_tmem, ad + 2 * k, bd + 2 * k, idesc, (kb > 0 || k > 0) ? 1u : 0u);
          issued = true;
          mma_commit_pair(&empty_bar[stage], 0x3);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
        ring.stage = stage;
        ring.phase = phase;
        if (ring.ok && a.ext_on[tl.g]) {
          // the XA and BX copies have landed
          if (!mbar_wait(&full_bar[ring.stage], ring.phase, &abort_flag, a.status)) {
            ring.ok = 0;
          } else {
            tc_fence_after();
            const uint32_t sa = smem_u32(smem + ring.stage * kStageBytes);
            const uint64_t ad = smem_desc(sa, 16, 1024, kSwizzle128B);
            const uint64_t bd = smem_desc(sa + kABytes, 16, 1024, kSwizzle128B);
            for (int k = 0; k < a.ext_steps[tl.g]; ++k) mma_bf16_ss_pair(d_tmem, ad + 2 * k, bd + 2 * k, idesc, 1u);
            mma_commit_pair(&empty_bar[ring.stage], 0x3);
            ring_next<STAGES>(ring);
          }
        }
        if (!ring.ok) break;
        mma_commit_pair(&tfull_bar[acc], 0x3);
      }
      if (!ring.ok && issued) {
        mma_commit_pair(&drain_bar, 0x1);
        volatile int never = 0;
        mbar_wait(&drain_bar, 0, &never, nullptr);
      }
    }
  } else {
    // ------------------------------------------------------------ epilogue (warps 2..5, every CTA)
    const int quarter = warp & 3;  // TMEM lane quarter this warp may access
    const int row_in_cta = quarter * 32 + lane;
    uint32_t tempty_addr[2];
    for (int i = 0; i < 2; ++i) tempty_addr[i] = mapa_shared(&tempty_bar[i], 0);
    int pos = 0;             // producer stages used by the tiles before this one
    uint32_t xa_it = 0;      // XA tiles so far (phase of xa_full)
    int it = 0;
    for (int t = unit; t < a.total_tiles; t += n_units, ++it) {
      const Tile tl = decode_tile(t, a);
      const int acc = it & 1;
      const uint32_t acc_phase = (it >> 1) & 1;
      const bool ext_tile = a.ext_on[tl.g] != 0;
      const int st = (pos + a.num_kb) % STAGES;  // the tile's LoRA stage
      const int row = tl.m_blk * (BM * kPair) + static_cast<int>(rank) * BM + row_in_cta;
      if (tl.xa) {
        const uint32_t x_tmem = tmem_base + (static_cast<uint32_t>(quarter * 32) << 16) + (acc ^ 1) * BN;
        if (!drain_xa<BN>(a, tl, x_tmem, row, row_in_cta, st, lane, smem, &xa_full, &xa_done, xa_it & 1u,
                          &abort_flag))
          break;
        ++xa_it;
      }
      pos += a.num_kb + (ext_tile ? 1 : 0);
      // warp-uniform outcome: the TMEM loads of the epilogue are warp-collective
      if (!__all_sync(0xffffffffu, mbar_wait(&tfull_bar[acc], acc_phase, &abort_flag, a.status)))
        break;
      tc_fence_after();
      const uint32_t tacc = tmem_base + (static_cast<uint32_t>(quarter * 32) << 16) + acc * BN;
      epilogue_tile<BN, EPI>(a, tl, tacc, row);
      // the accumulator is free once this warp's TMEM loads have completed (tcgen05.wait::ld in
      // the epilogue); the tile's global stores need not be visible first, so the arrival on
      // the MMA-issuing CTA's barrier is relaxed
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster_relaxed(tempty_addr[acc]);
    }
  }

  tc_fence_before();
  cluster_sync();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, TMEM_COLS);
  }
}

// ---------------------------------------------------------------- host side
using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                   const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                   const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

// 2-D bf16 map over rows x cols (row stride ld elements), box box_rows x box_cols.
bool make_map(CUtensorMap* m, const void* base, int rows, int cols, int ld, int box_rows,
              int box_cols, CUtensorMapSwizzle sw) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(ld) * 2};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(box_cols), static_cast<cuuint32_t>(box_rows)};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides,
                  box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

template <int BN, int STAGES, int EPI>
cudaError_t launch_impl(GemmArgs& args, int num_sms, cudaStream_t stream) {
  constexpr int PAIR = kPair;
  constexpr int smem = STAGES * kStageBytes + 1024;
  auto kern = gemm_tc_kernel<BN, STAGES, EPI>;
  // the attributes and the co-resident cluster count are per device
  static PerDevice once;
  static std::atomic<int> units_of[64];
  int dev = 0, max_units = 0;
  if (!once.pending(&dev)) {
    max_units = units_of[dev].load(std::memory_order_relaxed);
  } else {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 0);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = PAIR;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.gridDim = dim3(num_sms);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int clusters = 0;
    e = cudaOccupancyMaxActiveClusters(&clusters, kern, &cfg);
    if (e != cudaSuccess) return e;
    max_units = std::max(1, std::min(clusters, num_sms / PAIR));
    if (dev >= 0 && dev < 64) units_of[dev].store(max_units, std::memory_order_relaxed);
    once.done(dev);
  }
  // every unit of the grid is resident at once (one CTA per SM): a tile that waits for its row
  // block's XA tile never waits on a unit that has not started
  const int units = std::max(1, std::min(max_units, args.total_tiles));
  // every XA tile first: consecutive tiles go to consecutive units, so the XA products (and the
  // extra MMAs they cost) spread over the units instead of piling on a few
  args.xa_lead = args.row_tiles;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = PAIR;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.gridDim = dim3(PAIR * units);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, args);
}

}  // namespace

cudaError_t launch_gemm(const GemmDesc& d, int num_sms, cudaStream_t stream) {
  constexpr int bn = 256, pair = 2;
  GemmArgs a;
  std::memset(&a, 0, sizeof(a));
  if (d.nseg != 1 && d.nseg != 2) return cudaErrorInvalidValue;
  // rows of one B load: the CTA's share of the tile (plain) or one stacked segment
  const int b_box = d.nseg == 1 ? bn / pair : bn / d.nseg;
  if (!make_map(&a.tmA, d.A, d.M, d.K, d.lda, BM, BK, CU_TENSOR_MAP_SWIZZLE_128B))
    return cudaErrorInvalidValue;
  const int nmaps = d.ngroups + d.nseg - 1;
  for (int i = 0; i < 3; ++i) {
    const int src = i < nmaps ? i : 0;  // unused slots alias a valid map
    if (!make_map(&a.tmB[i], d.B[src], d.B_rows[src], d.K, d.ldb[src], b_box, BK,
                  CU_TENSOR_MAP_SWIZZLE_128B))
      return cudaErrorInvalidValue;
  }
  bool any_ext = false;
  for (int g = 0; g < d.ngroups; ++g) any_ext |= d.ext_on[g] != 0;
  if (any_ext != (d.n_slots > 0) || d.n_slots < 0 || d.n_slots > 3) return cudaErrorInvalidValue;
  if (any_ext) {
    if (!d.XA || !d.xa_flags || (d.rank != 4 && d.rank != 8 && d.rank != 16)) return cudaErrorInvalidValue;
    if (!make_map(&a.tmXA, d.XA, d.M, kXaCols, kXaCols, BM, BK, CU_TENSOR_MAP_SWIZZLE_128B))
      return cudaErrorInvalidValue;
    for (int j = 0; j < 3; ++j) {
      const int src = j < d.n_slots ? j : 0;
      if (!d.LA[src] || !make_map(&a.tmLA[j], d.LA[src], d.rank, d.K, d.K, 16, BK, CU_TENSOR_MAP_SWIZZLE_128B))
        return cudaErrorInvalidValue;
    }
    for (int g = 0; g < d.ngroups; ++g) {
      if (!d.ext_on[g]) continue;
      // the 64-wide block must lie inside the XA row, 16-byte aligned (TMA x coordinate)
      if (d.xa_base[g] < 0 || d.xa_base[g] % 32 != 0 || d.xa_base[g] + BK > kXaCols ||
          d.ext_steps[g] < 1 || d.ext_steps[g] > BK / 16)
        return cudaErrorInvalidValue;
    }
    for (int i = 0; i < 3; ++i) {
      int src = (i < nmaps && d.BX[i]) ? i : -1;
      if (src < 0)
        for (int j = 0; j < nmaps; ++j)
          if (d.BX[j]) src = j;  // unused slots alias a valid map
      if (src < 0) return cudaErrorInvalidValue;
      if (!make_map(&a.tmBX[i], d.BX[src], d.B_rows[src], kBxCols, kBxCols, b_box, BK, CU_TENSOR_MAP_SWIZZLE_128B))
        return cudaErrorInvalidValue;
    }
    for (int g = 0; g < d.ngroups; ++g)
      for (int s = 0; s < (d.ngroups == 1 ? d.nseg : 1); ++s)
        if (d.ext_on[g] && !d.BX[g + s]) return cudaErrorInvalidValue;
  } else {
    a.tmXA = a.tmA;
    for (int i = 0; i < 3; ++i) a.tmLA[i] = a.tmBX[i] = a.tmA;
  }
  a.M = d.M;
  a.K = d.K;
  a.num_kb = (d.K + BK - 1) / BK;
  a.ngroups = d.ngroups;
  a.nseg = d.nseg;
  a.total_n = 0;
  for (int g = 0; g < d.ngroups; ++g) {
    const int cols_per_tile = (d.nseg > 1 && d.epi == kEpiSwiGLU) ? bn / d.nseg : bn;
    a.group_cols[g] = d.group_cols[g];
    a.group_tiles[g] = (d.nseg > 1 && d.epi != kEpiSwiGLU) ? 1
                                                            : (d.group_cols[g] + cols_per_tile - 1) /
                                                                  cols_per_tile;
    a.total_n += a.group_tiles[g];
    a.ext_on[g] = d.ext_on[g];
    a.ext_steps[g] = d.ext_steps[g];
    a.xa_base[g] = d.xa_base[g];
  }
  a.row_tiles = (d.M + BM * pair - 1) / (BM * pair);
  a.n_slots = any_ext ? d.n_slots : 0;
  // two CTA halves of 16 x ceil(n_slots / 2) rows: N = 32 for one or two slots, 64 for three
  a.xa_n = 32 * ((a.n_slots + 1) / 2);
  a.rank = d.rank;
  a.xa = static_cast<__nv_bfloat16*>(d.XA);
  a.xa_flags = d.xa_flags;
  a.total_tiles = a.row_tiles * a.total_n;
  a.epi = d.epi;
  a.scale = d.scale;
  a.out = static_cast<__nv_bfloat16*>(d.out);
  a.ldo = d.ldo;
  a.resid = static_cast<const __nv_bfloat16*>(d.resid);
  a.ld_resid = d.ld_resid;
  for (int i = 0; i < 3; ++i) a.bias[i] = static_cast<const __nv_bfloat16*>(d.bias[i]);
  a.rope = d.rope;
  a.head_dim = d.head_dim;
  a.n_kv_heads = d.n_kv_heads;
  a.qbuf = static_cast<__nv_bfloat16*>(d.qbuf);
  a.ldq = d.ldq;
  a.kpages = static_cast<__nv_bfloat16*>(d.kpages);
  a.vpages = static_cast<__nv_bfloat16*>(d.vpages);
  a.req = d.req;
  a.status = d.status;
  a.abort = d.abort;
  if (a.total_tiles == 0) return cudaSuccess;
  // one kernel per epilogue: each carries only its own epilogue code, which keeps the hot loops
  // of all its warps inside the SM's instruction cache
  switch (d.epi) {
    case kEpiQkv: return launch_impl<bn, 6, kEpiQkv>(a, num_sms, stream);
    case kEpiResid: return launch_impl<bn, 6, kEpiResid>(a, num_sms, stream);
    case kEpiSwiGLU: return launch_impl<bn, 6, kEpiSwiGLU>(a, num_sms, stream);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace crf
