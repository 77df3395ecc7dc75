// Persistent tcgen05 GEMM for sm_103a with fused LoRA-up and fused epilogues.
//
//   D[BM*PAIR x BN] = A[BM*PAIR x K] * B[BN x K]^T  (+ XA[. x 64] * BX[BN x 64]^T)
//
// PAIR = 2 (the projection GEMMs): a cluster of two CTAs on one TPC works on a
// 256 x 256 tile with cta_group::2 MMAs. Each CTA stages its own 128 rows of A
// and its own half of the B rows, so the operand bytes each SM pulls through L2
// per FLOP are two thirds of the single-CTA 128 x 256 tile's. The even CTA
// issues the MMAs; both CTAs hold 128 accumulator lanes in their own TMEM and
// drain them through the same epilogue. PAIR = 1: one CTA per tile (the narrow
// LoRA-down products).
//
// Per CTA: warp 0 issues TMA loads into a STAGES-deep shared-memory ring, warp 1
// owns TMEM (two accumulators, so the epilogue of tile i overlaps the main loop
// of tile i+1) and, in the MMA-issuing CTA, issues tcgen05.mma from one thread;
// warps 2..5 drain the accumulator (one TMEM lane = one output row per thread)
// through the fused epilogue. Operands are bf16, K-major, staged with 128-byte
// swizzle; accumulation is fp32 in TMEM.
//
// The unmerged adapter term (alpha/r) (x A^T) B^T of every adapted projection
// (Eq. S3 with W = W0 + (alpha/r) B A) enters as one extra 64-wide K block per
// tile: A side = the scaled down product of the tile's rows stored as a bf16
// pair [hi | lo] per module (16 + 16 columns), B side = rows of BX = [B | B]
// placed under that module's columns (zeros elsewhere), so one K block serves
// up to two stacked modules and the two halves of a pair alike.
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
  CUtensorMap tmBX[3];
  int M, K, num_kb;
  int ngroups, nseg;
  int group_tiles[3];
  int group_cols[3];
  int ext_on[3];      // per group: tile has the LoRA K block
  int ext_steps[3];   // per group: K = 16 steps of that block that carry data
  int xa_base[3];     // per group: first XA column of that block
  int row_tiles, total_n, total_tiles;
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
};

__device__ __forceinline__ Tile decode_tile(int t, const GemmArgs& a) {
  const int band_tiles = a.row_tiles * kRasterGroup;
  const int band = t / band_tiles;
  const int idx = t - band * band_tiles;
  const int n0 = band * kRasterGroup;
  const int width = min(kRasterGroup, a.total_n - n0);
  Tile r;
  r.m_blk = idx / width;
  int n = n0 + (idx - r.m_blk * width);
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

template <int BN>
__device__ __forceinline__ void epilogue_tile(const GemmArgs& a, const Tile& tl, uint32_t tacc,
                                              int row) {
  const bool row_ok = row < a.M;
  uint32_t r0[16], r1[16];
  float v[16], w[16];

  if (a.epi == kEpiScaleBf16 || a.epi == kEpiResid) {
    const int col0 = tl.n_loc * BN;
    const int ncols = a.group_cols[tl.g];
    const bool resid = a.epi == kEpiResid;
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
    if (resid && row_ok && col0 < ncols) load_resid(col0, w);
#pragma unroll 1
    for (int c = 0; c < BN; c += 16) {
      tmem_ld16(tacc + c, r0);
      const bool more = resid && row_ok && c + 16 < BN && col0 + c + 16 < ncols;
      if (more) load_resid(col0 + c + 16, wn);
      tmem_ld_wait();
      const int col = col0 + c;
      if (!row_ok || col >= ncols) continue;
      const int n = min(16, ncols - col);
      if (a.epi == kEpiScaleBf16) {
        // hi = bf16(v), lo = bf16(v - hi): the pair carries the product to ~16 mantissa bits.
        // Module slot j = col / 16 keeps hi at columns 32j.. and lo at 32j + 16..
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          v[j] = __uint_as_float(r0[j]) * a.scale;
          w[j] = v[j] - __bfloat162float(__float2bfloat16_rn(v[j]));
        }
        store_bf16_n(a.out + (size_t)row * a.ldo + 2 * col + 16, w, n);
        store_bf16_n(a.out + (size_t)row * a.ldo + 2 * col, v, n);
        continue;
      } else {
#pragma unroll
        for (int j = 0; j < 16; ++j) v[j] = w[j] + __uint_as_float(r0[j]);
      }
      store_bf16_n(a.out + (size_t)row * a.ldo + col, v, n);
      if (more) {
#pragma unroll
        for (int j = 0; j < 16; ++j) w[j] = wn[j];
      }
    }
    return;
  }

  if (a.epi == kEpiSwiGLU) {
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

template <int BN, int STAGES, int PAIR>
__global__ void __launch_bounds__(kThreads, 1) gemm_tc_kernel(const __grid_constant__ GemmArgs a) {
  constexpr int CTA_ROWS = BN / PAIR;  // B rows staged by this CTA
  constexpr int A_BYTES = BM * BK * 2;
  constexpr int B_BYTES = CTA_ROWS * BK * 2;
  constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  constexpr uint32_t TMEM_COLS = (2 * BN <= 32) ? 32 : (2 * BN <= 64) ? 64 : (2 * BN <= 128) ? 128
                                                    : (2 * BN <= 256) ? 256 : 512;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  __shared__ __align__(8) uint64_t full_bar[STAGES];
  __shared__ __align__(8) uint64_t empty_bar[STAGES];
  __shared__ __align__(8) uint64_t tfull_bar[2];
  __shared__ __align__(8) uint64_t tempty_bar[2];
  __shared__ __align__(8) uint64_t drain_bar;
  __shared__ uint32_t tmem_base_sh;
  __shared__ volatile int abort_flag;
  // a rejected call: every CTA of every cluster sees the same word and leaves before any set-up
  if (call_aborted(a.abort)) return;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = PAIR == 2 ? cluster_ctarank() : 0u;
  const bool leader = rank == 0;
  const int unit = blockIdx.x / PAIR;
  const int n_units = gridDim.x / PAIR;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&tfull_bar[i], 1);
      mbar_init(&tempty_bar[i], 4 * PAIR);
    }
    mbar_init(&drain_bar, 1);
    abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&a.tmA);
    for (int i = 0; i < 3; ++i) tma_prefetch_desc(&a.tmB[i]);
  }
  if (warp == 1) {
    if constexpr (PAIR == 2) {
      tmem_alloc_pair(&tmem_base_sh, TMEM_COLS);
      tmem_relinquish_pair();
    } else {
      tmem_alloc(&tmem_base_sh, TMEM_COLS);
      tmem_relinquish();
    }
  }
  tc_fence_before();
  if constexpr (PAIR == 2) cluster_sync(); else __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = tmem_base_sh;

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer (every CTA)
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      int armed_parity[STAGES];
      for (int s = 0; s < STAGES; ++s) armed_parity[s] = -1;
      bool ok = true;
      for (int t = unit; t < a.total_tiles && ok; t += n_units) {
        const Tile tl = decode_tile(t, a);
        const int m0 = tl.m_blk * (BM * PAIR) + static_cast<int>(rank) * BM;
        const bool ext_tile = a.ext_on[tl.g] != 0;
        const int nkb = a.num_kb + (ext_tile ? 1 : 0);
        const int nseg = a.nseg;
        const int seg_rows = BN / nseg;
        const int per = nseg / PAIR;
        // B rows of this CTA: the tile's CTA share (one segment) or its stacked segments
        const int g0 = nseg == 1 ? tl.g : tl.g + static_cast<int>(rank) * per;
        const int nb = nseg == 1 ? 1 : per;
        const int yb = nseg == 1 ? tl.n_loc * BN + static_cast<int>(rank) * CTA_ROWS : tl.n_loc * seg_rows;
        const int b_step = nseg == 1 ? 0 : seg_rows * BK * 2;
        const int xa_ext = a.xa_base[tl.g];
        for (int kb = 0; kb < nkb; ++kb) {
          if (!mbar_wait(&empty_bar[stage], phase ^ 1, &abort_flag, a.status)) {
            ok = false;
            break;
          }
          uint8_t* sa = smem + stage * STAGE_BYTES;
          uint8_t* sb = sa + A_BYTES;
          // the MMA-issuing CTA's full barrier counts the bytes of both CTAs
          if (leader) {
            mbar_arrive_expect_tx(&full_bar[stage], PAIR * STAGE_BYTES);
            armed_parity[stage] = phase;
          }
          const bool ext = kb == a.num_kb;
          const CUtensorMap* mA = ext ? &a.tmXA : &a.tmA;
          const CUtensorMap* mB = ext ? &a.tmBX[g0] : &a.tmB[g0];
          const int xa = ext ? xa_ext : kb * BK;
          const int xb = ext ? 0 : kb * BK;
          if constexpr (PAIR == 2) {
            const uint32_t bar = mapa_shared(&full_bar[stage], 0);
            tma_load_2d_pair(sa, mA, bar, xa, m0);
            for (int j = 0; j < nb; ++j) tma_load_2d_pair(sb + j * b_step, mB + j, bar, xb, yb);
          } else {
            tma_load_2d(sa, mA, &full_bar[stage], xa, m0);
            for (int j = 0; j < nb; ++j) tma_load_2d(sb + j * b_step, mB + j, &full_bar[stage], xb, yb);
          }
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
      }
      if (!ok) {
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
      int stage = 0;
      uint32_t phase = 0;
      int it = 0;
      bool ok = true;
      bool issued = false;
      const uint32_t idesc = idesc_bf16_f32(BM * PAIR, BN);
      for (int t = unit; t < a.total_tiles && ok; t += n_units, ++it) {
        const Tile tl = decode_tile(t, a);
        const int acc = it & 1;
        const uint32_t acc_phase = (it >> 1) & 1;
        if (!mbar_wait<PAIR == 2>(&tempty_bar[acc], acc_phase ^ 1, &abort_flag, a.status)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * BN;
        const int ext_steps = a.ext_on[tl.g] ? a.ext_steps[tl.g] : 0;
        auto mma = [&](uint64_t ad, uint64_t bd, uint32_t accum) {
          if constexpr (PAIR == 2)
            mma_bf16_ss_pair(d_tmem, ad, bd, idesc, accum);
          else
            mma_bf16_ss(d_tmem, ad, bd, idesc, accum);
        };
        auto release = [&]() {
          if constexpr (PAIR == 2) mma_commit_pair(&empty_bar[stage], 0x3); else mma_commit(&empty_bar[stage]);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1;
          }
        };
        for (int kb = 0; kb < a.num_kb; ++kb) {
          if (!mbar_wait(&full_bar[stage], phase, &abort_flag, a.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sa = smem_u32(smem + stage * STAGE_BYTES);
          const uint64_t ad = smem_desc(sa, 16, 1024, kSwizzle128B);
          const uint64_t bd = smem_desc(sa + A_BYTES, 16, 1024, kSwizzle128B);
          // K = 16 steps advance 32 bytes = 2 units of the descriptor's start-address field
#pragma unroll
          for (int k = 0; k < BK / 16; ++k) mma(ad + 2 * k, bd + 2 * k, (kb > 0 || k > 0) ? 1u : 0u);
          issued = true;
          release();
        }
        if (ok && ext_steps > 0) {
          if (!mbar_wait(&full_bar[stage], phase, &abort_flag, a.status)) {
            ok = false;
          } else {
            tc_fence_after();
            const uint32_t sa = smem_u32(smem + stage * STAGE_BYTES);
            const uint64_t ad = smem_desc(sa, 16, 1024, kSwizzle128B);
            const uint64_t bd = smem_desc(sa + A_BYTES, 16, 1024, kSwizzle128B);
            for (int k = 0; k < ext_steps; ++k) mma(ad + 2 * k, bd + 2 * k, 1u);
            release();
          }
        }
        if (!ok) break;
        if constexpr (PAIR == 2) mma_commit_pair(&tfull_bar[acc], 0x3); else mma_commit(&tfull_bar[acc]);
      }
      if (!ok && issued) {
        if constexpr (PAIR == 2) mma_commit_pair(&drain_bar, 0x1); else mma_commit(&drain_bar);
        volatile int never = 0;
        mbar_wait(&drain_bar, 0, &never, nullptr);
      }
    }
  } else {
    // ------------------------------------------------------------ epilogue (warps 2..5, every CTA)
    const int quarter = warp & 3;  // TMEM lane quarter this warp may access
    const int row_in_cta = quarter * 32 + lane;
    uint32_t tempty_addr[2];
    for (int i = 0; i < 2; ++i)
      tempty_addr[i] = PAIR == 2 ? mapa_shared(&tempty_bar[i], 0) : smem_u32(&tempty_bar[i]);
    int it = 0;
    for (int t = unit; t < a.total_tiles; t += n_units, ++it) {
      const Tile tl = decode_tile(t, a);
      const int acc = it & 1;
      const uint32_t acc_phase = (it >> 1) & 1;
      // warp-uniform outcome: the TMEM loads of the epilogue are warp-collective
      if (!__all_sync(0xffffffffu, mbar_wait(&tfull_bar[acc], acc_phase, &abort_flag, a.status)))
        break;
      tc_fence_after();
      const uint32_t tacc = tmem_base + (static_cast<uint32_t>(quarter * 32) << 16) + acc * BN;
      epilogue_tile<BN>(a, tl, tacc, tl.m_blk * (BM * PAIR) + static_cast<int>(rank) * BM + row_in_cta);
      // the accumulator is free once this warp's TMEM loads have completed (tcgen05.wait::ld in
      // the epilogue); the tile's global stores need not be visible first, so the arrival on
      // the MMA-issuing CTA's barrier is relaxed
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        if constexpr (PAIR == 2) mbar_arrive_cluster_relaxed(tempty_addr[acc]); else mbar_arrive(&tempty_bar[acc]);
      }
    }
  }

  tc_fence_before();
  if constexpr (PAIR == 2) cluster_sync(); else __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    if constexpr (PAIR == 2) tmem_dealloc_pair(tmem_base, TMEM_COLS); else tmem_dealloc(tmem_base, TMEM_COLS);
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

template <int BN, int STAGES, int PAIR>
cudaError_t launch_impl(const GemmArgs& args, int num_sms, cudaStream_t stream) {
  constexpr int smem = STAGES * (BM * BK * 2 + (BN / PAIR) * BK * 2) + 1024;
  auto kern = gemm_tc_kernel<BN, STAGES, PAIR>;
  // the attributes and the co-resident cluster count are per device
  static PerDevice once;
  static std::atomic<int> units_of[64];
  int dev = 0, max_units = 0;
  if (!once.pending(&dev)) {
    max_units = units_of[dev].load(std::memory_order_relaxed);
  } else {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    if (PAIR == 2) {
      e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 0);
      cudaLaunchConfig_t cfg = {};
      cudaLaunchAttribute attr[1];
      attr[0].id = cudaLaunchAttributeClusterDimension;
      attr[0].val.clusterDim.x = 2;
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
      max_units = std::max(1, std::min(clusters, num_sms / 2));
    } else {
      max_units = num_sms;
    }
    if (dev >= 0 && dev < 64) units_of[dev].store(max_units, std::memory_order_relaxed);
    once.done(dev);
  }
  const int units = std::max(1, std::min(max_units, args.total_tiles));
  if (PAIR == 1) {
    kern<<<units, kThreads, smem, stream>>>(args);
    return cudaGetLastError();
  }
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.gridDim = dim3(2 * units);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, args);
}

}  // namespace

cudaError_t launch_gemm(const GemmDesc& d, int bn, int num_sms, cudaStream_t stream) {
  GemmArgs a;
  std::memset(&a, 0, sizeof(a));
  // the 256-wide projection tiles run on CTA pairs; the narrow LoRA-down tiles on single CTAs
  if (bn == 256 && d.nseg != 1 && d.nseg != 2) return cudaErrorInvalidValue;
  const int pair = bn == 256 ? 2 : 1;
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
  if (any_ext) {
    if (!d.XA || d.ldxa < kXaCols) return cudaErrorInvalidValue;
    if (!make_map(&a.tmXA, d.XA, d.M, d.ldxa, d.ldxa, BM, BK, CU_TENSOR_MAP_SWIZZLE_128B))
      return cudaErrorInvalidValue;
    for (int i = 0; i < 3; ++i) {
      int src = (i < nmaps && d.BX[i]) ? i : -1;
      if (src < 0)
        for (int j = 0; j < nmaps; ++j)
          if (d.BX[j]) src = j;
      if (src < 0) return cudaErrorInvalidValue;
      if (!make_map(&a.tmBX[i], d.BX[src], d.B_rows[src], BK, BK, b_box, BK,
                    CU_TENSOR_MAP_SWIZZLE_128B))
        return cudaErrorInvalidValue;
    }
    for (int g = 0; g < d.ngroups; ++g) {
      if (!d.ext_on[g]) continue;
      // the 64-wide block must lie inside the XA row, 16-byte aligned (TMA x coordinate)
      if (d.xa_base[g] < 0 || d.xa_base[g] % 8 != 0 || d.xa_base[g] + BK > kXaCols ||
          d.ext_steps[g] < 1 || d.ext_steps[g] > BK / 16)
        return cudaErrorInvalidValue;
      for (int s = 0; s < (d.ngroups == 1 ? d.nseg : 1); ++s)
        if (!d.BX[g + s]) return cudaErrorInvalidValue;
    }
  } else {
    a.tmXA = a.tmA;
    for (int i = 0; i < 3; ++i) a.tmBX[i] = a.tmB[i];
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
  if (pair == 2) return launch_impl<256, 6, 2>(a, num_sms, stream);
  switch (bn) {
    case 48: return launch_impl<48, 8, 1>(a, num_sms, stream);
    case 32: return launch_impl<32, 8, 1>(a, num_sms, stream);
    case 16: return launch_impl<16, 8, 1>(a, num_sms, stream);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace crf
