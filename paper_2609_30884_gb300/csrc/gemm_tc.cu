// Persistent tcgen05 GEMM for sm_103a with fused LoRA-up and fused epilogues.
//
//   D[128 x BN] = A[128 x K] * B[BN x K]^T  (+ XA[128 x 16] * BL[BN x 16]^T)
//
// One CTA per SM; warp 0 issues TMA loads into a STAGES-deep shared-memory
// ring, warp 1 allocates TMEM and issues tcgen05.mma from one thread into one
// of two TMEM accumulators (so the epilogue of tile i overlaps the main loop of
// tile i+1), warps 2..5 drain the accumulator (one TMEM lane = one output row
// per thread) through the fused epilogue. Operands are bf16, K-major, staged
// with 128-byte swizzle; accumulation is fp32 in TMEM.
//
// The unmerged adapter term (alpha/r) (x A^T) B^T of every adapted projection
// (Eq. S3 with W = W0 + (alpha/r) B A) enters as one extra K = 16 block per
// tile: the rank-padded down product XA (computed by this same kernel with a
// narrow tile, epilogue kEpiScaleBf16) against the B factor rows of the tile.
#include "common.cuh"
#include "kernels.h"

#include <algorithm>
#include <cstdio>
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
  CUtensorMap tmBL[3];
  int M, K, num_kb;
  int ngroups, nseg;
  int group_tiles[3];
  int group_cols[3];
  int lora_on[3][3];
  int xa_col[3][3];
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

__device__ __forceinline__ bool group_has_lora(const GemmArgs& a, int g) {
  return a.lora_on[g][0] | a.lora_on[g][1] | a.lora_on[g][2];
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
                                              int row_in_tile) {
  const int row = tl.m_blk * BM + row_in_tile;
  const bool row_ok = row < a.M;
  uint32_t r0[16], r1[16];
  float v[16], w[16];

  if (a.epi == kEpiScaleBf16 || a.epi == kEpiResid) {
    const int col0 = tl.n_loc * BN;
    const int ncols = a.group_cols[tl.g];
#pragma unroll 1
    for (int c = 0; c < BN; c += 16) {
      tmem_ld16(tacc + c, r0);
      tmem_ld_wait();
      const int col = col0 + c;
      if (!row_ok || col >= ncols) continue;
      const int n = min(16, ncols - col);
      if (a.epi == kEpiScaleBf16) {
        // hi = bf16(v), lo = bf16(v - hi): the pair carries the product to ~16 mantissa bits
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          v[j] = __uint_as_float(r0[j]) * a.scale;
          w[j] = v[j] - __bfloat162float(__float2bfloat16_rn(v[j]));
        }
        store_bf16_n(a.out + (size_t)row * a.ldo + kXaLoCol + col, w, n);
      } else {
        if (n >= 16) {
          load16_bf16(a.resid + (size_t)row * a.ld_resid + col, w);
        } else {
#pragma unroll
          for (int j = 0; j < 16; ++j)
            w[j] = j < n ? __bfloat162float(a.resid[(size_t)row * a.ld_resid + col + j]) : 0.f;
        }
#pragma unroll
        for (int j = 0; j < 16; ++j) v[j] = w[j] + __uint_as_float(r0[j]);
      }
      store_bf16_n(a.out + (size_t)row * a.ldo + col, v, n);
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
      const int page = pt[pos / kPage];
      __nv_bfloat16* base = (g == 1) ? a.kpages : a.vpages;
      dst_row = base + ((size_t)page * a.n_kv_heads * kPage + (pos % kPage)) * d;
      head_stride = (size_t)kPage * d;
    }
  }
  const float2* rope_row = a.rope + (size_t)pos * half;
#pragma unroll 1
  for (int hh = 0; hh < BN / d; ++hh) {
    const int head = (tl.n_loc * BN) / d + hh;
    const int gcol = head * d;
#pragma unroll 1
    for (int i0 = 0; i0 < half; i0 += 16) {
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
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          v[j] += __bfloat162float(bias[gcol + i0 + j]);
          w[j] += __bfloat162float(bias[gcol + half + i0 + j]);
        }
      }
      if (g < 2) {
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          const float2 cs = rope_row[i0 + j];
          const float x1 = v[j], x2 = w[j];
          v[j] = x1 * cs.x - x2 * cs.y;
          w[j] = x2 * cs.x + x1 * cs.y;
        }
      }
      __nv_bfloat16* dst = dst_row + head * head_stride;
      store16_bf16(dst + i0, v);
      store16_bf16(dst + half + i0, w);
    }
  }
}

template <int BN, int STAGES>
__global__ void __launch_bounds__(kThreads, 1) gemm_tc_kernel(const __grid_constant__ GemmArgs a) {
  constexpr int A_BYTES = BM * BK * 2;
  constexpr int B_BYTES = BN * BK * 2;
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

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&tfull_bar[i], 1);
      mbar_init(&tempty_bar[i], 4);
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
    tmem_alloc(&tmem_base_sh, TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = tmem_base_sh;

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      int armed_parity[STAGES];
      for (int s = 0; s < STAGES; ++s) armed_parity[s] = -1;
      bool ok = true;
      for (int t = blockIdx.x; t < a.total_tiles && ok; t += gridDim.x) {
        const Tile tl = decode_tile(t, a);
        const int m0 = tl.m_blk * BM;
        const int seg_rows = BN / a.nseg;
        const int nkb = a.num_kb + (group_has_lora(a, tl.g) ? 1 : 0);
        for (int kb = 0; kb < nkb; ++kb) {
          if (!mbar_wait(&empty_bar[stage], phase ^ 1, &abort_flag, a.status)) {
            ok = false;
            break;
          }
          uint8_t* sa = smem + stage * STAGE_BYTES;
          uint8_t* sb = sa + A_BYTES;
          if (kb < a.num_kb) {
            mbar_arrive_expect_tx(&full_bar[stage], STAGE_BYTES);
            tma_load_2d(sa, &a.tmA, &full_bar[stage], kb * BK, m0);
            for (int s = 0; s < a.nseg; ++s)
              tma_load_2d(sb + s * seg_rows * BK * 2, &a.tmB[tl.g + s], &full_bar[stage], kb * BK,
                          tl.n_loc * seg_rows);
          } else {
            // Extension block: per adapted segment s, the XA slice [128 x 16] of that
            // module (A slot + s * 4 KB) and the B-factor rows of the tile (B slot).
            // A slot: [hi | lo] slices of 4 KB per adapted segment (at most 2 segments here)
            uint32_t bytes = 0;
            for (int s = 0; s < a.nseg; ++s)
              if (a.lora_on[tl.g][s]) bytes += 2 * BM * kRankPad * 2 + seg_rows * kRankPad * 2;
            mbar_arrive_expect_tx(&full_bar[stage], bytes);
            for (int s = 0; s < a.nseg; ++s) {
              if (!a.lora_on[tl.g][s]) continue;
              tma_load_2d(sa + (2 * s) * BM * kRankPad * 2, &a.tmXA, &full_bar[stage],
                          a.xa_col[tl.g][s], m0);
              tma_load_2d(sa + (2 * s + 1) * BM * kRankPad * 2, &a.tmXA, &full_bar[stage],
                          a.xa_col[tl.g][s] + kXaLoCol, m0);
              tma_load_2d(sb + s * seg_rows * kRankPad * 2, &a.tmBL[tl.g + s], &full_bar[stage], 0,
                          tl.n_loc * seg_rows);
            }
          }
          armed_parity[stage] = phase;
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
      }
      if (!ok) {
        // Let every copy already issued land before the CTA can exit.
        for (int s = 0; s < STAGES; ++s)
          if (armed_parity[s] >= 0) {
            volatile int never = 0;
            mbar_wait(&full_bar[s], static_cast<uint32_t>(armed_parity[s]), &never, nullptr);
          }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      int it = 0;
      bool ok = true;
      bool issued = false;
      const uint32_t idesc_main = idesc_bf16_f32(BM, BN);
      for (int t = blockIdx.x; t < a.total_tiles && ok; t += gridDim.x, ++it) {
        const Tile tl = decode_tile(t, a);
        const int acc = it & 1;
        const uint32_t acc_phase = (it >> 1) & 1;
        if (!mbar_wait(&tempty_bar[acc], acc_phase ^ 1, &abort_flag, a.status)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * BN;
        const bool lora = group_has_lora(a, tl.g);
        const int seg_rows = BN / a.nseg;
        const int nkb = a.num_kb + (lora ? 1 : 0);
        for (int kb = 0; kb < nkb; ++kb) {
          if (!mbar_wait(&full_bar[stage], phase, &abort_flag, a.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sa = smem_u32(smem + stage * STAGE_BYTES);
          const uint32_t sb = sa + A_BYTES;
          if (kb < a.num_kb) {
#pragma unroll
            for (int k = 0; k < BK / 16; ++k) {
              const uint64_t ad = smem_desc(sa + k * 32, 16, 1024, kSwizzle128B);
              const uint64_t bd = smem_desc(sb + k * 32, 16, 1024, kSwizzle128B);
              mma_bf16_ss(d_tmem, ad, bd, idesc_main, (kb > 0 || k > 0) ? 1u : 0u);
            }
          } else {
            const uint32_t idesc_seg = idesc_bf16_f32(BM, seg_rows);
            for (int s = 0; s < a.nseg; ++s) {
              if (!a.lora_on[tl.g][s]) continue;
              const uint64_t bd = smem_desc(sb + s * seg_rows * kRankPad * 2, 16, 256, kSwizzle32B);
#pragma unroll
              for (int h = 0; h < 2; ++h) {
                const uint64_t ad =
                    smem_desc(sa + (2 * s + h) * BM * kRankPad * 2, 16, 256, kSwizzle32B);
                mma_bf16_ss(d_tmem + s * seg_rows, ad, bd, idesc_seg, 1u);
              }
            }
          }
          issued = true;
          mma_commit(&empty_bar[stage]);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
        if (!ok) break;
        mma_commit(&tfull_bar[acc]);
      }
      if (!ok && issued) {
        mma_commit(&drain_bar);
        volatile int never = 0;
        mbar_wait(&drain_bar, 0, &never, nullptr);
      }
    }
  } else {
    // ------------------------------------------------------------ epilogue (warps 2..5)
    const int quarter = warp & 3;  // TMEM lane quarter this warp may access
    const int row_in_tile = quarter * 32 + lane;
    int it = 0;
    for (int t = blockIdx.x; t < a.total_tiles; t += gridDim.x, ++it) {
      const Tile tl = decode_tile(t, a);
      const int acc = it & 1;
      const uint32_t acc_phase = (it >> 1) & 1;
      // warp-uniform outcome: the TMEM loads of the epilogue are warp-collective
      if (!__all_sync(0xffffffffu, mbar_wait(&tfull_bar[acc], acc_phase, &abort_flag, a.status)))
        break;
      tc_fence_after();
      const uint32_t tacc = tmem_base + (static_cast<uint32_t>(quarter * 32) << 16) + acc * BN;
      epilogue_tile<BN>(a, tl, tacc, row_in_tile);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty_bar[acc]);
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, TMEM_COLS);
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

template <int BN, int STAGES>
cudaError_t launch_impl(const GemmArgs& args, int num_sms, cudaStream_t stream) {
  constexpr int smem = STAGES * (BM * BK * 2 + BN * BK * 2) + 1024;
  auto kern = gemm_tc_kernel<BN, STAGES>;
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  const int grid = std::max(1, std::min(num_sms, args.total_tiles));
  kern<<<grid, kThreads, smem, stream>>>(args);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_gemm(const GemmDesc& d, int bn, int num_sms, cudaStream_t stream) {
  GemmArgs a;
  std::memset(&a, 0, sizeof(a));
  const int seg_rows = bn / d.nseg;
  if (!make_map(&a.tmA, d.A, d.M, d.K, d.lda, BM, BK, CU_TENSOR_MAP_SWIZZLE_128B))
    return cudaErrorInvalidValue;
  const int nmaps = d.ngroups + d.nseg - 1;
  for (int i = 0; i < 3; ++i) {
    const int src = i < nmaps ? i : 0;  // unused slots alias a valid map
    if (!make_map(&a.tmB[i], d.B[src], d.B_rows[src], d.K, d.ldb[src], seg_rows, BK,
                  CU_TENSOR_MAP_SWIZZLE_128B))
      return cudaErrorInvalidValue;
  }
  bool any_lora = false;
  for (int g = 0; g < 3; ++g)
    for (int s = 0; s < 3; ++s) any_lora |= d.lora_on[g][s] != 0;
  if (any_lora && d.nseg > 2) return cudaErrorInvalidValue;  // A slot holds 2 hi/lo pairs
  if (any_lora) {
    if (!make_map(&a.tmXA, d.XA, d.M, d.ldxa, d.ldxa, BM, kRankPad, CU_TENSOR_MAP_SWIZZLE_32B))
      return cudaErrorInvalidValue;
    for (int i = 0; i < 3; ++i) {
      int src = -1;
      if (i < nmaps && d.BL[i]) src = i;
      if (src < 0)
        for (int j = 0; j < nmaps; ++j)
          if (d.BL[j]) src = j;
      if (src < 0) return cudaErrorInvalidValue;
      if (!make_map(&a.tmBL[i], d.BL[src], d.B_rows[src], d.rank, d.rank, seg_rows, kRankPad,
                    CU_TENSOR_MAP_SWIZZLE_32B))
        return cudaErrorInvalidValue;
    }
  } else {
    a.tmXA = a.tmA;
    for (int i = 0; i < 3; ++i) a.tmBL[i] = a.tmB[i];
  }
  a.M = d.M;
  a.K = d.K;
  a.num_kb = (d.K + BK - 1) / BK;
  a.ngroups = d.ngroups;
  a.nseg = d.nseg;
  a.total_n = 0;
  for (int g = 0; g < d.ngroups; ++g) {
    const int cols_per_tile = (d.nseg > 1 && d.epi == kEpiSwiGLU) ? seg_rows : bn;
    a.group_cols[g] = d.group_cols[g];
    a.group_tiles[g] = (d.nseg > 1 && d.epi != kEpiSwiGLU) ? 1
                                                            : (d.group_cols[g] + cols_per_tile - 1) /
                                                                  cols_per_tile;
    a.total_n += a.group_tiles[g];
  }
  for (int g = 0; g < 3; ++g)
    for (int s = 0; s < 3; ++s) {
      a.lora_on[g][s] = d.lora_on[g][s];
      a.xa_col[g][s] = d.xa_col[g][s];
    }
  a.row_tiles = (d.M + BM - 1) / BM;
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
  if (a.total_tiles == 0) return cudaSuccess;
  switch (bn) {
    case 256: return launch_impl<256, 4>(a, num_sms, stream);
    case 128: return launch_impl<128, 6>(a, num_sms, stream);
    case 48: return launch_impl<48, 8>(a, num_sms, stream);
    case 32: return launch_impl<32, 8>(a, num_sms, stream);
    case 16: return launch_impl<16, 8>(a, num_sms, stream);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace crf
