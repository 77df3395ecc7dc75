// Causal grouped-query prefill attention on tcgen05, reading K/V from the
// paged cache of the layer being recomputed: the self-attention of every layer
// that bounded recovery re-executes over the complete prefix (Section 4.2),
// whose K/V are the cache entries of Eq. 1 (projections of Eq. S3).
//
// softmax(q k^T / sqrt(d) + causal mask) v over the whole prefix for every
// query head; query head h reads kv head h / (Hq / Hkv). One CTA takes two
// consecutive 128-row query tiles of one head (rows q0 .. q0+255): both read
// the same K/V tiles except the last, which only the second tile needs, so
// each K/V tile is fetched once for 256 query rows whatever the group size.
// Warp roles (three warpgroups; setmaxnreg moves registers from the first to
// the two softmax warpgroups):
//   warp 0      TMA producer: the two Q tiles, then K0, V0, K1, V1, ... (8
//               pages of 16 tokens each per tile, one 4-D copy per page)
//               through one ring of kSlots shared-memory slots, so page
//               gathers run two kv tiles ahead
//   warp 1      allocates TMEM and issues tcgen05.mma from one thread:
//               S_t = Q_t K^T into TMEM, then O_t += P_t V with P_t read
//               from TMEM (A operand) and V an MN-major shared operand.
//               The SM's MMA queue holds about two instructions, so every
//               wait or commit of this thread between two blocks of MMAs
//               leaves the tensor pipe idle: per kv tile it waits only for
//               each query tile's P and commits only each tile's S; the
//               softmax warps check that the next K/V tiles have landed and
//               release consumed ring slots
//   warps 2-3   idle
//   warps 4-7   softmax of query tile 0, warps 8-11 of query tile 1: one thread
//               per query row; S from TMEM, online max / sum in fp32, P back
//               into TMEM as bf16 over the S columns; O rescaled in TMEM only
//               when the running max grows by more than 2^8
// TMEM: S0 | S1 | O0 | O1, 128 columns each. Every wait is bounded.
//
// K/V slot layout: the 128 keys of a tile in 16 groups of 8 keys, group c at
// c * HALVES * 1024 bytes, and within a group one 1 KB 128B-swizzled atom per
// 64-column half of the head dimension. A page (two groups, both halves) is
// then one contiguous 4 KB box of a 4-D view of the pool: a K or V tile is 8
// copies (one per page, 16 with one copy per page and half); both MMAs see a
// uniform 8-row stride.
#include "common.cuh"
#include "kernels.h"

#include <algorithm>
#include <cfloat>
#include <cstring>

namespace crf {

namespace {

constexpr int kM = 128;          // query rows per tile
constexpr int kN = 128;          // keys per kv tile
constexpr int kPagesPerTile = kN / kPage;
constexpr int kSlots = 5;        // K/V ring: slot of sequence item i = i % kSlots (K(j): 2j, V(j): 2j+1)
constexpr int kThreadsAttn = 384;
// setmaxnreg split: warpgroup 0 (producer, MMA) keeps kRegsCtl registers per thread, the
// two softmax warpgroups take kRegsSoftmax; the sum must fit what the CTA launched with.
constexpr int kRegsCtl = 56;
constexpr int kRegsSoftmax = 208;
constexpr int kRegsNeeded = 128 * kRegsCtl + 256 * kRegsSoftmax;
constexpr float kRescaleThreshold = 8.0f;  // log2 units

struct AttnTcArgs {
  CUtensorMap tmQ;  // q [rows, Hq*D], box {64, 128}
  CUtensorMap tmK;  // K pool viewed as {64 cols, 8 rows, D/64 halves, rows/8}, box {64, 8, D/64, 2}
  CUtensorMap tmV;
  __nv_bfloat16* out;
  int ldo;
  int n_q_heads, n_kv_heads, group;
  int total_items;
  ReqTable req;
  int* status;
  const int* abort;
};

struct AttnWork {
  int req, qp, head, g;
};

// Items: (request, 256-row query pair, head), longest (latest) query pairs first.
__device__ __forceinline__ bool attn_work(const AttnTcArgs& a, int idx, AttnWork& w) {
  for (int i = 0; i < a.req.n; ++i) {
    const int nqp = (a.req.len[i] + 2 * kM - 1) / (2 * kM);
    const int items = nqp * a.n_q_heads;
    if (idx < items) {
      w.req = i;
      w.qp = nqp - 1 - idx / a.n_q_heads;
      w.head = idx % a.n_q_heads;
      w.g = w.head / a.group;
      return true;
    }
    idx -= items;
  }
  return false;
}

// One query row's share of one kv tile: S row (128 raw scores) from TMEM, running max
// and sum update, O rescaled in TMEM when the max grows by more than 2^8, and P (bf16,
// unnormalised) written back over the S columns. MASK (diagonal tile only) sets every
// key index above `lim` to -inf; the common off-diagonal instance has no masking code.
template <int D, bool MASK>
__device__ __forceinline__ void softmax_tile(uint32_t tS, uint32_t tO, bool first, int lim,
                                             float sl2, float& m_run, float& l_run) {
  uint32_t sr[4][32];
#pragma unroll
  for (int c = 0; c < 4; ++c) tmem_ld32(tS + c * 32, sr[c]);
  tmem_ld_wait();
  // eight independent max chains (one thread owns the whole row), two scores per max
  float mx[8];
#pragma unroll
  for (int k = 0; k < 8; ++k) mx[k] = -INFINITY;
#pragma unroll
  for (int c = 0; c < 4; ++c)
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      float x0 = __uint_as_float(sr[c][2 * i]), x1 = __uint_as_float(sr[c][2 * i + 1]);
      if (MASK) {
        if (c * 32 + 2 * i > lim) {
          x0 = -INFINITY;
          sr[c][2 * i] = __float_as_uint(x0);
        }
        if (c * 32 + 2 * i + 1 > lim) {
          x1 = -INFINITY;
          sr[c][2 * i + 1] = __float_as_uint(x1);
        }
      }
      mx[i & 7] = fmax3(mx[i & 7], x0, x1);
    }
  const float mt = fmax3(fmax3(mx[0], mx[1], mx[2]), fmax3(mx[3], mx[4], mx[5]), fmaxf(mx[6], mx[7]));
  // the running max is kept in raw score units; p = 2^(s * sl2 - m_run * sl2)
  const bool grow = (mt - m_run) * sl2 > kRescaleThreshold;
  const float alpha = grow ? ex2_approx((m_run - mt) * sl2) : 1.0f;
  if (!first && __any_sync(0xffffffffu, grow)) {
#pragma unroll 1
    for (int c = 0; c < D / 32; ++c) {
      uint32_t o[32];
      tmem_ld32(tO + c * 32, o);
      tmem_ld_wait();
#pragma unroll
      for (int i = 0; i < 32; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * alpha);
      tmem_st32(tO + c * 32, o);
    }
    tmem_st_wait();
  }
  if (grow) {
    l_run *= alpha;
    m_run = mt;
  }
  const float neg_m = -m_run * sl2;
  // x = s * sl2 - m * sl2 and the row sum on paired fp32 lanes: two keys per instruction
  const uint64_t sl2x2 = f32x2(sl2, sl2), negm2 = f32x2(neg_m, neg_m);
  uint64_t rs2[2] = {f32x2(0.f, 0.f), f32x2(0.f, 0.f)};
#pragma unroll
  for (int c = 0; c < 4; ++c) {
    // keys 32c .. 32c+31 -> packed bf16 P columns 16c .. 16c+15 (S already in registers)
    uint32_t pk[16];
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      float x0, x1;
      f32x2_split(fma_f32x2(f32x2(__uint_as_float(sr[c][2 * i]), __uint_as_float(sr[c][2 * i + 1])),
                            sl2x2, negm2), x0, x1);
      const float p0 = ex2_approx(x0);
      const float p1 = ex2_approx(x1);
      rs2[i & 1] = add_f32x2(rs2[i & 1], f32x2(p0, p1));
      pk[i] = pack_bf16(p0, p1);
    }
    tmem_st16(tS + 16 * c, pk);
  }
  tmem_st_wait();
  float r0, r1, r2, r3;
  f32x2_split(rs2[0], r0, r1);
  f32x2_split(rs2[1], r2, r3);
  l_run += (r0 + r1) + (r2 + r3);
}

__device__ __forceinline__ void regs_dec_ctl() {
  asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(kRegsCtl));
}
__device__ __forceinline__ void regs_inc_softmax() {
  asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(kRegsSoftmax));
}

template <int D>
__global__ void __launch_bounds__(kThreadsAttn, 1) attn_tc_kernel(const __grid_constant__ AttnTcArgs a) {
  constexpr int HALVES = D / 64;
  constexpr int Q_BYTES = kM * D * 2;
  constexpr int KV_BYTES = kN * D * 2;
  constexpr int HALF_ROWS_BYTES = kN * 128;  // one 64-column half of a 128-row Q tile
  constexpr int GROUP_BYTES = HALVES * 1024;  // 8 keys, all halves, in a K/V slot
  constexpr uint32_t TMEM_COLS = 512;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sQ = smem;
  uint8_t* sKV = sQ + 2 * Q_BYTES;  // kSlots x KV_BYTES
  __shared__ __align__(8) uint64_t q_full, o_full, drain_bar;
  __shared__ __align__(8) uint64_t kv_full[kSlots], kv_empty[kSlots];
  __shared__ __align__(8) uint64_t s_full[2], p_full[2];
  __shared__ uint32_t tmem_base_sh;
  __shared__ volatile int abort_flag;

  AttnWork w;
  if (call_aborted(a.abort) || !attn_work(a, blockIdx.x, w)) return;
  const int n = a.req.len[w.req];
  const int row0 = a.req.row0[w.req];
  const int32_t* pt = a.req.page_table[w.req];
  const int q0 = w.qp * 2 * kM;
  const int ntiles = q0 + kM < n ? 2 : 1;
  const int kv_end = min(q0 + ntiles * kM, n);
  const int J = (kv_end + kN - 1) / kN;    // kv tiles of the last query tile
  const int J0 = ntiles == 2 ? J - 1 : J;  // kv tiles of query tile 0 (its diagonal is tile J0-1)
  const int n_pages = (n + kPage - 1) / kPage;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    mbar_init(&q_full, 1);
    mbar_init(&o_full, 1);
    mbar_init(&drain_bar, 1);
    for (int i = 0; i < 2; ++i) {

      mbar_init(&s_full[i], 1);
      mbar_init(&p_full[i], 4);
    }
    // a ring slot is free once the softmax of every query tile has released it
    for (int i = 0; i < kSlots; ++i) {
      mbar_init(&kv_full[i], 1);
      mbar_init(&kv_empty[i], ntiles);
    }
    abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 1) {
    tmem_alloc(&tmem_base_sh, TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base_sh;

  if (warp < 4) {
    // setmaxnreg inside each role's branch: the softmax code is never reachable from here
    regs_dec_ctl();
    if (warp == 0 && lane == 0) {
      // ---------------------------------------------------------------- producer
      bool ok = true;
      int armed[kSlots];
      for (int i = 0; i < kSlots; ++i) armed[i] = -1;
      mbar_arrive_expect_tx(&q_full, ntiles * Q_BYTES);
      for (int t = 0; t < ntiles; ++t)
        for (int h = 0; h < HALVES; ++h)
          tma_load_2d(sQ + t * Q_BYTES + h * (kM * 128), &a.tmQ, &q_full, w.head * D + 64 * h,
                      row0 + q0 + t * kM);
      int slot = 0;
      uint32_t ph = 0;
      for (int i = 0; i < 2 * J && ok; ++i) {
        const int j = i >> 1;
        const int kv = i & 1;
        if (!mbar_wait(&kv_empty[slot], ph ^ 1, &abort_flag, a.status)) {
          ok = false;
          break;
        }
        mbar_arrive_expect_tx(&kv_full[slot], KV_BYTES);
        uint8_t* dst = sKV + slot * KV_BYTES;
        const CUtensorMap* map = kv == 0 ? &a.tmK : &a.tmV;
        for (int p = 0; p < kPagesPerTile; ++p) {
          // pages past the prefix repeat the last page: finite data, masked below
          const int page = checked_page(pt[min(j * kPagesPerTile + p, n_pages - 1)], a.req.num_pages, a.status);
          const int group = (page * a.n_kv_heads + w.g) * (kPage / 8);
          tma_load_4d(dst + p * (kPage / 8) * GROUP_BYTES, map, &kv_full[slot], 0, 0, 0, group);
        }
        armed[slot] = ph;
        if (++slot == kSlots) {
          slot = 0;
          ph ^= 1;
        }
      }
      if (!ok) {
        volatile int never = 0;
        for (int i = 0; i < kSlots; ++i)
          if (armed[i] >= 0) mbar_wait(&kv_full[i], armed[i], &never, nullptr);
        mbar_wait(&q_full, 0, &never, nullptr);
      }
    } else if (warp == 1) {
      // -------------------------------------------------------------- MMA issuer
      // Order: S0(0) S1(0) | PV0(j) S0(j+1) PV1(j) S1(j+1) | ... so that the softmax of one
      // query tile overlaps the products of the other; query tile 0 stops one kv tile early
      // (its diagonal), after which tile 1 runs alone. tcgen05.mma of one thread execute in
      // issue order, so S_t(j+1) overwrites the S/P columns only after PV_t(j) has read P_t(j).
      if (lane == 0) {
        bool ok = mbar_wait(&q_full, 0, &abort_flag, a.status);
        bool issued = false;
        const uint32_t idesc_s = idesc_bf16_f32(kM, kN);
        const uint32_t idesc_o = idesc_bf16_f32(kM, D, false, true);
        // ring position of sequence item i (K(j): i = 2j, V(j): i = 2j + 1)
        auto slot_of = [](int i) { return i % kSlots; };
        auto parity_of = [](int i) { return static_cast<uint32_t>((i / kSlots) & 1); };
        auto issue_s = [&](int t, int ks) {
          const uint32_t kb = smem_u32(sKV + ks * KV_BYTES);
          const uint32_t qb = smem_u32(sQ + t * Q_BYTES);
  #pragma unroll
          for (int kk = 0; kk < D / 16; ++kk) {
            const uint32_t in_row = (kk & 3) * 32;
            mma_bf16_ss(tmem + t * 128,
                        smem_desc(qb + (kk >> 2) * HALF_ROWS_BYTES + in_row, 16, 1024, kSwizzle128B),
                        smem_desc(kb + (kk >> 2) * 1024 + in_row, 16, GROUP_BYTES, kSwizzle128B),
                        idesc_s, kk > 0 ? 1u : 0u);
          }
          mma_commit(&s_full[t]);
        };
        if (ok) ok = mbar_wait(&kv_full[slot_of(0)], parity_of(0), &abort_flag, a.status);
        if (ok) {
          tc_fence_after();
          for (int t = 0; t < ntiles; ++t) issue_s(t, slot_of(0));
          issued = true;
        }
        for (int j = 0; j < J && ok; ++j) {
          const uint32_t vb = smem_u32(sKV + slot_of(2 * j + 1) * KV_BYTES);
          const int ks = slot_of(2 * j + 2);
          for (int t = (j < J0 ? 0 : 1); t < ntiles; ++t) {
            // phase j of p_full[t]: P_t(j) is in TMEM, and V(j) and K(j + 1) have landed
            if (!mbar_wait(&p_full[t], j & 1, &abort_flag, a.status)) {
              ok = false;
              break;
            }
            tc_fence_after();
  #pragma unroll
            for (int kk = 0; kk < kN / 16; ++kk) {
              // P: 16 keys = 8 packed bf16x2 columns; V: 16 key rows = two 8-key groups
              mma_bf16_ts(tmem + 256 + t * 128, tmem + t * 128 + kk * 8,
                          smem_desc(vb + kk * 2 * GROUP_BYTES, 1024, GROUP_BYTES, kSwizzle128B), idesc_o,
                          (j > 0 || kk > 0) ? 1u : 0u);
            }
            if (j + 1 < (t == 0 ? J0 : J)) issue_s(t, ks);
          }
        }
        if (ok) {
          mma_commit(&o_full);
        } else if (issued) {
          mma_commit(&drain_bar);
          volatile int never = 0;
          mbar_wait(&drain_bar, 0, &never, nullptr);
        }
      }
    }
  } else {
    regs_inc_softmax();
    // ---------------------------------------------------------------- softmax + epilogue
    const int t = (warp - 4) >> 2;
    const int quarter = warp & 3;
    const int r = quarter * 32 + lane;  // query row within the tile (= TMEM lane)
    if (t < ntiles) {
      const uint32_t lane_off = static_cast<uint32_t>(quarter * 32) << 16;
      const uint32_t tS = tmem + lane_off + t * 128;
      const uint32_t tO = tmem + lane_off + 256 + t * 128;
      const float sl2 = 1.4426950408889634f * rsqrtf(static_cast<float>(D));
      const int qrow = q0 + t * kM + r;
      const int Jt = t == 0 ? J0 : J;
      float m_run = -INFINITY, l_run = 0.f;  // running max in raw score units
      bool ok = true;
      for (int j = 0; j < Jt && ok; ++j) {
        // warp-uniform outcome: the TMEM accesses below are warp-collective
        ok = __all_sync(0xffffffffu, mbar_wait(&s_full[t], j & 1, &abort_flag, a.status));
        if (!ok) break;
        tc_fence_after();
        // S_t(j) complete: so is P_t(j - 1) V(j - 1), issued before it; this tile is done with
        // K(j) and V(j - 1). Items past the last one the producer refills are released too
        // (harmless: no wait ever targets those phases).
        if (quarter == 0 && lane == 0) {
          mbar_arrive(&kv_empty[(2 * j) % kSlots]);
          if (j > 0) mbar_arrive(&kv_empty[(2 * j - 1) % kSlots]);
        }
        const int k0 = j * kN;
        const bool last = j == Jt - 1;
        if (last) {
          // keys above min(query row, prefix end - 1) are masked on the diagonal tile
          softmax_tile<D, true>(tS, tO, j == 0, min(qrow, kv_end - 1) - k0, sl2, m_run, l_run);
        } else {
          softmax_tile<D, false>(tS, tO, j == 0, 0, sl2, m_run, l_run);
        }
        if (last && t == ntiles - 1 && kv_end - k0 < kN) {
          // zero V rows past the prefix so that 0 * stale data cannot produce NaN (only the
          // last query tile reads the last kv tile)
          const int vi = 2 * j + 1;
          ok = __all_sync(0xffffffffu, mbar_wait(&kv_full[vi % kSlots], (vi / kSlots) & 1, &abort_flag, a.status));
          if (ok) {
            uint8_t* vt = sKV + (vi % kSlots) * KV_BYTES;
            const int zr0 = kv_end - k0;
            const int chunks = (kN - zr0) * HALVES * 8;
            for (int i = threadIdx.x - 128 - 128 * t; i < chunks; i += 128) {
              const int rr = zr0 + i / (HALVES * 8);
              const int h = (i / 8) % HALVES;
              const int ch = i % 8;
              *reinterpret_cast<uint4*>(vt + (rr >> 3) * GROUP_BYTES + h * 1024 + (rr & 7) * 128 + ch * 16) =
                  make_uint4(0, 0, 0, 0);
            }
            fence_proxy_async_smem();
          }
        }
        if (quarter == 0 && ok) {
          // the products that read P_t(j) also need V(j) and (unless this is the tile's last
          // kv tile) K(j + 1): hand over only once they have landed
          const int vi = 2 * j + 1;
          ok = __all_sync(0xffffffffu, mbar_wait(&kv_full[vi % kSlots], (vi / kSlots) & 1, &abort_flag, a.status));
          if (ok && !last)
            ok = __all_sync(0xffffffffu, mbar_wait(&kv_full[(vi + 1) % kSlots], ((vi + 1) / kSlots) & 1,
                                                   &abort_flag, a.status));
          if (!ok) break;
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&p_full[t]);
      }
      if (ok) ok = __all_sync(0xffffffffu, mbar_wait(&o_full, 0, &abort_flag, a.status));
      if (ok) {
        tc_fence_after();
        const float inv = l_run > 0.f ? 1.0f / l_run : 0.f;
        const bool store = qrow < n;
        __nv_bfloat16* dst = a.out + (size_t)(row0 + qrow) * a.ldo + w.head * D;
        for (int c = 0; c < D / 32; ++c) {
          uint32_t o[32];
          tmem_ld32(tO + c * 32, o);
          tmem_ld_wait();
          if (store) {
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              uint4 v;
              v.x = pack_bf16(__uint_as_float(o[8 * i + 0]) * inv, __uint_as_float(o[8 * i + 1]) * inv);
              v.y = pack_bf16(__uint_as_float(o[8 * i + 2]) * inv, __uint_as_float(o[8 * i + 3]) * inv);
              v.z = pack_bf16(__uint_as_float(o[8 * i + 4]) * inv, __uint_as_float(o[8 * i + 5]) * inv);
              v.w = pack_bf16(__uint_as_float(o[8 * i + 6]) * inv, __uint_as_float(o[8 * i + 7]) * inv);
              reinterpret_cast<uint4*>(dst + c * 32)[i] = v;
            }
          }
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
}

using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                   const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                   const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode() {
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

// K or V pool of one layer, [rows = pages * Hkv * 16, D] row-major, as the 4-D view
// {64 columns, 8 rows, D/64 halves, rows/8 groups} with strides {2D, 128, 16D} bytes; the box
// {64, 8, D/64, 2} is one page of one kv head, written to shared memory group-major, halves
// inside a group, each half an 8 x 128-byte swizzled atom.
bool map_pool(CUtensorMap* m, const void* base, long rows, int D) {
  EncodeTiledFn fn = encode();
  if (!fn) return false;
  cuuint64_t dims[4] = {64, 8, static_cast<cuuint64_t>(D / 64), static_cast<cuuint64_t>(rows / 8)};
  cuuint64_t strides[3] = {static_cast<cuuint64_t>(D) * 2, 128, static_cast<cuuint64_t>(D) * 16};
  cuuint32_t box[4] = {64, 8, static_cast<cuuint32_t>(D / 64), kPage / 8};
  cuuint32_t estr[4] = {1, 1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool map2d(CUtensorMap* m, const void* base, long rows, int cols, int box_rows) {
  EncodeTiledFn fn = encode();
  if (!fn) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(cols) * 2};
  cuuint32_t box[2] = {64, static_cast<cuuint32_t>(box_rows)};
  cuuint32_t estr[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int D>
cudaError_t launch_tc(const AttnTcArgs& args, cudaStream_t stream) {
  constexpr int smem = 2 * kM * D * 2 + kSlots * kN * D * 2 + 1024;
  static PerDevice once;
  int dev = 0;
  if (once.pending(&dev)) {
    cudaError_t e = cudaFuncSetAttribute(attn_tc_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    // setmaxnreg.inc waits until the CTA's register pool can serve it: refuse to launch a
    // build whose per-thread launch count leaves the split short
    cudaFuncAttributes fa;
    e = cudaFuncGetAttributes(&fa, attn_tc_kernel<D>);
    if (e != cudaSuccess) return e;
    if (fa.numRegs * kThreadsAttn < kRegsNeeded) return cudaErrorInvalidConfiguration;
    once.done(dev);
  }
  attn_tc_kernel<D><<<args.total_items, kThreadsAttn, smem, stream>>>(args);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_attention_tc(const AttnDesc& d, int num_pages, int total_rows, cudaStream_t stream) {
  AttnTcArgs a;
  std::memset(&a, 0, sizeof(a));
  const int D = d.head_dim;
  if (!map2d(&a.tmQ, d.q, total_rows, d.n_q_heads * D, kM)) return cudaErrorInvalidValue;
  const long pool_rows = static_cast<long>(num_pages) * d.n_kv_heads * kPage;
  if (!map_pool(&a.tmK, d.kpages, pool_rows, D)) return cudaErrorInvalidValue;
  if (!map_pool(&a.tmV, d.vpages, pool_rows, D)) return cudaErrorInvalidValue;
  a.out = d.out;
  a.ldo = d.ldo;
  a.n_q_heads = d.n_q_heads;
  a.n_kv_heads = d.n_kv_heads;
  a.group = d.n_q_heads / d.n_kv_heads;
  a.req = d.req;
  a.status = d.status;
  a.abort = d.abort;
  a.total_items = 0;
  for (int i = 0; i < d.req.n; ++i)
    a.total_items += ((d.req.len[i] + 2 * kM - 1) / (2 * kM)) * d.n_q_heads;
  if (a.total_items == 0) return cudaSuccess;
  if (D == 128) return launch_tc<128>(a, stream);
  if (D == 64) return launch_tc<64>(a, stream);
  return cudaErrorInvalidValue;
}

}  // namespace crf
