// Decode attention of single rows over the paged cache (the first-step rows carried
// through layers e..N-1: the hybrid execution of Section 3.1 that reads historical states
// from the window end on, and the generated tokens of Section S2.1): for each decode row at
// position pos and query head h,
//   o = softmax(q k^T / sqrt(d)) v over the cached keys 0..pos-1 of that layer plus the
//   row's own fresh (k, v) at position pos.
// The work is memory-bound (K and V of every cached position are read once): the positions
// are cut into chunks of 128 and streamed.
//   decode_attn_stream  one block per SM, walking a run of consecutive chunks of one (row,
//                       kv head) through a two- or three-stage ring: a copy warp gathers the next
//                       chunk's K and V pages with TMA (128-byte swizzle) while four compute
//                       warps score the current one. The group's query heads (padded to 16 rows)
//                       meet the chunk on mma.sync m16n8k16 (each warp takes a 32-key slice),
//                       q entering as a bf16 pair hi + lo so the scores keep fp32 accuracy (K
//                       is exact in bf16). Every warp keeps an online-softmax state (running
//                       max, sum and unnormalised o in registers, P as the A operand of P V)
//                       over its slices; at the end the warps and the row's own key and value
//                       (scored and added in fp32) meet at the common max in a fixed order and
//                       the block writes one (max, sum, unnormalised o) partial in log2 units.
//                       The chunks per block are the fewest that keep all blocks in one wave;
//   decode_attn_merge   one block per (query head, row, 32-column slice): rescales the blocks'
//                       partials to the common max and normalises, every partial's loads
//                       independent of the others.
#include "common.cuh"
#include "kernels.h"

#include <algorithm>
#include <cfloat>
#include <cstring>

namespace crf {

namespace {

constexpr int kChunk = 128;                     // positions per chunk
// The K/V ring depth is the stream kernel's template parameter (64 KB per stage at d = 128): 3
// for a single decode row, 2 from two rows on (measured per generation step: one row 4.39 ->
// 4.22 ms with 3 stages, eight rows 6.5 -> 10.4 ms)
constexpr int kThreadsStream = 160;             // four compute warps + one copy warp
constexpr int kMaxGroup = 8;

__device__ __forceinline__ void named_bar_sync_dec(int id, int nthreads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}
// Named barrier that also ANDs a flag over its threads: the compute warps take every later
// barrier together even when one of them gave up on a timed-out wait.
__device__ __forceinline__ bool named_bar_and_dec(int id, int nthreads, bool flag) {
  uint32_t out;
  asm volatile(
      "{\n\t.reg .pred pi, po;\n\t"
      "setp.ne.u32 pi, %1, 0;\n\t"
      "bar.red.and.pred po, %2, %3, pi;\n\t"
      "selp.u32 %0, 1, 0, po;\n\t}"
      : "=r"(out)
      : "r"(flag ? 1u : 0u), "r"(id), "r"(nthreads)
      : "memory");
  return out != 0;
}

struct DecodeArgs {
  CUtensorMap tmK;  // K pool of the layer viewed as [pages*Hkv*16, d], box {64, 16}
  CUtensorMap tmV;
  DecodeAttnDesc d;
  int num_pages;
  int* status;
};

template <int D, int kStages>
__global__ void __launch_bounds__(kThreadsStream) decode_attn_stream(const __grid_constant__ DecodeArgs a) {
  constexpr int HALVES = D / 64;
  constexpr int HALF = kChunk * 128;     // bytes of one 64-column half of a K (or V) tile
  constexpr int TILE = HALVES * HALF;
  constexpr int QHALF = 16 * 128;        // one 64-column half of the 16-row Q tile
  const DecodeAttnDesc& p = a.d;
  griddep_begin();  // q, k, v of the rows come from the kernel before
  if (call_aborted(p.abort)) return;
  // block -> (row, kv head, its chunks c_beg .. c_end - 1, partial slot)
  int r = -1, g = 0, slot = 0, c_beg = 0, c_end = 0;
  {
    int b = blockIdx.x;
    for (int i = 0; i < p.rows; ++i) {
      const int chunks = p.pos[i] / kChunk + 1;
      const int bpp = (chunks + p.chunks_per_block - 1) / p.chunks_per_block;
      if (b < bpp * p.n_kv_heads) {
        r = i;
        g = b / bpp;
        slot = b % bpp;
        c_beg = slot * p.chunks_per_block;
        c_end = min(chunks, c_beg + p.chunks_per_block);
        break;
      }
      b -= bpp * p.n_kv_heads;
    }
  }
  if (r < 0) return;
  const int pos = p.pos[r];
  const int grp = p.n_q_heads / p.n_kv_heads;
  const bool self_here = c_end - 1 == pos / kChunk;  // the chunk holding the row's own position

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sKV = smem;                                      // [kStages][K tile | V tile]
  uint8_t* sQ = smem + 2 * kStages * TILE;                  // hi: [HALVES][16 rows][128 B], swizzled
  uint8_t* sQl = sQ + HALVES * QHALF;                       // lo, same layout
  __shared__ float red_m[4][16], red_l[4][16];
  __shared__ float s_self[16];  // the row's own key, scored in fp32
  __shared__ __align__(8) uint64_t full[kStages], empty[kStages];
  __shared__ volatile int abort_flag;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
    for (int i = 0; i < kStages; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], 4);
    }
    abort_flag = 0;
    fence_barrier_init();
  }
  __syncthreads();

  if (warp == 4) {
    // ---------------------------------------------------------------- producer
    if (lane == 0) {
      const int32_t* pt = p.page_table[r];
      int armed[kStages];
      for (int st = 0; st < kStages; ++st) armed[st] = -1;
      for (int c = c_beg; c < c_end; ++c) {
        const int i = c - c_beg, st = i % kStages;
        if (i >= kStages && !mbar_wait(&empty[st], (i / kStages - 1) & 1, &abort_flag, a.status)) break;
        const int t0 = c * kChunk;
        const int pages = (min(kChunk, pos - t0) + kPage - 1) / kPage;
        uint8_t* sK = sKV + st * 2 * TILE;
        uint8_t* sV = sK + TILE;
        if (pages == 0) {
          mbar_arrive(&full[st]);  // only the row's own key here: nothing to copy
        } else {
          mbar_arrive_expect_tx(&full[st], 2 * pages * HALVES * kPage * 128);
          for (int pg = 0; pg < pages; ++pg) {
            const int page = checked_page(pt[t0 / kPage + pg], a.num_pages, a.status);
            const int row = (page * p.n_kv_heads + g) * kPage;
            for (int h = 0; h < HALVES; ++h) {
              const int off = h * HALF + pg * (kPage * 128);
              tma_load_2d(sK + off, &a.tmK, &full[st], 64 * h, row);
              tma_load_2d(sV + off, &a.tmV, &full[st], 64 * h, row);
            }
          }
          armed[st] = (i / kStages) & 1;
        }
      }
      // copies still in flight land before the block's shared memory is released
      volatile int never = 0;
      for (int st = 0; st < kStages; ++st)
        if (armed[st] >= 0) mbar_wait(&full[st], armed[st], &never, nullptr);
    }
    return;
  }

  // -------------------------------------------------------------------- compute warps 0..3
  // q of the group's heads (rows >= grp zero) as bf16 hi + lo, pre-scaled so scores are in
  // log2 units
  const float qscale = 1.4426950408889634f * rsqrtf(static_cast<float>(D));
  const float* qrow0 = p.q + (size_t)r * p.n_q_heads * D + (size_t)(g * grp) * D;
  for (int i = tid; i < 16 * (D / 2); i += 128) {
    const int row = i / (D / 2), d = 2 * (i % (D / 2));
    float v0 = 0.f, v1 = 0.f;
    if (row < grp) {
      v0 = qrow0[(size_t)row * D + d] * qscale;
      v1 = qrow0[(size_t)row * D + d + 1] * qscale;
    }
    const float h0 = __bfloat162float(__float2bfloat16_rn(v0));
    const float h1 = __bfloat162float(__float2bfloat16_rn(v1));
    const int c = (d % 64) / 8;
    const uint32_t off = (d / 64) * QHALF + row * 128 + ((c ^ (row & 7)) << 4) + (d % 8) * 2;
    *reinterpret_cast<uint32_t*>(sQ + off) = pack_bf16(h0, h1);
    *reinterpret_cast<uint32_t*>(sQl + off) = pack_bf16(v0 - h0, v1 - h1);
  }
  if (self_here) {
    // the row's own key, scored in fp32 (warp w takes heads w, w + 4)
    const float* ks = p.k_self + (size_t)r * p.n_kv_heads * D + g * D;
    for (int h = warp; h < grp; h += 4) {
      float dot = 0.f;
      for (int d = lane; d < D; d += 32) dot += qrow0[(size_t)h * D + d] * ks[d];
      dot = warp_sum(dot);
      if (lane == 0) s_self[h] = dot * qscale;
    }
  }
  named_bar_sync_dec(1, 128);

  const uint32_t q_base = smem_u32(sQ), ql_base = smem_u32(sQl);
  const int mi = lane >> 3, li = lane & 7;  // ldmatrix: matrix index, row within it
  const int r0 = lane >> 2, cq = 2 * (lane & 3);
  // this warp's running state over its 32-key slice of every chunk: max and partial sum of
  // rows r0 and r0 + 8 (log2 units), and its share of the unnormalised o
  float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
  float O[D / 8][4];
#pragma unroll
  for (int dn = 0; dn < D / 8; ++dn)
#pragma unroll
    for (int e = 0; e < 4; ++e) O[dn][e] = 0.f;
  bool ok = true;
  for (int c = c_beg; c < c_end; ++c) {
    const int i = c - c_beg, st = i % kStages;
    const int t0 = c * kChunk;
    const int n_cached = min(kChunk, pos - t0);  // cached keys of this chunk
    if (ok) ok = __all_sync(0xffffffffu, mbar_wait(&full[st], (i / kStages) & 1, &abort_flag, a.status));
    const uint32_t k_base = smem_u32(sKV + st * 2 * TILE), v_base = k_base + TILE;
    if (n_cached < kChunk) {
      // the last chunk: V rows from the row's own slot on are zeroed (its value is added in
      // fp32 at the end, and 0 * stale data must not produce NaN in P V); all four warps read
      // every row of V, so they meet before the products
      if (ok) {
        for (int q = tid; q < (kChunk - n_cached) * HALVES * 8; q += 128) {
          const int t2 = n_cached + q / (HALVES * 8);
          const int hf = (q / 8) % HALVES, cc = q % 8;
          *reinterpret_cast<uint4*>(sKV + st * 2 * TILE + TILE + hf * HALF + t2 * 128 + (cc << 4)) =
              make_uint4(0, 0, 0, 0);
        }
      }
      ok = named_bar_and_dec(1, 128, ok);
    }
    if (ok) {
      // 1. S = Q K^T for this warp's 32 keys: 4 n-tiles of 8 keys
      float S[4][4];
#pragma unroll
      for (int nt = 0; nt < 4; ++nt)
#pragma unroll
        for (int e = 0; e < 4; ++e) S[nt][e] = 0.f;
#pragma unroll
      for (int ks = 0; ks < D / 16; ++ks) {
        const int hf = ks / 4;
        uint32_t af[4], al[4];
        {
          const int row = (mi & 1) * 8 + li, cc = 2 * (ks % 4) + (mi >> 1);
          const uint32_t off = hf * QHALF + row * 128 + ((cc ^ (row & 7)) << 4);
          ldsm_x4(q_base + off, af[0], af[1], af[2], af[3]);
          ldsm_x4(ql_base + off, al[0], al[1], al[2], al[3]);
        }
#pragma unroll
        for (int np = 0; np < 2; ++np) {
          const int key = warp * 32 + (2 * np + (mi >> 1)) * 8 + li, cc = 2 * (ks % 4) + (mi & 1);
          uint32_t b0, b1, b2, b3;
          ldsm_x4(k_base + hf * HALF + key * 128 + ((cc ^ (key & 7)) << 4), b0, b1, b2, b3);
          mma16816(S[2 * np], af, b0, b1);
          mma16816(S[2 * np + 1], af, b2, b3);
          mma16816(S[2 * np], al, b0, b1);
          mma16816(S[2 * np + 1], al, b2, b3);
        }
      }
      // 2. mask the keys past this chunk's cached ones, online max / sum update of the slice
      float c0 = -INFINITY, c1 = -INFINITY;
#pragma unroll
      for (int nt = 0; nt < 4; ++nt)
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          const bool valid = warp * 32 + nt * 8 + cq + e < n_cached;
          S[nt][e] = valid ? S[nt][e] : -INFINITY;
          S[nt][2 + e] = valid ? S[nt][2 + e] : -INFINITY;
          c0 = fmaxf(c0, S[nt][e]);
          c1 = fmaxf(c1, S[nt][2 + e]);
        }
#pragma unroll
      for (int o = 1; o <= 2; o <<= 1) {
        c0 = fmaxf(c0, __shfl_xor_sync(0xffffffffu, c0, o));
        c1 = fmaxf(c1, __shfl_xor_sync(0xffffffffu, c1, o));
      }
      const float n0 = fmaxf(m0, c0), n1 = fmaxf(m1, c1);
      // a slice with nothing valid so far keeps max -inf: no rescale, P = 0
      const float a0 = n0 == -INFINITY ? 1.f : ex2_approx(m0 - n0);
      const float a1 = n1 == -INFINITY ? 1.f : ex2_approx(m1 - n1);
      const float z0 = n0 == -INFINITY ? 0.f : n0, z1 = n1 == -INFINITY ? 0.f : n1;
      m0 = n0;
      m1 = n1;
      l0 *= a0;
      l1 *= a1;
#pragma unroll
      for (int dn = 0; dn < D / 8; ++dn) {
        O[dn][0] *= a0;
        O[dn][1] *= a0;
        O[dn][2] *= a1;
        O[dn][3] *= a1;
      }
#pragma unroll
      for (int nt = 0; nt < 4; ++nt)
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          S[nt][e] = ex2_approx(S[nt][e] - z0);
          S[nt][2 + e] = ex2_approx(S[nt][2 + e] - z1);
          l0 += S[nt][e];
          l1 += S[nt][2 + e];
        }
      // 3. O += P V over this warp's keys: P from the S fragments, V by transposing loads
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        uint32_t pa[4];
        pa[0] = pack_bf16(S[2 * j][0], S[2 * j][1]);
        pa[1] = pack_bf16(S[2 * j][2], S[2 * j][3]);
        pa[2] = pack_bf16(S[2 * j + 1][0], S[2 * j + 1][1]);
        pa[3] = pack_bf16(S[2 * j + 1][2], S[2 * j + 1][3]);
        const int key = warp * 32 + 16 * j + (mi & 1) * 8 + li;
#pragma unroll
        for (int dp = 0; dp < D / 16; ++dp) {
          const int gc = 2 * dp + (mi >> 1);  // 16-byte chunk of the row (8 dims)
          const int hf = gc / 8, cc = gc % 8;
          uint32_t b0, b1, b2, b3;
          ldsm_x4_t(v_base + hf * HALF + key * 128 + ((cc ^ (key & 7)) << 4), b0, b1, b2, b3);
          mma16816(O[2 * dp], pa, b0, b1);
          mma16816(O[2 * dp + 1], pa, b2, b3);
        }
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&empty[st]);  // this warp is done with the stage
  }

  // 4. the warps' states (and the row's own key) meet at the common max, in a fixed order
#pragma unroll
  for (int o = 1; o <= 2; o <<= 1) {
    l0 += __shfl_xor_sync(0xffffffffu, l0, o);
    l1 += __shfl_xor_sync(0xffffffffu, l1, o);
  }
  if ((lane & 3) == 0) {
    red_m[warp][r0] = m0;
    red_m[warp][r0 + 8] = m1;
  }
  ok = named_bar_and_dec(1, 128, ok);
  float M0 = red_m[0][r0], M1 = red_m[0][r0 + 8];
#pragma unroll
  for (int w = 1; w < 4; ++w) {
    M0 = fmaxf(M0, red_m[w][r0]);
    M1 = fmaxf(M1, red_m[w][r0 + 8]);
  }
  if (self_here) {
    M0 = fmaxf(M0, r0 < grp ? s_self[r0] : -INFINITY);
    M1 = fmaxf(M1, r0 + 8 < grp ? s_self[r0 + 8] : -INFINITY);
  }
  const float f0 = m0 == -INFINITY ? 0.f : ex2_approx(m0 - M0);
  const float f1 = m1 == -INFINITY ? 0.f : ex2_approx(m1 - M1);
  if ((lane & 3) == 0) {
    red_l[warp][r0] = l0 * f0;
    red_l[warp][r0 + 8] = l1 * f1;
  }
  // partial o of every warp summed over the stage-0 K tile (every copy has landed and been read)
  float (*o_red)[D] = reinterpret_cast<float (*)[D]>(sKV);
  static_assert(16 * D * 4 <= TILE, "partial products fit in a K tile");
  for (int w = 0; w < 4; ++w) {
    if (warp == w && ok) {
#pragma unroll
      for (int dn = 0; dn < D / 8; ++dn) {
        float* p0 = &o_red[r0][dn * 8 + cq];
        float* p1 = &o_red[r0 + 8][dn * 8 + cq];
        if (w == 0) {
          p0[0] = O[dn][0] * f0;
          p0[1] = O[dn][1] * f0;
          p1[0] = O[dn][2] * f1;
          p1[1] = O[dn][3] * f1;
        } else {
          p0[0] += O[dn][0] * f0;
          p0[1] += O[dn][1] * f0;
          p1[0] += O[dn][2] * f1;
          p1[1] += O[dn][3] * f1;
        }
      }
    }
    named_bar_sync_dec(1, 128);
  }
  if (!ok) return;
  const float* vs = p.v_self + (size_t)r * p.n_kv_heads * D + g * D;
  for (int q = tid; q < grp * D; q += 128) {
    const int h = q / D, d = q % D;
    float M = red_m[0][h];
#pragma unroll
    for (int w = 1; w < 4; ++w) M = fmaxf(M, red_m[w][h]);
    float ps = 0.f;
    if (self_here) {
      M = fmaxf(M, s_self[h]);
      ps = ex2_approx(s_self[h] - M);
    }
    float* out = p.part + (((size_t)r * p.n_q_heads + g * grp + h) * p.splits + slot) * (D + 2);
    out[d] = o_red[h][d] + ps * vs[d];
    if (d == 0) {
      float L = ps;
#pragma unroll
      for (int w = 0; w < 4; ++w) L += red_l[w][h];
      out[D] = M;
      out[D + 1] = L;
    }
  }
}

// One block per (query head, row, 32-column slice of o): warp w takes chunks w, w + 4, ...
// (each chunk's loads independent of the others), lane = one output column; the warps'
// sums meet in a fixed order.
template <int D>
__global__ void __launch_bounds__(128) decode_attn_merge(const DecodeAttnDesc p) {
  griddep_begin();  // the partials come from decode_attn_stream
  const int h = blockIdx.x, r = blockIdx.y, tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int col = blockIdx.z * 32 + lane;
  const int n_chunks = (p.pos[r] / kChunk + p.chunks_per_block) / p.chunks_per_block;  // partials
  const float* base = p.part + ((size_t)r * p.n_q_heads + h) * p.splits * (D + 2);
  __shared__ float red_m[4], red_l[4], red_o[4][32];
  float m = -INFINITY;
  for (int s = tid; s < n_chunks; s += 128) m = fmaxf(m, base[(size_t)s * (D + 2) + D]);
  m = warp_max(m);
  if (lane == 0) red_m[warp] = m;
  __syncthreads();
  m = fmaxf(fmaxf(red_m[0], red_m[1]), fmaxf(red_m[2], red_m[3]));
  float acc = 0.f, l = 0.f;
#pragma unroll 8
  for (int s = warp; s < n_chunks; s += 4) {
    const float* ps = base + (size_t)s * (D + 2);
    const float f = ex2_approx(ps[D] - m);
    l += f * ps[D + 1];
    acc += f * ps[col];
  }
  red_o[warp][lane] = acc;
  if (lane == 0) red_l[warp] = l;
  __syncthreads();
  if (warp == 0) {
    const float o = (red_o[0][lane] + red_o[1][lane]) + (red_o[2][lane] + red_o[3][lane]);
    const float L = (red_l[0] + red_l[1]) + (red_l[2] + red_l[3]);
    p.out[(size_t)r * p.n_q_heads * D + h * D + col] = o / L;
  }
}

using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                   const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                   const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn_dec() {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(ptr);
  }
  return fn;
}

bool pool_map(CUtensorMap* m, const void* base, long rows, int cols) {
  EncodeTiledFn fn = encode_fn_dec();
  if (!fn) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(cols) * 2};
  cuuint32_t box[2] = {64, static_cast<cuuint32_t>(kPage)};
  cuuint32_t estr[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int D, int kStages>
cudaError_t launch_dec(const DecodeArgs& args, int blocks, cudaStream_t stream) {
  constexpr int smem = 2 * kStages * kChunk * D * 2 + 2 * 16 * D * 2 + 1024;  // K/V stages, q hi/lo
  static PerDevice once;
  int dev = 0;
  if (once.pending(&dev)) {
    cudaError_t e =
        cudaFuncSetAttribute(decode_attn_stream<D, kStages>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    once.done(dev);
  }
  const DecodeAttnDesc& d = args.d;
  cudaError_t e =
      launch_kernel(decode_attn_stream<D, kStages>, dim3(blocks), dim3(kThreadsStream), smem, stream, args);
  if (e != cudaSuccess) return e;
  // d carries chunks_per_block
  return launch_kernel(decode_attn_merge<D>, dim3(d.n_q_heads, d.rows, D / 32), dim3(128), 0, stream, d);
}

}  // namespace

int decode_attention_splits(int max_positions) { return std::max(1, (max_positions + kChunk - 1) / kChunk); }

cudaError_t launch_decode_attention(const DecodeAttnDesc& d, int num_pages, int num_sms, int* status,
                                    cudaStream_t stream) {
  if (d.rows < 1) return cudaSuccess;
  if (d.n_q_heads % d.n_kv_heads != 0 || d.n_q_heads / d.n_kv_heads > kMaxGroup)
    return cudaErrorInvalidValue;
  int max_pos = 0;
  for (int r = 0; r < d.rows; ++r) max_pos = std::max(max_pos, d.pos[r]);
  if (max_pos / kChunk + 1 > d.splits) return cudaErrorInvalidValue;
  // one block per SM (two or three 64 KB K/V stages each), each streaming a run of consecutive chunks
  // of one (row, kv head): the fewest chunks per block that keeps every block in one wave
  if (num_sms < 1) return cudaErrorInvalidValue;
  long items = 0;
  for (int r = 0; r < d.rows; ++r) items += static_cast<long>(d.n_kv_heads) * (d.pos[r] / kChunk + 1);
  int cpb = static_cast<int>(std::max(1L, (items + num_sms - 1) / num_sms));
  auto blocks_for = [&](int c) {
    long b = 0;
    for (int r = 0; r < d.rows; ++r) b += static_cast<long>(d.n_kv_heads) * ((d.pos[r] / kChunk + c) / c);
    return b;
  };
  while (blocks_for(cpb) > num_sms) ++cpb;
  const int blocks = static_cast<int>(blocks_for(cpb));
  DecodeArgs a;
  std::memset(&a, 0, sizeof(a));
  const long pool_rows = static_cast<long>(num_pages) * d.n_kv_heads * kPage;
  if (!pool_map(&a.tmK, d.kpages, pool_rows, d.head_dim)) return cudaErrorInvalidValue;
  if (!pool_map(&a.tmV, d.vpages, pool_rows, d.head_dim)) return cudaErrorInvalidValue;
  a.d = d;
  a.d.chunks_per_block = cpb;
  a.num_pages = num_pages;
  a.status = status;
  const bool one_row = d.rows == 1;
  if (d.head_dim == 128) return one_row ? launch_dec<128, 3>(a, blocks, stream) : launch_dec<128, 2>(a, blocks, stream);
  if (d.head_dim == 64) return one_row ? launch_dec<64, 3>(a, blocks, stream) : launch_dec<64, 2>(a, blocks, stream);
  return cudaErrorInvalidValue;
}

}  // namespace crf
