// Decode attention of single rows over the paged cache (the first-step rows carried
// through layers e..N-1): for each decode row at position pos and query head h,
//   o = softmax(q k^T / sqrt(d)) v over the cached keys 0..pos-1 of that layer plus the
//   row's own fresh (k, v) at position pos.
// The work is memory-bound (K and V of every cached position are read once), so the
// positions are split into chunks of 128 that run as independent blocks:
//   decode_attn_chunk   one block per (chunk, kv head, row): TMA gathers the chunk's K and
//                       V pages (128-byte swizzle). The group's query heads (padded to 16
//                       rows) are scored against the chunk with mma.sync m16n8k16 (each warp
//                       takes 32 keys), q entering as a bf16 pair hi + lo so the scores keep
//                       fp32 accuracy (K is exact in bf16); the row's own key is scored and
//                       its value added in fp32. Softmax runs on the accumulator fragments,
//                       P stays in registers as the A operand of P V, and the warps' partial
//                       products are summed in shared memory in a fixed order. The chunk's
//                       (max, sum, unnormalised o) are written in log2 units;
//   decode_attn_merge   one block per (query head, row, 32-column slice): rescales the chunk
//                       partials to the common max and normalises, every chunk's loads
//                       independent of the others.
#include "common.cuh"
#include "kernels.h"

#include <algorithm>
#include <cfloat>
#include <cstring>

namespace crf {

namespace {

constexpr int kChunk = 128;                     // positions per block
constexpr int kThreadsChunk = 128;
constexpr int kMaxGroup = 8;

struct DecodeArgs {
  CUtensorMap tmK;  // K pool of the layer viewed as [pages*Hkv*16, d], box {64, 16}
  CUtensorMap tmV;
  DecodeAttnDesc d;
  int* status;
};

template <int D>
__global__ void __launch_bounds__(kThreadsChunk) decode_attn_chunk(const __grid_constant__ DecodeArgs a) {
  constexpr int HALVES = D / 64;
  constexpr int HALF = kChunk * 128;     // bytes of one 64-column half of a K (or V) tile
  constexpr int TILE = HALVES * HALF;
  constexpr int QHALF = 16 * 128;        // one 64-column half of the 16-row Q tile
  const DecodeAttnDesc& p = a.d;
  const int r = blockIdx.z, g = blockIdx.y, chunk = blockIdx.x;
  const int pos = p.pos[r];
  const int t0 = chunk * kChunk;
  if (t0 > pos) return;
  const int grp = p.n_q_heads / p.n_kv_heads;
  const int n_cached = min(kChunk, pos - t0);               // cached keys of this chunk
  const bool has_self = pos < t0 + kChunk;                  // the row's own key falls here
  const int n_valid = n_cached + (has_self ? 1 : 0);
  const int pages = (n_cached + kPage - 1) / kPage;

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sK = smem;
  uint8_t* sV = smem + TILE;
  uint8_t* sQ = smem + 2 * TILE;                            // hi: [HALVES][16 rows][128 B], swizzled
  uint8_t* sQl = sQ + HALVES * QHALF;                       // lo, same layout
  __shared__ __align__(16) float o_red[16][D];
  __shared__ float red_m[kThreadsChunk / 32][16], red_l[kThreadsChunk / 32][16];
  __shared__ float s_self[16], p_self[16];  // the row's own key: fp32 score, then weight
  __shared__ __align__(8) uint64_t full;
  __shared__ volatile int abort_flag;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
    mbar_init(&full, 1);
    abort_flag = 0;
    fence_barrier_init();
  }
  __syncthreads();
  if (tid == 0 && pages > 0) {
    const int32_t* pt = p.page_table[r];
    mbar_arrive_expect_tx(&full, 2 * pages * HALVES * kPage * 128);
    for (int i = 0; i < pages; ++i) {
      const int row = (pt[t0 / kPage + i] * p.n_kv_heads + g) * kPage;
      for (int h = 0; h < HALVES; ++h) {
        const int off = h * HALF + i * (kPage * 128);
        tma_load_2d(sK + off, &a.tmK, &full, 64 * h, row);
        tma_load_2d(sV + off, &a.tmV, &full, 64 * h, row);
      }
    }
  }
  // q of the group's heads (rows >= grp zero) as bf16 hi + lo, pre-scaled so scores are in
  // log2 units
  const float qscale = 1.4426950408889634f * rsqrtf(static_cast<float>(D));
  const float* qrow0 = p.q + (size_t)r * p.n_q_heads * D + (size_t)(g * grp) * D;
  for (int i = tid; i < 16 * (D / 2); i += kThreadsChunk) {
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
  // the row's own key, scored in fp32 (warp w takes heads w, w + 4)
  if (has_self) {
    const float* ks = p.k_self + (size_t)r * p.n_kv_heads * D + g * D;
    for (int h = warp; h < grp; h += kThreadsChunk / 32) {
      float dot = 0.f;
      for (int d = lane; d < D; d += 32) dot += qrow0[(size_t)h * D + d] * ks[d];
      dot = warp_sum(dot);
      if (lane == 0) s_self[h] = dot * qscale;
    }
  }
  bool ok = true;
  if (pages > 0) ok = mbar_wait(&full, 0, &abort_flag, a.status);
  if (!__syncthreads_and(ok)) return;
  // V rows from the row's own slot on are zeroed: its value is added in fp32 at the end, and
  // 0 * stale data must not produce NaN in P V (masked scores need no cleaning)
  if (has_self) {
    for (int i = tid; i < (kChunk - n_cached) * HALVES * 8; i += kThreadsChunk) {
      const int t2 = n_cached + i / (HALVES * 8);
      const int hf = (i / 8) % HALVES, c = i % 8;
      *reinterpret_cast<uint4*>(sV + hf * HALF + t2 * 128 + (c << 4)) = make_uint4(0, 0, 0, 0);
    }
  }
  __syncthreads();

  // 1. S = Q K^T for this warp's 32 keys: 4 n-tiles of 8 keys
  const uint32_t q_base = smem_u32(sQ), ql_base = smem_u32(sQl), k_base = smem_u32(sK),
                 v_base = smem_u32(sV);
  const int mi = lane >> 3, li = lane & 7;  // ldmatrix: matrix index, row within it
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
      const int row = (mi & 1) * 8 + li, c = 2 * (ks % 4) + (mi >> 1);
      const uint32_t off = hf * QHALF + row * 128 + ((c ^ (row & 7)) << 4);
      ldsm_x4(q_base + off, af[0], af[1], af[2], af[3]);
      ldsm_x4(ql_base + off, al[0], al[1], al[2], al[3]);
    }
#pragma unroll
    for (int np = 0; np < 2; ++np) {
      const int key = warp * 32 + (2 * np + (mi >> 1)) * 8 + li, c = 2 * (ks % 4) + (mi & 1);
      uint32_t b0, b1, b2, b3;
      ldsm_x4(k_base + hf * HALF + key * 128 + ((c ^ (key & 7)) << 4), b0, b1, b2, b3);
      mma16816(S[2 * np], af, b0, b1);
      mma16816(S[2 * np + 1], af, b2, b3);
      mma16816(S[2 * np], al, b0, b1);
      mma16816(S[2 * np + 1], al, b2, b3);
    }
  }
  // 2. mask, block row max, P = 2^(S - max), row sums
  const int r0 = lane >> 2, cq = 2 * (lane & 3);
  float m0 = -INFINITY, m1 = -INFINITY;
#pragma unroll
  for (int nt = 0; nt < 4; ++nt)
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      const int key = warp * 32 + nt * 8 + cq + e;
      const bool valid = key < n_valid;
      S[nt][e] = valid ? S[nt][e] : -INFINITY;
      S[nt][2 + e] = valid ? S[nt][2 + e] : -INFINITY;
      if (has_self && key == n_cached) {
        S[nt][e] = r0 < grp ? s_self[r0] : 0.f;
        S[nt][2 + e] = r0 + 8 < grp ? s_self[r0 + 8] : 0.f;
      }
      m0 = fmaxf(m0, S[nt][e]);
      m1 = fmaxf(m1, S[nt][2 + e]);
    }
#pragma unroll
  for (int o = 1; o <= 2; o <<= 1) {
    m0 = fmaxf(m0, __shfl_xor_sync(0xffffffffu, m0, o));
    m1 = fmaxf(m1, __shfl_xor_sync(0xffffffffu, m1, o));
  }
  if ((lane & 3) == 0) {
    red_m[warp][r0] = m0;
    red_m[warp][r0 + 8] = m1;
  }
  __syncthreads();
  float M0 = red_m[0][r0], M1 = red_m[0][r0 + 8];
#pragma unroll
  for (int w = 1; w < kThreadsChunk / 32; ++w) {
    M0 = fmaxf(M0, red_m[w][r0]);
    M1 = fmaxf(M1, red_m[w][r0 + 8]);
  }
  float l0 = 0.f, l1 = 0.f;
#pragma unroll
  for (int nt = 0; nt < 4; ++nt)
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      S[nt][e] = ex2_approx(S[nt][e] - M0);
      S[nt][2 + e] = ex2_approx(S[nt][2 + e] - M1);
      l0 += S[nt][e];
      l1 += S[nt][2 + e];
      if (has_self && warp * 32 + nt * 8 + cq + e == n_cached) {
        p_self[r0] = S[nt][e];
        p_self[r0 + 8] = S[nt][2 + e];
      }
    }
#pragma unroll
  for (int o = 1; o <= 2; o <<= 1) {
    l0 += __shfl_xor_sync(0xffffffffu, l0, o);
    l1 += __shfl_xor_sync(0xffffffffu, l1, o);
  }
  if ((lane & 3) == 0) {
    red_l[warp][r0] = l0;
    red_l[warp][r0 + 8] = l1;
  }
  // 3. O += P V over this warp's keys: P from the S fragments, V by transposing loads
  float O[D / 8][4];
#pragma unroll
  for (int dn = 0; dn < D / 8; ++dn)
#pragma unroll
    for (int e = 0; e < 4; ++e) O[dn][e] = 0.f;
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
      const int hf = gc / 8, c = gc % 8;
      uint32_t b0, b1, b2, b3;
      ldsm_x4_t(v_base + hf * HALF + key * 128 + ((c ^ (key & 7)) << 4), b0, b1, b2, b3);
      mma16816(O[2 * dp], pa, b0, b1);
      mma16816(O[2 * dp + 1], pa, b2, b3);
    }
  }
  // 4. sum the warps' partial products in warp order (a fixed order keeps every row's result
  // independent of what else is in the launch); write the chunk partial for the group's heads
  for (int w = 0; w < kThreadsChunk / 32; ++w) {
    if (warp == w) {
#pragma unroll
      for (int dn = 0; dn < D / 8; ++dn) {
        float* a0 = &o_red[r0][dn * 8 + cq];
        float* a1 = &o_red[r0 + 8][dn * 8 + cq];
        if (w == 0) {
          a0[0] = O[dn][0];
          a0[1] = O[dn][1];
          a1[0] = O[dn][2];
          a1[1] = O[dn][3];
        } else {
          a0[0] += O[dn][0];
          a0[1] += O[dn][1];
          a1[0] += O[dn][2];
          a1[1] += O[dn][3];
        }
      }
    }
    __syncthreads();
  }
  const float* vs = p.v_self + (size_t)r * p.n_kv_heads * D + g * D;
  for (int i = tid; i < grp * D; i += kThreadsChunk) {
    const int h = i / D, d = i % D;
    float* out = p.part + (((size_t)r * p.n_q_heads + g * grp + h) * p.splits + chunk) * (D + 2);
    out[d] = has_self ? o_red[h][d] + p_self[h] * vs[d] : o_red[h][d];
    if (d == 0) {
      float M = red_m[0][h], L = 0.f;
#pragma unroll
      for (int w = 1; w < kThreadsChunk / 32; ++w) M = fmaxf(M, red_m[w][h]);
#pragma unroll
      for (int w = 0; w < kThreadsChunk / 32; ++w) L += red_l[w][h];
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
  const int h = blockIdx.x, r = blockIdx.y, tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int col = blockIdx.z * 32 + lane;
  const int n_chunks = p.pos[r] / kChunk + 1;
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

template <int D>
cudaError_t launch_dec(const DecodeArgs& args, int chunks, cudaStream_t stream) {
  constexpr int smem = 2 * kChunk * D * 2 + 2 * 16 * D * 2 + 1024;
  static bool set = false;
  if (!set) {
    cudaError_t e = cudaFuncSetAttribute(decode_attn_chunk<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    set = true;
  }
  const DecodeAttnDesc& d = args.d;
  decode_attn_chunk<D><<<dim3(chunks, d.n_kv_heads, d.rows), kThreadsChunk, smem, stream>>>(args);
  decode_attn_merge<D><<<dim3(d.n_q_heads, d.rows, D / 32), 128, 0, stream>>>(d);
  return cudaGetLastError();
}

}  // namespace

int decode_attention_splits(int max_positions) { return std::max(1, (max_positions + kChunk - 1) / kChunk); }

cudaError_t launch_decode_attention(const DecodeAttnDesc& d, int num_pages, int* status,
                                    cudaStream_t stream) {
  if (d.rows < 1) return cudaSuccess;
  if (d.n_q_heads % d.n_kv_heads != 0 || d.n_q_heads / d.n_kv_heads > kMaxGroup)
    return cudaErrorInvalidValue;
  int max_pos = 0;
  for (int r = 0; r < d.rows; ++r) max_pos = std::max(max_pos, d.pos[r]);
  const int chunks = max_pos / kChunk + 1;
  if (chunks > d.splits) return cudaErrorInvalidValue;
  DecodeArgs a;
  std::memset(&a, 0, sizeof(a));
  const long pool_rows = static_cast<long>(num_pages) * d.n_kv_heads * kPage;
  if (!pool_map(&a.tmK, d.kpages, pool_rows, d.head_dim)) return cudaErrorInvalidValue;
  if (!pool_map(&a.tmV, d.vpages, pool_rows, d.head_dim)) return cudaErrorInvalidValue;
  a.d = d;
  a.status = status;
  if (d.head_dim == 128) return launch_dec<128>(a, chunks, stream);
  if (d.head_dim == 64) return launch_dec<64>(a, chunks, stream);
  return cudaErrorInvalidValue;
}

}  // namespace crf
