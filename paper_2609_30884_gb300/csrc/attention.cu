// Causal grouped-query prefill attention over the paged KV cache, and the
// single-row decode attention used to carry the last prefix row through the
// layers after a recomputed window.
//
// Prefill: softmax(q k^T / sqrt(d) + causal mask) v over the whole prefix, per
// query head; query head h reads kv head h / (Hq / Hkv). q arrives already
// rotated (RoPE is applied in the QKV projection epilogue, which also wrote
// this layer's rotated K and V into the pages), so the kernel reads K/V tiles
// straight from the 16-token pages of the request through its page table.
// Flash-style online softmax in fp32; bf16 operands on mma.sync m16n8k16.
#include "common.cuh"
#include "kernels.h"

#include <cfloat>

namespace crf {

namespace {

constexpr int kBM = 128;   // query rows per CTA (8 warps x 16 rows)
constexpr int kBN = 64;    // keys per iteration
constexpr int kWarps = 8;

__device__ __forceinline__ void cp_async16(void* smem, const void* gmem, bool valid) {
  const int sz = valid ? 16 : 0;
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_u32(smem)), "l"(gmem),
               "r"(sz)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                        uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                          uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void mma16816(float (&c)[4], const uint32_t (&a)[4], uint32_t b0,
                                         uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7},"
      " {%8, %9}, {%0, %1, %2, %3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// Row `r`, 16-byte chunk `c` of a tile whose rows are D*2 bytes: XOR-swizzled chunk.
template <int D>
__device__ __forceinline__ uint32_t swz(int r, int c) {
  return static_cast<uint32_t>(r * (D * 2) + ((c ^ (r & 7)) << 4));
}

struct Work {
  int req, qt, head;
};

__device__ __forceinline__ bool find_work(const ReqTable& rt, int hq, int idx, Work& w) {
  for (int i = 0; i < rt.n; ++i) {
    const int nqt = (rt.len[i] + kBM - 1) / kBM;
    const int items = nqt * hq;
    if (idx < items) {
      w.req = i;
      w.qt = nqt - 1 - idx / hq;  // longest (latest) query tiles first
      w.head = idx % hq;
      return true;
    }
    idx -= items;
  }
  return false;
}

template <int D>
__global__ void __launch_bounds__(kWarps * 32, 1) attn_prefill_kernel(const AttnDesc p) {
  extern __shared__ __align__(128) uint8_t smem[];
  uint8_t* sQ = smem;                              // [128][D]
  uint8_t* sK = sQ + kBM * D * 2;                  // [2][64][D]
  uint8_t* sV = sK + 2 * kBN * D * 2;              // [2][64][D]

  Work w;
  if (!find_work(p.req, p.n_q_heads, blockIdx.x, w)) return;
  const int n = p.req.len[w.req];
  const int row0 = p.req.row0[w.req];
  const int32_t* pt = p.req.page_table[w.req];
  const int q0 = w.qt * kBM;
  const int g = w.head / (p.n_q_heads / p.n_kv_heads);
  const int tid = threadIdx.x;
  const int warp = tid >> 5, lane = tid & 31;
  constexpr int CH = D / 8;  // 16-byte chunks per row

  // ---- load Q tile (rows past the prefix are zero)
  for (int i = tid; i < kBM * CH; i += kWarps * 32) {
    const int r = i / CH, c = i % CH;
    const bool ok = q0 + r < n;
    const __nv_bfloat16* src =
        p.q + (size_t)(row0 + (ok ? q0 + r : 0)) * p.ldq + w.head * D + c * 8;
    cp_async16(sQ + swz<D>(r, c), src, ok);
  }
  cp_async_commit();

  const int kv_end = min(q0 + kBM, n);  // keys needed by this tile (causal)
  const int n_tiles = (kv_end + kBN - 1) / kBN;

  auto load_kv = [&](int tile, int buf) {
    const int k0 = tile * kBN;
    for (int i = tid; i < kBN * CH; i += kWarps * 32) {
      const int r = i / CH, c = i % CH;
      const int t = k0 + r;
      const bool ok = t < kv_end;
      const int page = ok ? pt[t / kPage] : 0;
      const size_t off = (((size_t)page * p.n_kv_heads + g) * kPage + (t % kPage)) * D + c * 8;
      cp_async16(sK + buf * kBN * D * 2 + swz<D>(r, c), p.kpages + (ok ? off : 0), ok);
      cp_async16(sV + buf * kBN * D * 2 + swz<D>(r, c), p.vpages + (ok ? off : 0), ok);
    }
    cp_async_commit();
  };

  load_kv(0, 0);
  cp_async_wait<1>();
  __syncthreads();

  // Q fragments for this warp's 16 rows.
  uint32_t qf[D / 16][4];
  {
    const int r = warp * 16 + (lane & 15);
#pragma unroll
    for (int kk = 0; kk < D / 16; ++kk) {
      const int c = kk * 2 + (lane >> 4);
      ldsm_x4(smem_u32(sQ) + swz<D>(r, c), qf[kk][0], qf[kk][1], qf[kk][2], qf[kk][3]);
    }
  }

  float o[D / 8][4];
#pragma unroll
  for (int j = 0; j < D / 8; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;
  float m_i[2] = {-FLT_MAX, -FLT_MAX}, l_i[2] = {0.f, 0.f};
  const float sl2 = 1.4426950408889634f * rsqrtf(static_cast<float>(D));
  const int row_a = q0 + warp * 16 + (lane >> 2);  // rows of c0/c1 and c2/c3 (+8)

  for (int tile = 0; tile < n_tiles; ++tile) {
    const int buf = tile & 1;
    if (tile + 1 < n_tiles) {
      load_kv(tile + 1, buf ^ 1);
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    const int k0 = tile * kBN;
    const uint32_t kbase = smem_u32(sK + buf * kBN * D * 2);
    const uint32_t vbase = smem_u32(sV + buf * kBN * D * 2);

    // S = Q K^T for this warp's 16 rows x 64 keys
    float s[kBN / 8][4];
#pragma unroll
    for (int j = 0; j < kBN / 8; ++j) s[j][0] = s[j][1] = s[j][2] = s[j][3] = 0.f;
#pragma unroll
    for (int kk = 0; kk < D / 16; ++kk) {
#pragma unroll
      for (int nb = 0; nb < kBN / 16; ++nb) {
        const int r = nb * 16 + (lane & 7) + ((lane >> 4) << 3);
        const int c = kk * 2 + ((lane >> 3) & 1);
        uint32_t b0, b1, b2, b3;
        ldsm_x4(kbase + swz<D>(r, c), b0, b1, b2, b3);
        mma16816(s[2 * nb], qf[kk], b0, b1);
        mma16816(s[2 * nb + 1], qf[kk], b2, b3);
      }
    }
    // mask (causal and prefix end) and online softmax
    const bool need_mask = (k0 + kBN - 1 > q0 + warp * 16) || (k0 + kBN > kv_end);
    float mx[2] = {m_i[0], m_i[1]};
#pragma unroll
    for (int j = 0; j < kBN / 8; ++j) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        float v = s[j][e] * sl2;
        if (need_mask) {
          const int col = k0 + j * 8 + 2 * (lane & 3) + (e & 1);
          const int row = row_a + ((e >> 1) << 3);
          if (col > row || col >= kv_end) v = -FLT_MAX;
        }
        s[j][e] = v;
        mx[e >> 1] = fmaxf(mx[e >> 1], v);
      }
    }
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      mx[h] = fmaxf(mx[h], __shfl_xor_sync(0xffffffffu, mx[h], 1));
      mx[h] = fmaxf(mx[h], __shfl_xor_sync(0xffffffffu, mx[h], 2));
    }
    float alpha[2], rs[2] = {0.f, 0.f};
#pragma unroll
    for (int h = 0; h < 2; ++h) alpha[h] = exp2f(m_i[h] - mx[h]);
    uint32_t pf[kBN / 16][4];
#pragma unroll
    for (int j = 0; j < kBN / 8; ++j) {
      const float p0 = s[j][0] <= -FLT_MAX ? 0.f : exp2f(s[j][0] - mx[0]);
      const float p1 = s[j][1] <= -FLT_MAX ? 0.f : exp2f(s[j][1] - mx[0]);
      const float p2 = s[j][2] <= -FLT_MAX ? 0.f : exp2f(s[j][2] - mx[1]);
      const float p3 = s[j][3] <= -FLT_MAX ? 0.f : exp2f(s[j][3] - mx[1]);
      rs[0] += p0 + p1;
      rs[1] += p2 + p3;
      pf[j >> 1][(j & 1) * 2 + 0] = pack_bf16(p0, p1);
      pf[j >> 1][(j & 1) * 2 + 1] = pack_bf16(p2, p3);
    }
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      l_i[h] = l_i[h] * alpha[h] + rs[h];
      m_i[h] = mx[h];
    }
#pragma unroll
    for (int j = 0; j < D / 8; ++j) {
      o[j][0] *= alpha[0];
      o[j][1] *= alpha[0];
      o[j][2] *= alpha[1];
      o[j][3] *= alpha[1];
    }
    // O += P V
#pragma unroll
    for (int kk = 0; kk < kBN / 16; ++kk) {
      // A fragment of P: [row g | g+8] x keys [16kk, 16kk+16)
      uint32_t a[4] = {pf[kk][0], pf[kk][1], pf[kk][2], pf[kk][3]};
#pragma unroll
      for (int nb = 0; nb < D / 16; ++nb) {
        const int r = kk * 16 + (lane & 15);
        const int c = nb * 2 + (lane >> 4);
        uint32_t b0, b1, b2, b3;
        ldsm_x4_t(vbase + swz<D>(r, c), b0, b1, b2, b3);
        mma16816(o[2 * nb], a, b0, b1);
        mma16816(o[2 * nb + 1], a, b2, b3);
      }
    }
    __syncthreads();
  }

  // finalize: full row sums across the quad, normalise, store bf16
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    l_i[h] += __shfl_xor_sync(0xffffffffu, l_i[h], 1);
    l_i[h] += __shfl_xor_sync(0xffffffffu, l_i[h], 2);
  }
  const float inv0 = l_i[0] > 0.f ? 1.f / l_i[0] : 0.f;
  const float inv1 = l_i[1] > 0.f ? 1.f / l_i[1] : 0.f;
#pragma unroll
  for (int j = 0; j < D / 8; ++j) {
    const int col = w.head * D + j * 8 + 2 * (lane & 3);
    if (row_a < n)
      *reinterpret_cast<uint32_t*>(p.out + (size_t)(row0 + row_a) * p.ldo + col) =
          pack_bf16(o[j][0] * inv0, o[j][1] * inv0);
    if (row_a + 8 < n)
      *reinterpret_cast<uint32_t*>(p.out + (size_t)(row0 + row_a + 8) * p.ldo + col) =
          pack_bf16(o[j][2] * inv1, o[j][3] * inv1);
  }
}

// ---------------------------------------------------------------- decode attention
// One decode row per request: q [Hq*d] (fp32, rotated) attends to the request's
// cached keys at positions < pos (from the pages) plus its own fresh k/v at pos.
// A block takes one kv head and one chunk of 256 positions and serves every query
// head of that kv group, so each K/V row is read once per chunk:
//   1. thread t scores position chunk0 + t against all heads of the group,
//   2. warp h turns head h's scores into exp(s - max) and their sum,
//   3. warp w accumulates positions 32w..32w+31 into per-lane 4-dim slices of O,
//      and the 8 warp partials are summed through shared memory.
// The chunk partials (max, sum, O) are merged by decode_attn_combine.
constexpr int kDecThreads = 256;
constexpr int kDecChunk = 256;
constexpr int kDecMaxGroup = 8;

template <int D>
__global__ void __launch_bounds__(kDecThreads) decode_attn_partial(const DecodeAttnDesc p) {
  constexpr int DPL = D / 32;  // dims per lane in the PV accumulation
  const int r = blockIdx.z;
  const int g = blockIdx.y;
  const int chunk = blockIdx.x;
  const int pos = p.pos[r];
  const int grp = p.n_q_heads / p.n_kv_heads;
  const int32_t* pt = p.page_table[r];
  const int total = pos + 1;
  const int t0 = chunk * kDecChunk;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __shared__ float q_s[kDecMaxGroup][D];
  __shared__ float sc[kDecMaxGroup][kDecChunk];
  __shared__ float stat[kDecMaxGroup][2];
  __shared__ float red[kDecThreads / 32][kDecMaxGroup][D];
  __shared__ int page_s[kDecChunk / kPage];
  if (t0 >= total) return;
  const float scale = rsqrtf(static_cast<float>(D));
  for (int i = threadIdx.x; i < grp * D; i += kDecThreads)
    q_s[i / D][i % D] = p.q[(size_t)r * p.n_q_heads * D + (g * grp + i / D) * D + i % D] * scale;
  if (threadIdx.x < kDecChunk / kPage) {
    const int t = t0 + threadIdx.x * kPage;
    page_s[threadIdx.x] = t < pos ? pt[t / kPage] : 0;
  }
  __syncthreads();
  // 1. scores
  {
    const int t = t0 + threadIdx.x;
    float dot[kDecMaxGroup];
#pragma unroll
    for (int h = 0; h < kDecMaxGroup; ++h) dot[h] = 0.f;
    if (t < total) {
      if (t < pos) {
        const uint4* kr = reinterpret_cast<const uint4*>(
            p.kpages + (((size_t)page_s[threadIdx.x / kPage] * p.n_kv_heads + g) * kPage + t % kPage) * D);
#pragma unroll 4
        for (int i = 0; i < D / 8; ++i) {
          const uint4 u = kr[i];
          const float k8[8] = {bf16_lo(u.x), bf16_hi(u.x), bf16_lo(u.y), bf16_hi(u.y),
                               bf16_lo(u.z), bf16_hi(u.z), bf16_lo(u.w), bf16_hi(u.w)};
#pragma unroll
          for (int h = 0; h < kDecMaxGroup; ++h)
            if (h < grp)
#pragma unroll
              for (int e = 0; e < 8; ++e) dot[h] += q_s[h][8 * i + e] * k8[e];
        }
      } else {
        const float* kr = p.k_self + (size_t)r * p.n_kv_heads * D + g * D;
        for (int i = 0; i < D; ++i) {
          const float kv = kr[i];
#pragma unroll
          for (int h = 0; h < kDecMaxGroup; ++h)
            if (h < grp) dot[h] += q_s[h][i] * kv;
        }
      }
    }
#pragma unroll
    for (int h = 0; h < kDecMaxGroup; ++h)
      if (h < grp) sc[h][threadIdx.x] = t < total ? dot[h] : -FLT_MAX;
  }
  __syncthreads();
  // 2. per-head max, exponentials, sum (warp h)
  if (warp < grp) {
    float m = -FLT_MAX;
    for (int i = lane; i < kDecChunk; i += 32) m = fmaxf(m, sc[warp][i]);
    m = warp_max(m);
    float l = 0.f;
    for (int i = lane; i < kDecChunk; i += 32) {
      const float e = sc[warp][i] == -FLT_MAX ? 0.f : __expf(sc[warp][i] - m);
      sc[warp][i] = e;
      l += e;
    }
    l = warp_sum(l);
    if (lane == 0) {
      stat[warp][0] = m;
      stat[warp][1] = l;
    }
  }
  __syncthreads();
  // 3. O partial: warp w takes positions t0 + 32w .. t0 + 32w + 31
  float acc[kDecMaxGroup][DPL];
#pragma unroll
  for (int h = 0; h < kDecMaxGroup; ++h)
#pragma unroll
    for (int e = 0; e < DPL; ++e) acc[h][e] = 0.f;
  const int kb = warp * 32;
  const int kend = max(0, min(32, total - t0 - kb));
#pragma unroll 8
  for (int k = 0; k < kend; ++k) {
    const int t = t0 + kb + k;
    float v[DPL];
    if (t < pos) {
      const __nv_bfloat16* vr = p.vpages +
          (((size_t)page_s[(kb + k) / kPage] * p.n_kv_heads + g) * kPage + t % kPage) * D + lane * DPL;
      if (DPL == 4) {
        const uint2 u = __ldg(reinterpret_cast<const uint2*>(vr));
        v[0] = bf16_lo(u.x);
        v[1 % DPL] = bf16_hi(u.x);
        v[2 % DPL] = bf16_lo(u.y);
        v[3 % DPL] = bf16_hi(u.y);
      } else {
        const uint32_t u = __ldg(reinterpret_cast<const uint32_t*>(vr));
        v[0] = bf16_lo(u);
        v[1 % DPL] = bf16_hi(u);
      }
    } else {
      const float* vr = p.v_self + (size_t)r * p.n_kv_heads * D + g * D + lane * DPL;
#pragma unroll
      for (int e = 0; e < DPL; ++e) v[e] = vr[e];
    }
#pragma unroll
    for (int h = 0; h < kDecMaxGroup; ++h)
      if (h < grp) {
        const float ph = sc[h][kb + k];
#pragma unroll
        for (int e = 0; e < DPL; ++e) acc[h][e] += ph * v[e];
      }
  }
#pragma unroll
  for (int h = 0; h < kDecMaxGroup; ++h)
    if (h < grp)
#pragma unroll
      for (int e = 0; e < DPL; ++e) red[warp][h][lane * DPL + e] = acc[h][e];
  __syncthreads();
  for (int i = threadIdx.x; i < grp * D; i += kDecThreads) {
    const int h = i / D, d = i % D;
    float o = 0.f;
#pragma unroll
    for (int w = 0; w < kDecThreads / 32; ++w) o += red[w][h][d];
    float* part = p.part + (((size_t)r * p.n_q_heads + g * grp + h) * p.splits + chunk) * (D + 2);
    part[d] = o;
    if (d == 0) {
      part[D] = stat[h][0];
      part[D + 1] = stat[h][1];
    }
  }
}

template <int D>
__global__ void decode_attn_combine(const DecodeAttnDesc p) {
  const int r = blockIdx.y, h = blockIdx.x;
  const int dd = threadIdx.x;
  const int n_chunks = (p.pos[r] + 1 + kDecChunk - 1) / kDecChunk;
  const float* base = p.part + ((size_t)r * p.n_q_heads + h) * p.splits * (D + 2);
  float m = -FLT_MAX;
  for (int s = 0; s < n_chunks; ++s) m = fmaxf(m, base[s * (D + 2) + D]);
  float l = 0.f, acc = 0.f;
  for (int s = 0; s < n_chunks; ++s) {
    const float f = __expf(base[s * (D + 2) + D] - m);
    l += f * base[s * (D + 2) + D + 1];
    if (dd < D) acc += f * base[s * (D + 2) + dd];
  }
  if (dd < D) p.out[(size_t)r * p.n_q_heads * D + h * D + dd] = acc / l;
}

}  // namespace

cudaError_t launch_attention(const AttnDesc& d, int num_sms, cudaStream_t stream) {
  (void)num_sms;
  int items = 0;
  for (int i = 0; i < d.req.n; ++i) items += ((d.req.len[i] + kBM - 1) / kBM) * d.n_q_heads;
  if (items == 0) return cudaSuccess;
  if (d.head_dim == 128) {
    constexpr int smem = (kBM + 4 * kBN) * 128 * 2;
    static bool set = false;
    if (!set) {
      cudaError_t e = cudaFuncSetAttribute(attn_prefill_kernel<128>,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
      if (e != cudaSuccess) return e;
      set = true;
    }
    attn_prefill_kernel<128><<<items, kWarps * 32, smem, stream>>>(d);
  } else if (d.head_dim == 64) {
    constexpr int smem = (kBM + 4 * kBN) * 64 * 2;
    static bool set = false;
    if (!set) {
      cudaError_t e = cudaFuncSetAttribute(attn_prefill_kernel<64>,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
      if (e != cudaSuccess) return e;
      set = true;
    }
    attn_prefill_kernel<64><<<items, kWarps * 32, smem, stream>>>(d);
  } else {
    return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

cudaError_t launch_decode_attention(const DecodeAttnDesc& d, cudaStream_t stream) {
  if (d.n_q_heads / d.n_kv_heads > kDecMaxGroup) return cudaErrorInvalidValue;
  int max_pos = 0;
  for (int r = 0; r < d.rows; ++r) max_pos = max(max_pos, d.pos[r]);
  const int chunks = (max_pos + 1 + kDecChunk - 1) / kDecChunk;
  if (chunks > d.splits) return cudaErrorInvalidValue;
  dim3 g1(chunks, d.n_kv_heads, d.rows), g2(d.n_q_heads, d.rows);
  if (d.head_dim == 128) {
    decode_attn_partial<128><<<g1, kDecThreads, 0, stream>>>(d);
    decode_attn_combine<128><<<g2, 128, 0, stream>>>(d);
  } else if (d.head_dim == 64) {
    decode_attn_partial<64><<<g1, kDecThreads, 0, stream>>>(d);
    decode_attn_combine<64><<<g2, 64, 0, stream>>>(d);
  } else {
    return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

}  // namespace crf
