// Causal grouped-query prefill attention over the paged KV cache on mma.sync
// (the alternative to the tcgen05 kernel, selected with CRF_ATTENTION=mma): the
// self-attention of a recomputed layer (Section 4.2, Eq. 1, Eq. S3).
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
      const int page = ok ? checked_page(pt[t / kPage], p.req.num_pages, p.status) : 0;
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

}  // namespace

cudaError_t launch_attention(const AttnDesc& d, int num_sms, cudaStream_t stream) {
  (void)num_sms;
  int items = 0;
  for (int i = 0; i < d.req.n; ++i) items += ((d.req.len[i] + kBM - 1) / kBM) * d.n_q_heads;
  if (items == 0) return cudaSuccess;
  if (d.head_dim == 128) {
    constexpr int smem = (kBM + 4 * kBN) * 128 * 2;
    static PerDevice once;
    int dev = 0;
    if (once.pending(&dev)) {
      cudaError_t e = cudaFuncSetAttribute(attn_prefill_kernel<128>,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
      if (e != cudaSuccess) return e;
      once.done(dev);
    }
    attn_prefill_kernel<128><<<items, kWarps * 32, smem, stream>>>(d);
  } else if (d.head_dim == 64) {
    constexpr int smem = (kBM + 4 * kBN) * 64 * 2;
    static PerDevice once;
    int dev = 0;
    if (once.pending(&dev)) {
      cudaError_t e = cudaFuncSetAttribute(attn_prefill_kernel<64>,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
      if (e != cudaSuccess) return e;
      once.done(dev);
    }
    attn_prefill_kernel<64><<<items, kWarps * 32, smem, stream>>>(d);
  } else {
    return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}


}  // namespace crf
