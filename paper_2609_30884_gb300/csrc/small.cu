// Memory-bound kernels: RMSNorm, embedding gather, RoPE angle table, the
// small-M decode path (GEMV with fused LoRA, RoPE on rows, SwiGLU), the LM
// head and the first-step KL reduction (Section S2.1).
#include "common.cuh"
#include "kernels.h"

#include <cfloat>
#include <cmath>
#include <cstdlib>
#include <cstring>

namespace crf {

namespace {

// ------------------------------------------------------------------ RoPE table
// table[p][i] = (cos, sin)(p * theta^(-2i/d)): the angle in turns, p * theta^(-2i/d) / (2 pi),
// is formed in fp64 (per-frequency factors computed on the host in fp64), reduced to [0, 1)
// and evaluated with fp32 sincospi.
struct RopeFreqs {
  double turns_per_pos[64];
};

__global__ void rope_table_kernel(float2* table, int n_pos, int half, const __grid_constant__ RopeFreqs f) {
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= n_pos * half) return;
  const int p = idx / half, i = idx % half;
  double turns = static_cast<double>(p) * f.turns_per_pos[i];
  turns -= floor(turns);
  float s, c;
  sincospif(static_cast<float>(2.0 * turns), &s, &c);
  table[idx] = make_float2(c, s);
}

// ------------------------------------------------------------------ RMSNorm (+ BX rows)
// One 16-byte chunk (8 columns) of a BX row per thread: the module's B row (rank values, zero
// padded to 16) at columns col_off .. col_off + 15 and again at col_off + 16 .. col_off + 31.
__device__ __forceinline__ void bext_chunk(const BextDesc& d, long idx) {
  int m = 0;
  long base = 0;
  while (m < d.n && idx >= base + static_cast<long>(d.rows[m]) * (kBxCols / 8)) {
    base += static_cast<long>(d.rows[m]) * (kBxCols / 8);
    ++m;
  }
  if (m >= d.n) return;
  const long k = idx - base;
  const int r = static_cast<int>(k / (kBxCols / 8));
  const int c0 = static_cast<int>(k % (kBxCols / 8)) * 8;
  const __nv_bfloat16* B = d.B[m];
  uint32_t w[4];
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    float v[2];
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int c = c0 + 2 * j + h - d.col_off[m];
      const int q = c & 15;
      v[h] = (B && c >= 0 && c < 32 && q < d.rank) ? __bfloat162float(B[(size_t)r * d.rank + q]) : 0.f;
    }
    w[j] = pack_bf16(v[0], v[1]);
  }
  *reinterpret_cast<uint4*>(d.out[m] + (size_t)r * kBxCols + c0) = make_uint4(w[0], w[1], w[2], w[3]);
}

// Blocks [0, norm_blocks): one warp per row, y = x * rsqrt(mean(x^2) + eps) * g, fp32 math, bf16
// out. The blocks after them: the BX rows of `bx`, one chunk per thread.
__global__ void rmsnorm_kernel(const __nv_bfloat16* __restrict__ x,
                               const __nv_bfloat16* __restrict__ g, __nv_bfloat16* __restrict__ y,
                               int rows, int hidden, float eps, const __grid_constant__ BextDesc bx,
                               int norm_blocks) {
  if (static_cast<int>(blockIdx.x) >= norm_blocks) {
    bext_chunk(bx, static_cast<long>(blockIdx.x - norm_blocks) * blockDim.x + threadIdx.x);
    return;
  }
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (warp >= rows) return;
  const uint4* xr = reinterpret_cast<const uint4*>(x + (size_t)warp * hidden);
  const uint4* gr = reinterpret_cast<const uint4*>(g);
  uint4* yr = reinterpret_cast<uint4*>(y + (size_t)warp * hidden);
  const int nv = hidden / 8;
  float ss = 0.f;
  for (int i = lane; i < nv; i += 32) {
    const uint4 u = xr[i];
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float a = bf16_lo(w[j]), b = bf16_hi(w[j]);
      ss += a * a + b * b;
    }
  }
  ss = warp_sum(ss);
  const float inv = rsqrtf(ss / hidden + eps);
  for (int i = lane; i < nv; i += 32) {
    const uint4 u = xr[i];
    const uint4 gv = gr[i];
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
    const uint32_t gw[4] = {gv.x, gv.y, gv.z, gv.w};
    uint32_t o[4];
#pragma unroll
    for (int j = 0; j < 4; ++j)
      o[j] = pack_bf16(bf16_lo(w[j]) * inv * bf16_lo(gw[j]), bf16_hi(w[j]) * inv * bf16_hi(gw[j]));
    yr[i] = make_uint4(o[0], o[1], o[2], o[3]);
  }
}

__global__ void rmsnorm_f32_kernel(const float* __restrict__ x, const __nv_bfloat16* __restrict__ g,
                                   float* __restrict__ y, int rows, int hidden, float eps) {
  const int row = blockIdx.x;
  __shared__ float red[32];
  float ss = 0.f;
  for (int i = threadIdx.x; i < hidden; i += blockDim.x) {
    const float v = x[(size_t)row * hidden + i];
    ss += v * v;
  }
  ss = warp_sum(ss);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
  __syncthreads();
  if (threadIdx.x < 32) {
    float v = threadIdx.x < (blockDim.x >> 5) ? red[threadIdx.x] : 0.f;
    v = warp_sum(v);
    if (threadIdx.x == 0) red[0] = v;
  }
  __syncthreads();
  const float inv = rsqrtf(red[0] / hidden + eps);
  for (int i = threadIdx.x; i < hidden; i += blockDim.x)
    y[(size_t)row * hidden + i] = x[(size_t)row * hidden + i] * inv * __bfloat162float(g[i]);
}

// ------------------------------------------------------------------ embedding
__global__ void embed_kernel(const __nv_bfloat16* __restrict__ e, const int32_t* __restrict__ tok,
                             __nv_bfloat16* __restrict__ out, int n, int hidden, int vocab,
                             int* status) {
  const int nv = hidden / 8;
  const size_t idx = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= (size_t)n * nv) return;
  const int t = static_cast<int>(idx / nv), c = static_cast<int>(idx % nv);
  // Only the row's first chunk reports a bad id, so the status word sees one atomic per row.
  const int id = checked_token(tok[t], vocab, c == 0 ? status : nullptr);
  reinterpret_cast<uint4*>(out + (size_t)t * hidden)[c] =
      reinterpret_cast<const uint4*>(e + (size_t)id * hidden)[c];
}

// ------------------------------------------------------------------ decode-path GEMV
// A block of 8 warps takes 8/KS groups of OPW consecutive outputs of one segment; the KS
// warps of a group split the input dimension, each lane streaming 16-byte pieces of the
// OPW weight rows (x read through the cache and reused across the OPW rows). Partials are
// summed in shared memory in a fixed order (deterministic), then scaled, and bias and residual
// are added.
constexpr int kGemvWarps = 8;
constexpr int kGemvMaxRows = 8;

struct GemvLaunch {
  GemvDesc d;
  int opw, ks;
  int block0[kGemvMaxSeg + 1];  // first block of each segment
};

template <int OPW, int NR>
__global__ void __launch_bounds__(kGemvWarps * 32) gemv_kernel(const __grid_constant__ GemvLaunch L) {
  __shared__ float red[kGemvWarps][OPW][NR];
  const GemvDesc& d = L.d;
  const int ks = L.ks;
  int s = 0;
  while (s < d.nseg - 1 && static_cast<int>(blockIdx.x) >= L.block0[s + 1]) ++s;
  const GemvSeg& sg = d.seg[s];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int gl = warp / ks, kp = warp % ks;
  const int groups_per_block = kGemvWarps / ks;
  const int gb = (static_cast<int>(blockIdx.x) - L.block0[s]) * groups_per_block;
  if (d.prefetch) {  // the block's weight rows are contiguous
    const int jb0 = gb * OPW, jb1 = min(sg.out_dim, jb0 + groups_per_block * OPW);
    if (jb0 < jb1) prefetch_l2_range(sg.W + (size_t)jb0 * d.in_dim, (size_t)(jb1 - jb0) * d.in_dim * 2);
  }
  griddep_begin();  // x, xa and the residual come from the kernels before
  if (call_aborted(d.abort)) return;
  const int g = gb + gl;
  const int j0 = g * OPW;
  const int n8 = d.in_dim / 8;
  const int per = (n8 + ks - 1) / ks;
  const int p0 = kp * per, p1 = min(n8, p0 + per);
  float acc[OPW][NR];
#pragma unroll
  for (int o = 0; o < OPW; ++o)
#pragma unroll
    for (int r = 0; r < NR; ++r) acc[o][r] = 0.f;
  if (j0 < sg.out_dim) {
    const uint4* wrow[OPW];
#pragma unroll
    for (int o = 0; o < OPW; ++o)
      wrow[o] = reinterpret_cast<const uint4*>(sg.W + (size_t)min(j0 + o, sg.out_dim - 1) * d.in_dim);
#pragma unroll 2
    for (int c = p0 + lane; c < p1; c += 32) {
      uint4 u[OPW];
#pragma unroll
      for (int o = 0; o < OPW; ++o) u[o] = __ldg(wrow[o] + c);
#pragma unroll
      for (int r = 0; r < NR; ++r) {
        if (r < d.rows) {
          const float4* xr = reinterpret_cast<const float4*>(d.x + (size_t)r * d.in_dim) + 2 * c;
          const float4 a = __ldg(xr), b = __ldg(xr + 1);
#pragma unroll
          for (int o = 0; o < OPW; ++o)
            acc[o][r] += bf16_lo(u[o].x) * a.x + bf16_hi(u[o].x) * a.y + bf16_lo(u[o].y) * a.z +
                         bf16_hi(u[o].y) * a.w + bf16_lo(u[o].z) * b.x + bf16_hi(u[o].z) * b.y +
                         bf16_lo(u[o].w) * b.z + bf16_hi(u[o].w) * b.w;
        }
      }
    }
  }
#pragma unroll
  for (int o = 0; o < OPW; ++o)
#pragma unroll
    for (int r = 0; r < NR; ++r) {
      const float v = warp_sum(acc[o][r]);
      if (lane == 0) red[warp][o][r] = v;
    }
  __syncthreads();
  if (kp != 0 || lane >= OPW * NR) return;
  const int o = lane / NR, r = lane % NR;
  const int j = j0 + o;
  if (j >= sg.out_dim || r >= d.rows) return;
  float v = 0.f;
  for (int q = 0; q < ks; ++q) v += red[gl * ks + q][o][r];
  v *= sg.scale;
  if (sg.bias) v += __bfloat162float(sg.bias[j]);
  if (sg.resid) v += sg.resid[(size_t)r * sg.out_dim + j];
  sg.y[(size_t)r * sg.out_dim + j] = v;
}

// sum_k B[j, k] xa[k] for one output j of a rank-r up product (B row: r bf16, 8-byte aligned)
__device__ __forceinline__ float up_dot(const __nv_bfloat16* __restrict__ B, int j, const float* __restrict__ xa,
                                        int rank) {
  const __nv_bfloat16* br = B + (size_t)j * rank;
  float s = 0.f;
  if (rank == 16) {
    const uint4 u0 = __ldg(reinterpret_cast<const uint4*>(br)), u1 = __ldg(reinterpret_cast<const uint4*>(br) + 1);
    const uint32_t w[8] = {u0.x, u0.y, u0.z, u0.w, u1.x, u1.y, u1.z, u1.w};
#pragma unroll
    for (int i = 0; i < 8; ++i) s += bf16_lo(w[i]) * xa[2 * i] + bf16_hi(w[i]) * xa[2 * i + 1];
  } else if (rank == 8) {
    const uint4 u0 = __ldg(reinterpret_cast<const uint4*>(br));
    const uint32_t w[4] = {u0.x, u0.y, u0.z, u0.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) s += bf16_lo(w[i]) * xa[2 * i] + bf16_hi(w[i]) * xa[2 * i + 1];
  } else {
    for (int i = 0; i < rank; ++i) s += __bfloat162float(br[i]) * xa[i];
  }
  return s;
}

// x[r] += up(r) when r < up_rows, then xn[r] = rmsnorm(x[r]) * g, with each row cut into slices of
// kNormSlice elements, one block per (row, slice): the block adds its slice's up products (the
// rank-r B rows of the slice) and writes the slice's sum of squares to part[r][slice]; the last
// block of the row to finish (a counter per row, reset by it) sums the partials in slice order
// and normalises the whole row. Deterministic: the same partials, summed in the same order.
constexpr int kNormSlice = 256;
__global__ void __launch_bounds__(kNormSlice) norm_up_rows_kernel(float* __restrict__ x, int dim, RowUp up,
                                                                  int up_rows, int rank,
                                                                  const __nv_bfloat16* __restrict__ g, float eps,
                                                                  float* __restrict__ xn, float* __restrict__ part,
                                                                  int* __restrict__ counter, int slices) {
  __shared__ float red[kNormSlice / 32];
  __shared__ float xa_s[kRankPad];
  __shared__ int last_s;
  const int r = blockIdx.x / slices, sl = blockIdx.x % slices;
  const int j = sl * kNormSlice + threadIdx.x;
  const bool add = up.B != nullptr && r < up_rows;
  if (add && threadIdx.x == 0)
    prefetch_l2_range(up.B + (size_t)sl * kNormSlice * rank, (size_t)kNormSlice * rank * 2);
  griddep_begin();  // x and xa come from the kernels before
  float* xr = x + (size_t)r * dim;
  if (add && threadIdx.x < rank) xa_s[threadIdx.x] = up.xa[(size_t)r * rank + threadIdx.x];
  __syncthreads();
  float ss = 0.f;
  if (j < dim) {
    float v = xr[j];
    if (add) {
      v += up_dot(up.B, j, xa_s, rank);
      xr[j] = v;
    }
    ss = v * v;
  }
  ss = warp_sum(ss);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
  __syncthreads();
  if (threadIdx.x == 0) {
    float t = 0.f;
#pragma unroll
    for (int w = 0; w < kNormSlice / 32; ++w) t += red[w];
    part[(size_t)r * slices + sl] = t;
    __threadfence();  // the slice's x and its partial before the count
    last_s = atomicAdd(counter + r, 1) == slices - 1;
  }
  __syncthreads();
  if (!last_s) return;
  __threadfence();  // every slice's x and partial are visible to this block
  if (threadIdx.x == 0) {
    float t = 0.f;
    for (int q = 0; q < slices; ++q) t += __ldcg(part + (size_t)r * slices + q);
    red[0] = rsqrtf(t / dim + eps);
    counter[r] = 0;  // ready for the next launch
  }
  __syncthreads();
  const float inv = red[0];
  // eight elements per thread in flight: the row's other slices come from L2
  for (int i0 = threadIdx.x; i0 < dim; i0 += 8 * kNormSlice) {
    float xv[8], gv[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const int i = i0 + u * kNormSlice;
      xv[u] = i < dim ? __ldcg(xr + i) : 0.f;
      gv[u] = i < dim ? __bfloat162float(g[i]) : 0.f;
    }
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const int i = i0 + u * kNormSlice;
      if (i < dim) xn[(size_t)r * dim + i] = xv[u] * inv * gv[u];
    }
  }
}

// x[r, j] += up(r, j), one thread per element.
__global__ void rows_up_kernel(float* __restrict__ x, int dim, int rows, RowUp up, int rank) {
  griddep_begin();  // x and xa come from the kernels before
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= rows * dim) return;
  const int r = idx / dim, j = idx % dim;
  x[idx] += up_dot(up.B, j, up.xa + (size_t)r * rank, rank);
}

struct RowUp3 {
  RowUp m[3];  // q, k, v
};

// Threads [0, rows * (hq + hkv) * d/2): one rotation pair (i, i + d/2) of a q or k head: the up
// products added, then rotate-half RoPE at the row's position. The rest: one v element each,
// the up product added.
__global__ void rope_up_rows_kernel(float* q, int hq, float* k, int hkv, float* v, int rows, int d,
                                    const __grid_constant__ RowUp3 up, int rank,
                                    const float2* __restrict__ table, const RowPositions pos, int by_row) {
  griddep_begin();  // q, k, v and xa come from the GEMV before
  const int half = d / 2;
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  const int heads = hq + hkv;
  const int n_pairs = rows * heads * half;
  if (idx >= n_pairs) {
    const int e = idx - n_pairs;
    if (e >= rows * hkv * d) return;
    if (up.m[2].B) {
      const int r = e / (hkv * d), j = e % (hkv * d);
      v[e] += up_dot(up.m[2].B, j, up.m[2].xa + (size_t)r * rank, rank);
    }
    return;
  }
  const int i = idx % half;
  const int h = (idx / half) % heads;
  const int r = idx / (half * heads);
  const bool is_q = h < hq;
  const int hh = is_q ? h : h - hq;
  const RowUp& u = up.m[is_q ? 0 : 1];
  float* base = is_q ? q + ((size_t)r * hq + hh) * d : k + ((size_t)r * hkv + hh) * d;
  float x1 = base[i], x2 = base[i + half];
  if (u.B) {
    const float* xa = u.xa + (size_t)r * rank;
    x1 += up_dot(u.B, hh * d + i, xa, rank);
    x2 += up_dot(u.B, hh * d + i + half, xa, rank);
  }
  const float2 cs = table[(size_t)(by_row ? r : pos.pos[r]) * half + i];
  base[i] = x1 * cs.x - x2 * cs.y;
  base[i + half] = x2 * cs.x + x1 * cs.y;
}

// m[r, j] = silu(g + up_g) * (u + up_u) over [rows, f] (gate and up in separate buffers)
__global__ void swiglu_up_rows_kernel(const float* g, const float* u, float* m, int rows, int f, RowUp up_g,
                                      RowUp up_u, int rank) {
  griddep_begin();  // gate, up and xa come from the GEMV before
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= rows * f) return;
  const int r = idx / f, j = idx % f;
  float gv = g[idx], uv = u[idx];
  if (up_g.B) gv += up_dot(up_g.B, j, up_g.xa + (size_t)r * rank, rank);
  if (up_u.B) uv += up_dot(up_u.B, j, up_u.xa + (size_t)r * rank, rank);
  m[idx] = gv / (1.f + __expf(-gv)) * uv;
}

__global__ void f32_to_bf16_kernel(const float* x, __nv_bfloat16* y, int n, const int* abort) {
  if (call_aborted(abort)) return;
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) y[i] = __float2bfloat16_rn(x[i]);
}

__global__ void copy_bf16_kernel(__nv_bfloat16* __restrict__ dst, const __nv_bfloat16* __restrict__ src,
                                 size_t n, const int* abort) {
  if (call_aborted(abort)) return;
  for (size_t i = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x; i < n;
       i += static_cast<size_t>(gridDim.x) * blockDim.x)
    dst[i] = src[i];
}

// One thread per page id: outside [0, num_pages), or already in the open-addressing table
// (linear probing, at most mask + 1 probes), rejects the call.
__global__ void validate_pages_kernel(const PageCheck pc, int num_pages, int* table, uint32_t mask,
                                      int* abort, int* status) {
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= pc.first[pc.n]) return;
  int i = 0;
  while (i + 1 < pc.n && idx >= pc.first[i + 1]) ++i;
  const int id = pc.pt[i][idx - pc.first[i]];
  bool bad = id < 0 || id >= num_pages;
  if (!bad) {
    uint32_t h = (static_cast<uint32_t>(id) * 0x9E3779B1u) & mask;
    for (uint32_t probe = 0; probe <= mask; ++probe) {
      const int prev = atomicCAS(table + h, -1, id);
      if (prev == -1) break;
      if (prev == id) {
        bad = true;
        break;
      }
      h = (h + 1) & mask;
    }
  }
  if (bad) {
    atomicExch(abort, 1);
    atomicOr(status, kStatusPages);
  }
}
__global__ void bf16_to_f32_kernel(const __nv_bfloat16* x, float* y, int n) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) y[i] = __bfloat162float(x[i]);
}

// ------------------------------------------------------------------ KL
// Per (row, split): online (max, sum e^(z* - m), sum e^(z* - m)(z* - z)) for the
// reference and (max, sum e^(z - m)) for the current logits.
constexpr int kKlThreads = 256;

__global__ void __launch_bounds__(kKlThreads) kl_partial_kernel(const float* __restrict__ zr,
                                                                const float* __restrict__ zc,
                                                                int vocab, int splits,
                                                                float* __restrict__ part) {
  const int row = blockIdx.y, sp = blockIdx.x;
  const int per = (vocab + splits - 1) / splits;
  const int v0 = sp * per, v1 = min(vocab, v0 + per);
  const float* a = zr + (size_t)row * vocab;
  const float* b = zc + (size_t)row * vocab;
  float mr = -FLT_MAX, sr = 0.f, dr = 0.f, mc = -FLT_MAX, sc = 0.f;
  for (int i = v0 + threadIdx.x; i < v1; i += kKlThreads) {
    const float x = a[i], y = b[i];
    if (x > mr) {
      const float f = __expf(mr - x);
      sr *= f;
      dr *= f;
      mr = x;
    }
    const float e = __expf(x - mr);
    sr += e;
    dr += e * (x - y);
    if (y > mc) {
      sc *= __expf(mc - y);
      mc = y;
    }
    sc += __expf(y - mc);
  }
  // block combine
  __shared__ float s_mr[kKlThreads], s_sr[kKlThreads], s_dr[kKlThreads], s_mc[kKlThreads],
      s_sc[kKlThreads];
  s_mr[threadIdx.x] = mr;
  s_sr[threadIdx.x] = sr;
  s_dr[threadIdx.x] = dr;
  s_mc[threadIdx.x] = mc;
  s_sc[threadIdx.x] = sc;
  __syncthreads();
  for (int off = kKlThreads / 2; off > 0; off >>= 1) {
    if (threadIdx.x < off) {
      const int o = threadIdx.x + off;
      const float M = fmaxf(s_mr[threadIdx.x], s_mr[o]);
      const float f1 = s_mr[threadIdx.x] == -FLT_MAX ? 0.f : __expf(s_mr[threadIdx.x] - M);
      const float f2 = s_mr[o] == -FLT_MAX ? 0.f : __expf(s_mr[o] - M);
      s_sr[threadIdx.x] = s_sr[threadIdx.x] * f1 + s_sr[o] * f2;
      s_dr[threadIdx.x] = s_dr[threadIdx.x] * f1 + s_dr[o] * f2;
      s_mr[threadIdx.x] = M;
      const float Mc = fmaxf(s_mc[threadIdx.x], s_mc[o]);
      const float g1 = s_mc[threadIdx.x] == -FLT_MAX ? 0.f : __expf(s_mc[threadIdx.x] - Mc);
      const float g2 = s_mc[o] == -FLT_MAX ? 0.f : __expf(s_mc[o] - Mc);
      s_sc[threadIdx.x] = s_sc[threadIdx.x] * g1 + s_sc[o] * g2;
      s_mc[threadIdx.x] = Mc;
    }
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    float* p = part + ((size_t)row * splits + sp) * 5;
    p[0] = s_mr[0];
    p[1] = s_sr[0];
    p[2] = s_dr[0];
    p[3] = s_mc[0];
    p[4] = s_sc[0];
  }
}

// KL = D/S* + (M + log S) - (M* + log S*), combining the splits of one row (warp per row).
__global__ void kl_final_kernel(const float* part, int splits, float* out, int rows) {
  const int row = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (row >= rows) return;
  const float* p = part + (size_t)row * splits * 5;
  float Mr = -FLT_MAX, Mc = -FLT_MAX;
  for (int s = lane; s < splits; s += 32) {
    Mr = fmaxf(Mr, p[s * 5 + 0]);
    Mc = fmaxf(Mc, p[s * 5 + 3]);
  }
  Mr = warp_max(Mr);
  Mc = warp_max(Mc);
  float Sr = 0.f, Dr = 0.f, Sc = 0.f;
  for (int s = lane; s < splits; s += 32) {
    const float fr = p[s * 5 + 0] == -FLT_MAX ? 0.f : __expf(p[s * 5 + 0] - Mr);
    Sr += fr * p[s * 5 + 1];
    Dr += fr * p[s * 5 + 2];
    Sc += (p[s * 5 + 3] == -FLT_MAX ? 0.f : __expf(p[s * 5 + 3] - Mc)) * p[s * 5 + 4];
  }
  Sr = warp_sum(Sr);
  Dr = warp_sum(Dr);
  Sc = warp_sum(Sc);
  if (lane == 0) out[row] = Dr / Sr + (Mc + logf(Sc)) - (Mr + logf(Sr));
}

inline int cdiv(long a, long b) { return static_cast<int>((a + b - 1) / b); }

}  // namespace

cudaError_t launch_rope_table(float2* table, int n_pos, int head_dim, double theta,
                              cudaStream_t stream) {
  const int half = head_dim / 2;
  const int n = n_pos * half;
  if (n == 0) return cudaSuccess;
  if (half > 64) return cudaErrorInvalidValue;
  RopeFreqs f;
  for (int i = 0; i < half; ++i)
    f.turns_per_pos[i] = std::pow(theta, -2.0 * i / head_dim) / (2.0 * 3.14159265358979323846);
  rope_table_kernel<<<cdiv(n, 256), 256, 0, stream>>>(table, n_pos, half, f);
  return cudaGetLastError();
}

cudaError_t launch_rmsnorm(const __nv_bfloat16* x, const __nv_bfloat16* g, __nv_bfloat16* y,
                           int rows, int hidden, float eps, cudaStream_t stream, const BextDesc* bx) {
  BextDesc d{};
  long chunks = 0;
  if (bx) {
    d = *bx;
    if (d.n < 0 || d.n > 4 || d.rank < 1 || d.rank > kRankPad) return cudaErrorInvalidValue;
    for (int m = 0; m < d.n; ++m) chunks += static_cast<long>(d.rows[m]) * (kBxCols / 8);
  }
  const int norm_blocks = cdiv(rows, 8);
  const int blocks = norm_blocks + static_cast<int>(cdiv(chunks, 256));
  if (blocks == 0) return cudaSuccess;
  rmsnorm_kernel<<<blocks, 256, 0, stream>>>(x, g, y, rows, hidden, eps, d, norm_blocks);
  return cudaGetLastError();
}

cudaError_t launch_embed(const __nv_bfloat16* embed, const int32_t* tokens, __nv_bfloat16* out,
                         int n, int hidden, int vocab, int* status, cudaStream_t stream) {
  const long total = (long)n * (hidden / 8);
  if (total == 0) return cudaSuccess;
  embed_kernel<<<cdiv(total, 256), 256, 0, stream>>>(embed, tokens, out, n, hidden, vocab, status);
  return cudaGetLastError();
}

template <int OPW>
cudaError_t gemv_dispatch(const GemvLaunch& L, int blocks, cudaStream_t stream) {
  const dim3 grid(blocks), block(kGemvWarps * 32);
  if (L.d.rows == 1) return launch_kernel(gemv_kernel<OPW, 1>, grid, block, 0, stream, L);
  if (L.d.rows == 2) return launch_kernel(gemv_kernel<OPW, 2>, grid, block, 0, stream, L);
  if (L.d.rows <= 4) return launch_kernel(gemv_kernel<OPW, 4>, grid, block, 0, stream, L);
  return launch_kernel(gemv_kernel<OPW, 8>, grid, block, 0, stream, L);
}

namespace {
thread_local bool t_pdl = false;
}  // namespace

PdlScope::PdlScope() : prev_(t_pdl) { t_pdl = true; }
PdlScope::~PdlScope() { t_pdl = prev_; }
bool pdl_active() { return t_pdl; }

bool gemv_use_tensor(int total_rows, int in_dim) {
  // the MMA path pays for its 16-row tiles and x splitting from three rows on (measured: 1-2 rows
  // run faster on the CUDA-core kernel, 3 rows 20% and 8 rows 45% faster on the tensor cores)
  return total_rows >= 3 && in_dim % 16 == 0;
}

cudaError_t launch_gemv(const GemvDesc& d, int num_sms, cudaStream_t stream, int total_rows) {
  if (gemv_use_tensor(total_rows > 0 ? total_rows : d.rows, d.in_dim)) return launch_gemv_tc(d, num_sms, stream);
  if (d.rows < 1 || d.rows > kGemvMaxRows || d.nseg < 1 || d.nseg > kGemvMaxSeg || d.in_dim % 8 != 0)
    return cudaErrorInvalidValue;
  GemvLaunch L;
  L.d = d;
  L.d.prefetch = pdl_active() ? 1 : 0;
  int total_out = 0;
  for (int s = 0; s < d.nseg; ++s) total_out += d.seg[s].out_dim;
  if (total_out == 0) return cudaSuccess;
  // outputs per warp: reuse x across weight rows when there are many outputs
  L.opw = total_out >= 65536 ? 4 : total_out >= 16384 ? 2 : 1;
  // split the input dimension until the warps cover the GPU (pieces of >= 256 inputs)
  const int want_warps = 32 * num_sms;
  L.ks = 1;
  while (L.ks < kGemvWarps && (total_out / L.opw) * L.ks < want_warps &&
         d.in_dim / (2 * L.ks) >= 256)
    L.ks *= 2;
  const int groups_per_block = kGemvWarps / L.ks;
  int blocks = 0;
  for (int s = 0; s < kGemvMaxSeg; ++s) {
    L.block0[s] = blocks;
    if (s < d.nseg) {
      const int groups = (d.seg[s].out_dim + L.opw - 1) / L.opw;
      blocks += (groups + groups_per_block - 1) / groups_per_block;
    }
  }
  L.block0[kGemvMaxSeg] = blocks;
  switch (L.opw) {
    case 4: return gemv_dispatch<4>(L, blocks, stream);
    case 2: return gemv_dispatch<2>(L, blocks, stream);
    default: return gemv_dispatch<1>(L, blocks, stream);
  }
}


// Bounded-wait self-test: thread 0 waits on an mbarrier that nothing arrives on. The wait
// gives up after the library's limit, raises the status bit and the kernel returns, so the
// context stays usable (the same path every kernel's waits take).
__global__ void wait_selftest_kernel(int* status) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ volatile int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    abort_flag = 0;
    fence_barrier_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) (void)mbar_wait(&bar, 0, &abort_flag, status);
}

cudaError_t launch_wait_selftest(int* status, cudaStream_t stream) {
  wait_selftest_kernel<<<1, 32, 0, stream>>>(status);
  return cudaGetLastError();
}

cudaError_t launch_rmsnorm_f32(const float* x, const __nv_bfloat16* g, float* y, int rows,
                               int hidden, float eps, cudaStream_t stream) {
  if (rows == 0) return cudaSuccess;
  rmsnorm_f32_kernel<<<rows, 256, 0, stream>>>(x, g, y, rows, hidden, eps);
  return cudaGetLastError();
}

cudaError_t launch_rope_up_rows(float* q, int hq, float* k, int hkv, float* v, int rows, int head_dim,
                                const RowUp* up, int rank, const float2* table, const RowPositions& pos,
                                bool table_by_row, cudaStream_t stream) {
  const long n = (long)rows * (hq + hkv) * (head_dim / 2) + (long)rows * hkv * head_dim;
  if (n == 0) return cudaSuccess;
  if (rank != 4 && rank != 8 && rank != 16) return cudaErrorInvalidValue;
  RowUp3 u{};
  for (int i = 0; i < 3; ++i) u.m[i] = up[i];
  return launch_kernel(rope_up_rows_kernel, dim3(cdiv(n, 256)), dim3(256), 0, stream, q, hq, k, hkv, v, rows,
                       head_dim, u, rank, table, pos, table_by_row ? 1 : 0);
}

int norm_up_slices(int dim) { return cdiv(dim, kNormSlice); }

cudaError_t launch_norm_up_rows(float* x, int dim, int rows, RowUp up, int up_rows, int rank,
                                const __nv_bfloat16* g, float eps, float* xn, float* part, int* counter,
                                cudaStream_t stream) {
  if (rows == 0) return cudaSuccess;
  if (rank != 4 && rank != 8 && rank != 16) return cudaErrorInvalidValue;
  const int slices = norm_up_slices(dim);
  return launch_kernel(norm_up_rows_kernel, dim3(rows * slices), dim3(kNormSlice), 0, stream, x, dim, up, up_rows,
                       rank, g, eps, xn, part, counter, slices);
}

cudaError_t launch_rows_up(float* x, int dim, int rows, RowUp up, int rank, cudaStream_t stream) {
  if (rows == 0 || !up.B) return cudaSuccess;
  if (rank != 4 && rank != 8 && rank != 16) return cudaErrorInvalidValue;
  return launch_kernel(rows_up_kernel, dim3(cdiv((long)rows * dim, 256)), dim3(256), 0, stream, x, dim, rows, up,
                       rank);
}

// (cos, sin) of the rows' own positions only: table[r][i] for position pos[r].
__global__ void rope_table_rows_kernel(float2* table, int rows, int half, const RowPositions pos,
                                       const __grid_constant__ RopeFreqs f) {
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= rows * half) return;
  const int r = idx / half, i = idx % half;
  double turns = static_cast<double>(pos.pos[r]) * f.turns_per_pos[i];
  turns -= floor(turns);
  float s, c;
  sincospif(static_cast<float>(2.0 * turns), &s, &c);
  table[idx] = make_float2(c, s);
}

// x[r] = embed[token_r] as fp32, the token read from device memory.
__global__ void embed_rows_f32_kernel(const __nv_bfloat16* __restrict__ embed, const TokenRows t,
                                      float* __restrict__ x, int hidden, int vocab, int* status) {
  const int r = blockIdx.y;
  const int tok = checked_token(*t.token[r], vocab,
                                blockIdx.x == 0 && threadIdx.x == 0 ? status : nullptr);
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < hidden; i += gridDim.x * blockDim.x)
    x[(size_t)r * hidden + i] = __bfloat162float(embed[(size_t)tok * hidden + i]);
}

// The rows' fp32 k, v [rows, Hkv * d] into slot pos % 16 of page page_table[pos / 16], bf16.
__global__ void kv_write_rows_kernel(const float* __restrict__ k, const float* __restrict__ v,
                                     __nv_bfloat16* kpages, __nv_bfloat16* vpages, const RowPages rp,
                                     int hkv, int d, int* status, const int* abort) {
  griddep_begin();  // k, v come from the kernels before
  if (call_aborted(abort)) return;
  const int r = blockIdx.y;
  const int pos = rp.pos[r];
  const int page = checked_page(rp.page_table[r][pos / kPage], rp.num_pages,
                                blockIdx.x == 0 && threadIdx.x == 0 ? status : nullptr);
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < hkv * d; i += gridDim.x * blockDim.x) {
    const int h = i / d, j = i % d;
    const size_t dst = (((size_t)page * hkv + h) * kPage + pos % kPage) * d + j;
    kpages[dst] = __float2bfloat16_rn(k[(size_t)r * hkv * d + i]);
    vpages[dst] = __float2bfloat16_rn(v[(size_t)r * hkv * d + i]);
  }
}

// out[r] = argmax_i logits[r, i], the lowest index among equal maxima.
// One block per row; 16-byte loads, four in flight per thread before their compares.
__global__ void argmax_rows_kernel(const float* __restrict__ logits, int vocab, int32_t* out,
                                   const int* abort) {
  if (call_aborted(abort)) return;
  const int r = blockIdx.x;
  const float* z = logits + (size_t)r * vocab;
  float best = -INFINITY;
  int arg = 0x7fffffff;
  auto take = [&](float v, int i) {
    if (v > best || (v == best && i < arg)) {
      best = v;
      arg = i;
    }
  };
  // elements before the row's first 16-byte boundary, then whole float4s, then the tail
  const int mis = static_cast<int>(reinterpret_cast<uintptr_t>(z) & 15) / 4;
  const int head = min(vocab, mis ? 4 - mis : 0);
  for (int i = threadIdx.x; i < head; i += blockDim.x) take(z[i], i);
  const int n4 = (vocab - head) / 4;
  const float4* z4 = reinterpret_cast<const float4*>(z + head);
  constexpr int kU = 4;
  for (int i0 = threadIdx.x; i0 < n4; i0 += kU * blockDim.x) {
    float4 v[kU];
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const int i = i0 + u * blockDim.x;
      v[u] = i < n4 ? __ldg(z4 + i) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const int i = i0 + u * blockDim.x;
      if (i < n4) {
        const int b = head + 4 * i;
        take(v[u].x, b);
        take(v[u].y, b + 1);
        take(v[u].z, b + 2);
        take(v[u].w, b + 3);
      }
    }
  }
  for (int i = head + 4 * n4 + threadIdx.x; i < vocab; i += blockDim.x) take(z[i], i);
  __shared__ float sb[32];
  __shared__ int sa[32];
  for (int o = 16; o > 0; o >>= 1) {
    const float ob = __shfl_xor_sync(0xffffffffu, best, o);
    const int oa = __shfl_xor_sync(0xffffffffu, arg, o);
    if (ob > best || (ob == best && oa < arg)) {
      best = ob;
      arg = oa;
    }
  }
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) {
    sb[w] = best;
    sa[w] = arg;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int i = 1; i < static_cast<int>(blockDim.x >> 5); ++i)
      if (sb[i] > best || (sb[i] == best && sa[i] < arg)) {
        best = sb[i];
        arg = sa[i];
      }
    out[r] = arg;
  }
}

cudaError_t launch_rope_table_rows(float2* table, const RowPositions& pos, int rows, int head_dim,
                                   double theta, cudaStream_t stream) {
  const int half = head_dim / 2;
  if (rows == 0) return cudaSuccess;
  if (half > 64) return cudaErrorInvalidValue;
  RopeFreqs f{};
  for (int i = 0; i < half; ++i)
    f.turns_per_pos[i] = std::pow(theta, -2.0 * i / head_dim) / (2.0 * 3.14159265358979323846);
  rope_table_rows_kernel<<<cdiv(rows * half, 256), 256, 0, stream>>>(table, rows, half, pos, f);
  return cudaGetLastError();
}

cudaError_t launch_embed_rows_f32(const __nv_bfloat16* embed, const TokenRows& t, int rows, float* x,
                                  int hidden, int vocab, int* status, cudaStream_t stream) {
  if (rows == 0) return cudaSuccess;
  embed_rows_f32_kernel<<<dim3(cdiv(hidden, 256), rows), 256, 0, stream>>>(embed, t, x, hidden, vocab,
                                                                            status);
  return cudaGetLastError();
}

cudaError_t launch_kv_write_rows(const float* k, const float* v, void* kpages, void* vpages,
                                 const RowPages& rp, int rows, int hkv, int head_dim, int* status,
                                 const int* abort, cudaStream_t stream) {
  if (rows == 0) return cudaSuccess;
  return launch_kernel(kv_write_rows_kernel, dim3(cdiv(hkv * head_dim, 256), rows), dim3(256), 0, stream, k, v,
                       static_cast<__nv_bfloat16*>(kpages), static_cast<__nv_bfloat16*>(vpages), rp, hkv,
                       head_dim, status, abort);
}

cudaError_t launch_argmax_rows(const float* logits, int rows, int vocab, int32_t* out,
                               cudaStream_t stream, const int* abort) {
  if (rows == 0) return cudaSuccess;
  argmax_rows_kernel<<<rows, 1024, 0, stream>>>(logits, vocab, out, abort);
  return cudaGetLastError();
}

cudaError_t launch_copy_bf16(__nv_bfloat16* dst, const __nv_bfloat16* src, size_t n, const int* abort,
                             cudaStream_t stream) {
  if (n == 0) return cudaSuccess;
  const size_t want = (n + 255) / 256;
  copy_bf16_kernel<<<static_cast<unsigned>(want < 4096 ? want : 4096), 256, 0, stream>>>(dst, src, n, abort);
  return cudaGetLastError();
}

cudaError_t launch_validate_pages(const PageCheck& pc, int num_pages, int* table, uint32_t mask, int* abort,
                                  int* status, cudaStream_t stream) {
  const int total = pc.first[pc.n];
  if (total == 0) return cudaSuccess;
  if (static_cast<uint32_t>(total) > (mask + 1u) / 2u) return cudaErrorInvalidValue;
  validate_pages_kernel<<<cdiv(total, 256), 256, 0, stream>>>(pc, num_pages, table, mask, abort, status);
  return cudaGetLastError();
}

cudaError_t launch_swiglu_up_rows(const float* g, const float* u, float* m, int rows, int f, RowUp up_g,
                                  RowUp up_u, int rank, cudaStream_t stream) {
  if (rows == 0) return cudaSuccess;
  if (rank != 4 && rank != 8 && rank != 16) return cudaErrorInvalidValue;
  return launch_kernel(swiglu_up_rows_kernel, dim3(cdiv((long)rows * f, 256)), dim3(256), 0, stream, g, u, m, rows,
                       f, up_g, up_u, rank);
}

cudaError_t launch_f32_to_bf16(const float* x, __nv_bfloat16* y, int n, cudaStream_t stream,
                               const int* abort) {
  if (n == 0) return cudaSuccess;
  f32_to_bf16_kernel<<<cdiv(n, 256), 256, 0, stream>>>(x, y, n, abort);
  return cudaGetLastError();
}
cudaError_t launch_bf16_to_f32(const __nv_bfloat16* x, float* y, int n, cudaStream_t stream) {
  if (n == 0) return cudaSuccess;
  bf16_to_f32_kernel<<<cdiv(n, 256), 256, 0, stream>>>(x, y, n);
  return cudaGetLastError();
}

cudaError_t launch_lm_head(const __nv_bfloat16* W, const float* h, int rows, int vocab, int hidden,
                           float* logits, int num_sms, cudaStream_t stream, const int* abort) {
  for (int r0 = 0; r0 < rows; r0 += kGemvMaxRows) {
    GemvDesc d{};
    d.abort = abort;
    d.seg[0].W = W;
    d.seg[0].out_dim = vocab;
    d.seg[0].scale = 1.f;
    d.seg[0].y = logits + (size_t)r0 * vocab;
    d.nseg = 1;
    d.in_dim = hidden;
    d.x = h + (size_t)r0 * hidden;
    d.rows = rows - r0 < kGemvMaxRows ? rows - r0 : kGemvMaxRows;
    cudaError_t e = launch_gemv(d, num_sms, stream, rows);  // one kernel for every chunk
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

cudaError_t launch_kl(const float* zref, const float* zcur, int rows, int vocab, float* out,
                      float* part, int splits, cudaStream_t stream) {
  if (rows == 0) return cudaSuccess;
  kl_partial_kernel<<<dim3(splits, rows), kKlThreads, 0, stream>>>(zref, zcur, vocab, splits, part);
  kl_final_kernel<<<cdiv(rows, 8), 256, 0, stream>>>(part, splits, out, rows);
  return cudaGetLastError();
}

}  // namespace crf
