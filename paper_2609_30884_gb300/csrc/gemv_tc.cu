// Multi-row GEMV on the tensor cores: y[r, j] = scale sum_i W[j, i] x[r, i] (+ bias, residual)
// for up to 8 fp32 rows x (the first-step rows of a window and the rows of a generation step): the
// adapted projections of Eq. S3 for single rows (Section 3.1 hybrid rows, Section S2.1 decoding).
//
// mma.sync m16n8k16 with W as the A operand (16 output rows per warp) and the rows as the B
// operand (n = 8 row slots; slots past the row count are zero). x enters as a bf16 pair
// hi = bf16(x), lo = bf16(x - hi), so each product keeps ~16 mantissa bits of x (the W entries are
// exact in bf16) and the fp32 accumulation matches the scalar path's accuracy. Inside one 16-wide
// K step the logical k of the fragments is mapped to physical columns so that thread (g, c) owns
// columns 4c..4c+3 of both W's rows and x's row: logical {2c, 2c+1} -> 4c, 4c+1 and
// {2c+8, 2c+9} -> 4c+2, 4c+3 (a bijection on the step's 16 columns, the same for A and B), so
// every load is a contiguous vector. Warps of a block split K; a fixed-order shared-memory
// reduction and the epilogue (scale, bias, residual) follow.
// The work is bound by the weight bytes: the MMAs replace the 8 fp32 FMAs per weight element
// and row of the scalar kernel.
#include "common.cuh"
#include "kernels.h"

#include <algorithm>

namespace crf {

namespace {

constexpr int kWarps = 8;
constexpr int kRowsMax = 8;

struct GemvTcLaunch {
  GemvDesc d;
  int ks;                        // warps per 16-row tile (split K)
  int block0[kGemvMaxSeg + 1];   // first block of each segment
};

__device__ __forceinline__ void split_pair(float a, float b, uint32_t& hi, uint32_t& lo) {
  const __nv_bfloat16 ha = __float2bfloat16_rn(a), hb = __float2bfloat16_rn(b);
  hi = pack_bf16(__bfloat162float(ha), __bfloat162float(hb));
  lo = pack_bf16(a - __bfloat162float(ha), b - __bfloat162float(hb));
}

__global__ void __launch_bounds__(kWarps * 32) gemv_tc_kernel(const __grid_constant__ GemvTcLaunch L) {
  __shared__ float red[kWarps][16][kRowsMax];
  const GemvDesc& d = L.d;
  const int ks = L.ks;
  int s = 0;
  while (s < d.nseg - 1 && static_cast<int>(blockIdx.x) >= L.block0[s + 1]) ++s;
  const GemvSeg& sg = d.seg[s];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int tl = warp / ks, kp = warp % ks;
  const int tiles_per_block = kWarps / ks;
  const int tb = (static_cast<int>(blockIdx.x) - L.block0[s]) * tiles_per_block;
  if (d.prefetch) {  // the block's weight rows are contiguous
    const int jb0 = tb * 16, jb1 = min(sg.out_dim, jb0 + tiles_per_block * 16);
    if (jb0 < jb1) prefetch_l2_range(sg.W + (size_t)jb0 * d.in_dim, (size_t)(jb1 - jb0) * d.in_dim * 2);
  }
  griddep_begin();  // x, xa and the residual come from the kernels before
  if (call_aborted(d.abort)) return;
  const int j0 = (tb + tl) * 16;
  const int g = lane >> 2, c = lane & 3;
  const int K = d.in_dim;
  // K range of this warp in 32-column blocks (a 16-column tail goes to the last warp)
  const int nb = K / 32;
  const int per = (nb + ks - 1) / ks;
  const int b0 = kp * per, b1 = min(nb, b0 + per);
  const bool tail16 = (K % 32) != 0 && kp == ks - 1;
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
  if (j0 < sg.out_dim) {
    const int ja = min(j0 + g, sg.out_dim - 1), jb = min(j0 + g + 8, sg.out_dim - 1);
    const __nv_bfloat16* wa = sg.W + (size_t)ja * K;
    const __nv_bfloat16* wb = sg.W + (size_t)jb * K;
    const bool row_ok = g < d.rows;
    const float* xr = d.x + (size_t)(row_ok ? g : 0) * K;
#pragma unroll 4
    for (int b = b0; b < b1; ++b) {
      // physical columns 32b + 8c .. 32b + 8c + 7: k-step 0 takes the first 4, k-step 1 the last 4
      const int col = 32 * b + 8 * c;
      const uint4 ua = __ldg(reinterpret_cast<const uint4*>(wa + col));
      const uint4 ub = __ldg(reinterpret_cast<const uint4*>(wb + col));
      float4 x0 = make_float4(0.f, 0.f, 0.f, 0.f), x1 = x0;
      if (row_ok) {
        x0 = __ldg(reinterpret_cast<const float4*>(xr + col));
        x1 = __ldg(reinterpret_cast<const float4*>(xr + col + 4));
      }
      uint32_t h0, l0, h1, l1, h2, l2, h3, l3;
      split_pair(x0.x, x0.y, h0, l0);
      split_pair(x0.z, x0.w, h1, l1);
      split_pair(x1.x, x1.y, h2, l2);
      split_pair(x1.z, x1.w, h3, l3);
      const uint32_t a0[4] = {ua.x, ub.x, ua.y, ub.y};
      const uint32_t a1[4] = {ua.z, ub.z, ua.w, ub.w};
      mma16816(acc, a0, h0, h1);
      mma16816(acc, a0, l0, l1);
      mma16816(acc, a1, h2, h3);
      mma16816(acc, a1, l2, l3);
    }
    if (tail16) {
      const int col = 32 * nb + 4 * c;
      const uint2 ua = __ldg(reinterpret_cast<const uint2*>(wa + col));
      const uint2 ub = __ldg(reinterpret_cast<const uint2*>(wb + col));
      float4 x0 = make_float4(0.f, 0.f, 0.f, 0.f);
      if (row_ok) x0 = __ldg(reinterpret_cast<const float4*>(xr + col));
      uint32_t h0, l0, h1, l1;
      split_pair(x0.x, x0.y, h0, l0);
      split_pair(x0.z, x0.w, h1, l1);
      const uint32_t a0[4] = {ua.x, ub.x, ua.y, ub.y};
      mma16816(acc, a0, h0, h1);
      mma16816(acc, a0, l0, l1);
    }
  }
  // D fragment: rows j0 + g (acc 0, 1) and j0 + g + 8 (acc 2, 3), row slots 2c and 2c + 1
  red[warp][g][2 * c] = acc[0];
  red[warp][g][2 * c + 1] = acc[1];
  red[warp][g + 8][2 * c] = acc[2];
  red[warp][g + 8][2 * c + 1] = acc[3];
  __syncthreads();
  if (kp != 0 || j0 >= sg.out_dim) return;
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    const int idx = lane + 32 * u;  // 128 outputs of the tile: (row in tile, row slot)
    const int jj = idx / kRowsMax, r = idx % kRowsMax;
    const int j = j0 + jj;
    if (j >= sg.out_dim || r >= d.rows) continue;
    float v = 0.f;
    for (int q = 0; q < ks; ++q) v += red[tl * ks + q][jj][r];
    v *= sg.scale;
    if (sg.bias) v += __bfloat162float(sg.bias[j]);
    if (sg.resid) v += sg.resid[(size_t)r * sg.out_dim + j];
    sg.y[(size_t)r * sg.out_dim + j] = v;
  }
}

}  // namespace

cudaError_t launch_gemv_tc(const GemvDesc& d, int num_sms, cudaStream_t stream) {
  if (d.rows < 1 || d.rows > kRowsMax || d.nseg < 1 || d.nseg > kGemvMaxSeg || d.in_dim % 16 != 0)
    return cudaErrorInvalidValue;
  GemvTcLaunch L;
  L.d = d;
  L.d.prefetch = pdl_active() ? 1 : 0;
  int tiles = 0;
  for (int s = 0; s < d.nseg; ++s) tiles += (d.seg[s].out_dim + 15) / 16;
  if (tiles == 0) return cudaSuccess;
  // split K until the warps cover the SMs several times (pieces of >= 4 column blocks)
  const int want_warps = 16 * num_sms;
  L.ks = 1;
  while (L.ks < kWarps && tiles * L.ks < want_warps && (d.in_dim / 32) / (2 * L.ks) >= 4) L.ks *= 2;
  const int tiles_per_block = kWarps / L.ks;
  int blocks = 0;
  for (int s = 0; s < kGemvMaxSeg; ++s) {
    L.block0[s] = blocks;
    if (s < d.nseg) blocks += ((d.seg[s].out_dim + 15) / 16 + tiles_per_block - 1) / tiles_per_block;
  }
  L.block0[kGemvMaxSeg] = blocks;
  return launch_kernel(gemv_tc_kernel, dim3(blocks), dim3(kWarps * 32), 0, stream, L);
}

}  // namespace crf
