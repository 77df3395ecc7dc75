// Internal launcher interface between the C ABI layer (api.cu) and the kernels.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include <atomic>

namespace crf {

// One-time set-up that CUDA keeps per device (kernel attributes): bit d of the mask records
// device d. Host threads may race to do it; doing it twice is harmless.
class PerDevice {
 public:
  // Sets *dev to the current device; true while its set-up is still to do.
  bool pending(int* dev) const {
    if (cudaGetDevice(dev) != cudaSuccess) *dev = -1;
    return *dev < 0 || *dev >= 64 || !((mask_.load(std::memory_order_acquire) >> *dev) & 1u);
  }
  void done(int dev) {
    if (dev >= 0 && dev < 64) mask_.fetch_or(1ull << dev, std::memory_order_acq_rel);
  }

 private:
  std::atomic<uint64_t> mask_{0};
};

constexpr int kMaxReq = 32;   // equals CRF_MAX_REQUESTS
constexpr int kPage = 16;
constexpr int kRankPad = 16;  // LoRA rank padded to one K=16 MMA step
// The scaled LoRA down product is kept as a bf16 pair hi + lo (lo = bf16(v - hi)): module
// slot j holds hi at columns [32j, 32j + 16) and lo at [32j + 16, 32j + 32) of a [rows, kXaCols]
// buffer. A projection GEMM computes it for its rows and reads it back as one 64-wide K block
// against BX = [B | B] rows (kBxCols wide) of the module (the up product).
constexpr int kXaCols = 128;
constexpr int kBxCols = 64;

// Programmatic dependent launch for chains of short kernels. While a PdlScope is alive on the
// calling thread, the launchers below that go through launch_kernel() give their kernels the
// programmatic-stream-serialization attribute: such a kernel becomes resident while its
// predecessor in the stream still runs, prefetches its weights and then waits for it
// (griddep_wait). Every kernel launched this way calls griddep_wait before it touches memory
// that an earlier kernel may write. The decode-row layer loop opens a scope.
class PdlScope {
 public:
  PdlScope();
  ~PdlScope();
  PdlScope(const PdlScope&) = delete;
  PdlScope& operator=(const PdlScope&) = delete;

 private:
  bool prev_;
};
bool pdl_active();

template <typename... KArgs, typename... Args>
cudaError_t launch_kernel(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                          cudaStream_t stream, Args&&... args) {
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = pdl_active() ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args&&>(args)...);
}

// Rows of a batched activation matrix that belong to each request.
struct ReqTable {
  int n;
  int num_pages;  // pool size; page ids are checked against it in a CRF_DEBUG build
  int row0[kMaxReq];
  int len[kMaxReq];
  const int32_t* page_table[kMaxReq];
};

enum EpiKind : int {
  kEpiQkv = 1,        // +bias, RoPE(q,k); q -> qbuf, k/v -> KV pages    (Eq. S3)
  kEpiResid = 2,      // out = bf16(resid + acc)                         (o / down projection)
  kEpiSwiGLU = 3      // out = bf16(silu(gate) * up), tile = [gate | up]  (MLP)
};

// Host description of one GEMM  D[M, cols] = A[M, K] * B[cols, K]^T (+ LoRA ext) -> epilogue.
// Column space: `ngroups` groups laid side by side, each with its own weight
// matrix (plain mode, nseg == 1), or one group whose tiles stack `nseg` equal
// row segments of different matrices (paired / stacked mode, ngroups == 1).
struct GemmDesc {
  const void* A;
  int M, K, lda;
  int ngroups, nseg;
  const void* B[3];       // map index g + s
  int B_rows[3];          // rows of each B matrix
  int ldb[3];
  int group_cols[3];      // valid output columns per group (plain) / per segment (stacked)
  // Unmerged LoRA (Eq. S3), computed inside the same launch. The first output tile of each
  // 256-row block also forms XA[:, 32j .. 32j + 32) = hi/lo of (alpha/r) x A_j^T for the n_slots
  // adapted modules (LA[j] = A_j, [rank, K]) and raises xa_flags[row block]; every output tile of
  // an adapted group then adds one K block: XA[:, xa_base[g] .. + 64] against BX[i] (the module's
  // [B | B] rows under its slot, zeros elsewhere; [B_rows[i], kBxCols], map index i like B).
  void* XA;
  int n_slots;
  const void* LA[3];
  const void* BX[3];
  int rank;
  float scale;            // alpha / r
  int* xa_flags;          // [row blocks of 256], zero before the launch
  int ext_on[3];          // per group
  int ext_steps[3];       // K = 16 steps of the block that carry data (2 per module)
  int xa_base[3];
  // epilogue
  int epi;
  void* out;
  int ldo;
  const void* resid;
  int ld_resid;
  const void* bias[3];
  const float2* rope;     // [positions][head_dim/2] (cos, sin)
  int head_dim, n_kv_heads;
  void* qbuf;
  int ldq;
  void* kpages;
  void* vpages;
  ReqTable req;
  int* status;
  const int* abort;       // per-call abort word (call_aborted), or null
};

// Launch the tcgen05 projection GEMM (CTA pairs, 256 x 256 tiles).
cudaError_t launch_gemm(const GemmDesc& d, int num_sms, cudaStream_t stream);

// ------------------------------------------------------------------ other kernels
cudaError_t launch_rope_table(float2* table, int n_pos, int head_dim, double theta,
                              cudaStream_t stream);
// BX rows of up to 4 modules: out[m][r, :] = 0 except columns [col_off[m], col_off[m] + 32) =
// [B_m[r, 0:16] | B_m[r, 0:16]] (rank padded with zeros); a null B_m gives all-zero rows.
struct BextDesc {
  const __nv_bfloat16* B[4];
  __nv_bfloat16* out[4];
  int rows[4];
  int col_off[4];
  int n, rank;
};
// RMSNorm of `rows` rows; with `bx`, the same launch also builds those BX rows (extra blocks).
cudaError_t launch_rmsnorm(const __nv_bfloat16* x, const __nv_bfloat16* g, __nv_bfloat16* y,
                           int rows, int hidden, float eps, cudaStream_t stream,
                           const BextDesc* bx = nullptr);
// Token ids outside [0, vocab) read row 0 and set kStatusBounds in *status.
cudaError_t launch_embed(const __nv_bfloat16* embed, const int32_t* tokens, __nv_bfloat16* out,
                         int n, int hidden, int vocab, int* status, cudaStream_t stream);

// Causal GQA prefill attention over the paged cache of the current layer.
struct AttnDesc {
  const __nv_bfloat16* q;  // [rows, Hq*d] post-RoPE
  int ldq;
  const __nv_bfloat16* kpages;  // [P][Hkv][16][d]
  const __nv_bfloat16* vpages;
  __nv_bfloat16* out;      // [rows, Hq*d]
  int ldo;
  int n_q_heads, n_kv_heads, head_dim;
  ReqTable req;
  int* status;
  const int* abort;
};
// tcgen05, S and O in TMEM: num_pages of the pool, total_rows of q (for the TMA maps).
cudaError_t launch_attention_tc(const AttnDesc& d, int num_pages, int total_rows,
                                cudaStream_t stream);

// Small-M decode path (the last prefix row through the layers after the window).
// Up to three row-stacked weight segments share one launch and one input x:
// y_s[r, j] = sum_i W_s[j, i] x[r, i] (+ bias_s[j]) (+ sum_k BL_s[j, k] xa_s[r, k]) (+ resid_s[r, j])
// y = scale * (W x) + bias + resid for each segment of weight rows sharing the input rows x: the
// projections' base rows and, as segments of their own, the LoRA A rows (y = the scaled down
// product xa, [rows, rank]).
struct GemvSeg {
  const __nv_bfloat16* W;  // [out_dim, in_dim]
  int out_dim;
  float scale;
  const __nv_bfloat16* bias;  // [out_dim] or null
  const float* resid;         // [rows, out_dim] fp32 or null
  float* y;                   // [rows, out_dim] fp32
};
constexpr int kGemvMaxSeg = 6;
struct GemvDesc {
  GemvSeg seg[kGemvMaxSeg];
  int nseg;
  int in_dim;
  const float* x;  // [rows, in_dim] fp32
  int rows;        // 1..8
  int prefetch;    // set by the launcher: prefetch the block's weight rows into L2 before the wait
  const int* abort;  // per-call abort word, or null
};
// Tensor-core GEMV (mma.sync, rows as a bf16 hi/lo pair); launch_gemv uses it when the call's
// rows (total_rows, the rows of all chunks one caller splits into launches of <= 8; 0 = d.rows)
// number three or more (one or two rows run faster on the CUDA-core kernel). One kernel per call
// keeps equal rows equal across chunks.
cudaError_t launch_gemv(const GemvDesc& d, int num_sms, cudaStream_t stream, int total_rows = 0);
cudaError_t launch_gemv_tc(const GemvDesc& d, int num_sms, cudaStream_t stream);
// The adapter's up product for decode rows, added where the projection's output is consumed:
// up[r, j] = sum_k B[j, k] xa[r, k] (B [out_dim, rank] bf16, xa [rows, rank] fp32 already scaled
// by alpha / r); a null B adds nothing.
struct RowUp {
  const __nv_bfloat16* B;
  const float* xa;
};
// x[r] += up(r) for r < up_rows (the rows that carry a pending product), then for every row
// xn[r] = rmsnorm(x[r]) * g (eps): the residual stream's update and the next RMSNorm in one launch,
// over norm_up_slices(dim) blocks per row. part: [rows, slices] fp32 scratch; counter: [rows] ints,
// zero before the first launch and left zero by every launch.
int norm_up_slices(int dim);
cudaError_t launch_norm_up_rows(float* x, int dim, int rows, RowUp up, int up_rows, int rank,
                                const __nv_bfloat16* g, float eps, float* xn, float* part, int* counter,
                                cudaStream_t stream);
// x[r] += up(r) for every row (the last projection's product, before the rows leave).
cudaError_t launch_rows_up(float* x, int dim, int rows, RowUp up, int rank, cudaStream_t stream);
cudaError_t launch_rmsnorm_f32(const float* x, const __nv_bfloat16* g, float* y, int rows,
                               int hidden, float eps, cudaStream_t stream);
// Single-query attention of `rows` decode rows (one per request) over pages [0, pos) plus own k/v.
struct DecodeAttnDesc {
  const float* q;          // [rows, Hq*d] fp32 post-RoPE
  const float* k_self;     // [rows, Hkv*d]
  const float* v_self;
  const __nv_bfloat16* kpages;
  const __nv_bfloat16* vpages;
  const int32_t* page_table[kMaxReq];  // per decode row
  int pos[kMaxReq];        // position of the decode row (= number of cached keys before it)
  float* out;              // [rows, Hq*d]
  float* part;             // scratch [rows, Hq, splits, d + 2]
  int rows, n_q_heads, n_kv_heads, head_dim, splits, max_pos;
  int chunks_per_block;    // set by launch_decode_attention
  const int* abort;        // per-call abort word, or null
};
// Decode attention streamed in 128-position chunks (TMA-staged pages, one block per SM walking
// a run of chunks of one row and kv head) + merge of the blocks' partials. `splits` in the
// descriptor must be at least decode_attention_splits(max position + 1).
cudaError_t launch_decode_attention(const DecodeAttnDesc& d, int num_pages, int num_sms, int* status,
                                    cudaStream_t stream);
int decode_attention_splits(int max_positions);
struct RowPositions {
  int pos[kMaxReq];
};
// q, k, v of decode rows: the up products added (up[0..2] for q, k, v), then rotate-half RoPE on
// q [rows, hq, head_dim] and k [rows, hkv, head_dim], row r at position pos.pos[r]; (cos, sin)
// from `table` [positions][head_dim / 2], or with table_by_row from row r of a
// [rows][head_dim / 2] table of the rows' own positions.
cudaError_t launch_rope_up_rows(float* q, int hq, float* k, int hkv, float* v, int rows, int head_dim,
                                const RowUp* up, int rank, const float2* table, const RowPositions& pos,
                                bool table_by_row, cudaStream_t stream);
// (cos, sin) of the rows' positions: table [rows][head_dim / 2].
cudaError_t launch_rope_table_rows(float2* table, const RowPositions& pos, int rows, int head_dim,
                                   double theta, cudaStream_t stream);
struct TokenRows {
  const int32_t* token[kMaxReq];  // device pointer to each row's input token id
};
// x [rows, hidden] fp32 = embed[token_r].
cudaError_t launch_embed_rows_f32(const __nv_bfloat16* embed, const TokenRows& t, int rows, float* x,
                                  int hidden, int vocab, int* status, cudaStream_t stream);
struct RowPages {
  const int32_t* page_table[kMaxReq];
  int pos[kMaxReq];
  int num_pages;
};
// Rows' fp32 k, v [rows, hkv * head_dim] into their page slot (page_table[pos / 16], pos % 16).
cudaError_t launch_kv_write_rows(const float* k, const float* v, void* kpages, void* vpages,
                                 const RowPages& rp, int rows, int hkv, int head_dim, int* status,
                                 const int* abort, cudaStream_t stream);
// out[r] = argmax of logits row r (lowest index among equal maxima).
// One block whose wait on an mbarrier nothing arrives on runs out after the bounded-wait limit
// and raises kStatusTimeout in *status (the failure path, exercised without a fault).
cudaError_t launch_wait_selftest(int* status, cudaStream_t stream);
cudaError_t launch_argmax_rows(const float* logits, int rows, int vocab, int32_t* out,
                               cudaStream_t stream, const int* abort = nullptr);
// m[r, j] = silu(g[r, j] + up_g) * (u[r, j] + up_u) over [rows, f] (gate and up in separate buffers).
cudaError_t launch_swiglu_up_rows(const float* g, const float* u, float* m, int rows, int f, RowUp up_g,
                                  RowUp up_u, int rank, cudaStream_t stream);
cudaError_t launch_f32_to_bf16(const float* x, __nv_bfloat16* y, int n, cudaStream_t stream,
                               const int* abort = nullptr);
// dst[0 .. n) = src[0 .. n) (bf16), unless the call's abort word is set.
cudaError_t launch_copy_bf16(__nv_bfloat16* dst, const __nv_bfloat16* src, size_t n, const int* abort,
                             cudaStream_t stream);
// The page-table check that opens crf_recompute_window and crf_decode_step: every id of every
// table in [0, num_pages) and no page twice across the tables. A failure sets *abort and raises
// kStatusPages in *status. `table` is scratch of (mask + 1) ints, mask + 1 a power of two at
// least twice the ids checked, filled with -1 (0xff bytes) before the launch.
struct PageCheck {
  const int32_t* pt[kMaxReq];
  int first[kMaxReq + 1];  // prefix of the tables' id counts
  int n;
};
cudaError_t launch_validate_pages(const PageCheck& pc, int num_pages, int* table, uint32_t mask, int* abort,
                                  int* status, cudaStream_t stream);
cudaError_t launch_bf16_to_f32(const __nv_bfloat16* x, float* y, int n, cudaStream_t stream);

// LM head + KL: logits [2*rows, V] (ref rows first) from final-normed hidden rows.
cudaError_t launch_lm_head(const __nv_bfloat16* W, const float* h, int rows, int vocab, int hidden,
                           float* logits, int num_sms, cudaStream_t stream, const int* abort = nullptr);
// KL per row from fp32 logits; part: scratch [rows][splits][5].
cudaError_t launch_kl(const float* zref, const float* zcur, int rows, int vocab, float* out,
                      float* part, int splits, cudaStream_t stream);
// Vocabulary splits per row of the KL reduction: about two blocks per SM over all rows, at least
// 1024 logits per split, at most kKlMaxSplits. Every KL entry point uses this count, so they
// reduce in the same order.
constexpr int kKlMaxSplits = 256;
inline int kl_split_count(int num_sms, int n_rows, int vocab) {
  int want = (2 * num_sms + n_rows - 1) / (n_rows > 0 ? n_rows : 1);
  const int by_vocab = (vocab + 1023) / 1024;
  want = want < by_vocab ? want : by_vocab;
  want = want < kKlMaxSplits ? want : kKlMaxSplits;
  return want < 1 ? 1 : want;
}

// Drift: per (layer, module) squared norms; see crf_drift.
struct DriftItem {
  const __nv_bfloat16* A0; const __nv_bfloat16* B0;
  const __nv_bfloat16* A1; const __nv_bfloat16* B1;
  int in_dim, out_dim;
  int out_index;           // layer * 7 + module
};
// Tensor-core drift (mma.sync Grams over the long dimensions, then a dependent-launched fp64
// combine per item); `workspace` is device scratch of drift_workspace_bytes(num_sms, rank,
// n_items) bytes (partial Grams). Launches drift_launches(n) kernels. out_sq holds n_out
// (layer, module) pairs; the entries of modules outside `adapted_mask` are cleared. A copy wait
// that exceeds its time limit sets kStatusTimeout in `status`.
size_t drift_workspace_bytes(int num_sms, int rank, int n_items);
int drift_launches(int n_items);
cudaError_t launch_drift(const DriftItem* items, int n_items, int rank, int n_out, int adapted_mask,
                         void* workspace, int num_sms, float* out_sq, int* status, cudaStream_t stream);

}  // namespace crf
