// C ABI of the bounded-recomputation library: argument validation, workspace
// planning and the per-layer launch sequence (see include/crf.h).
//
// Executable restart (Section 4.2): for each layer l of the union of the
// requests' windows, the rows of every request whose window covers l form one
// activation matrix, and the layer runs as
//   rmsnorm -> QKV GEMM (+LoRA down and up, bias, RoPE, q out, K/V to pages)
//   -> causal GQA attention over the pages -> O GEMM (+LoRA, residual)
//   -> rmsnorm -> gate|up GEMM (+LoRA, SwiGLU) -> down GEMM (+LoRA, residual)
// where each GEMM launch computes its own unmerged adapter term (Eq. S3).
// Then the last prefix row of each request that asks for it continues through
// layers e..N-1 against the historical cache (first-step state, Section S2.1).
#include "../../include/crf.h"
#include "common.cuh"
#include "kernels.h"

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <set>
#include <string>
#include <vector>

using namespace crf;

struct crf_ctx {
  int device;
  int num_sms;
  int* status_dev;
  // per-launch timing (crf_profile_enable)
  bool prof_on = false;
  std::vector<cudaEvent_t> ev;
  int ev_used = 0;
  struct Rec {
    int kind, idx, kernels;
  };
  std::vector<Rec> rec;
  int dropped = 0;
};

namespace {

enum ProfKind : int {
  kPQkv, kPO, kPGateUp, kPDown, kPAttn, kPNorm, kPEmbed, kPRope, kPCopy,
  kPDecode, kPLmHead, kPKl, kPDrift, kPCheck, kPNumKinds
};
const char* const kProfNames[kPNumKinds] = {
    "gemm_qkv_rope_paged", "gemm_o_resid", "gemm_gateup_swiglu", "gemm_down_resid",
    "attn_prefill_paged", "rmsnorm", "embed_gather", "rope_table", "row_copy",
    "tail_decode", "lm_head", "kl_reduce", "drift_gram", "page_check"};

// Brackets the launches issued in its lifetime with two events on `st` when
// profiling is on; `kernels` is how many kernels those launches are.
struct ProfScope {
  crf_ctx* c;
  int kind, kernels, idx;
  cudaStream_t st;
  ProfScope(crf_ctx* c_, int kind_, cudaStream_t st_, int kernels_ = 1)
      : c(c_), kind(kind_), kernels(kernels_), idx(-1), st(st_) {
    if (!c->prof_on) return;
    if (c->ev_used + 2 > static_cast<int>(c->ev.size())) {
      c->dropped += kernels;
      return;
    }
    idx = c->ev_used;
    c->ev_used += 2;
    cudaEventRecord(c->ev[idx], st);
  }
  ~ProfScope() {
    if (idx >= 0) {
      cudaEventRecord(c->ev[idx + 1], st);
      c->rec.push_back({kind, idx, kernels});
    }
  }
};

thread_local std::string g_err;

crf_status fail(crf_status st, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_err = buf;
  return st;
}

#define CRF_CUDA(expr)                                                                  \
  do {                                                                                  \
    cudaError_t _e = (expr);                                                            \
    if (_e != cudaSuccess)                                                              \
      return fail(CRF_ECUDA, "%s failed: %s (%s:%d)", #expr, cudaGetErrorString(_e), __FILE__, \
                  __LINE__);                                                            \
  } while (0)

inline size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

struct Dims {
  int N, h, hq, hkv, d, f, V, qd, kvd;
  float eps;
  double theta;
  bool bias;
};

Dims dims_of(const crf_model_dims& m) {
  Dims d;
  d.N = m.n_layers;
  d.h = m.hidden;
  d.hq = m.n_q_heads;
  d.hkv = m.n_kv_heads;
  d.d = m.head_dim;
  d.f = m.ffn;
  d.V = m.vocab;
  d.qd = m.n_q_heads * m.head_dim;
  d.kvd = m.n_kv_heads * m.head_dim;
  d.eps = m.rms_eps;
  d.theta = m.rope_theta;
  d.bias = m.qkv_bias != 0;
  return d;
}

void module_shape(const Dims& d, int m, int& out, int& in) {
  switch (m) {
    case CRF_MOD_Q: out = d.qd; in = d.h; break;
    case CRF_MOD_K:
    case CRF_MOD_V: out = d.kvd; in = d.h; break;
    case CRF_MOD_O: out = d.h; in = d.qd; break;
    case CRF_MOD_GATE:
    case CRF_MOD_UP: out = d.f; in = d.h; break;
    default: out = d.h; in = d.f; break;
  }
}

crf_status check_dims(const crf_model_dims& m) {
  if (m.n_layers < 1 || m.hidden < 1 || m.n_q_heads < 1 || m.n_kv_heads < 1 || m.ffn < 1 ||
      m.vocab < 1)
    return fail(CRF_EINVAL, "model dims must be positive");
  if (m.head_dim != 64 && m.head_dim != 128)
    return fail(CRF_EUNSUPPORTED, "head_dim %d unsupported (64 or 128)", m.head_dim);
  if (m.n_q_heads % m.n_kv_heads != 0)
    return fail(CRF_ESHAPE, "n_q_heads %d not a multiple of n_kv_heads %d", m.n_q_heads,
                m.n_kv_heads);
  if (m.hidden % 64 != 0 || m.ffn % 8 != 0)
    return fail(CRF_EUNSUPPORTED, "hidden must be a multiple of 64 and ffn of 8");
  if (!(m.rms_eps >= 0.f) || !(m.rope_theta > 0.f))
    return fail(CRF_EINVAL, "rms_eps must be >= 0 and rope_theta > 0");
  return CRF_OK;
}

crf_status check_lora(const crf_lora_dims& l) {
  if (l.rank != 4 && l.rank != 8 && l.rank != 16)
    return fail(CRF_EUNSUPPORTED, "LoRA rank %d unsupported (4, 8 or 16)", l.rank);
  if (!std::isfinite(l.alpha)) return fail(CRF_EINVAL, "LoRA alpha must be finite");
  if (l.module_mask & ~0x7Fu) return fail(CRF_EINVAL, "module_mask has bits beyond the 7 modules");
  return CRF_OK;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; }

// ---------------------------------------------------------------- workspace plan
struct Plan {
  int M = 0;          // max batched rows over layers
  int max_n = 0;
  int dec_rows = 0;   // requests asking for the first-step state
  int splits = 1;
  size_t off_g0, off_g1, off_x1, off_xn, off_q, off_o, off_mlp, off_xa, off_bx, off_rope;
  size_t off_dx0, off_dec;  // decode: bf16 starting rows, fp32 scratch
  size_t off_abort, off_ptab;  // the call's abort word; the page-check table (ptab_slots ints)
  // the projections' XA ready words (4 launches x ceil(M / 256) row blocks per layer) and the
  // decode-row norms' per-row counters (kMaxReq), laid out after the abort word so one clear at
  // the start of the call covers them all
  size_t flag_words = kMaxReq;
  uint32_t ptab_slots = 2;
  size_t dec_bytes;
  size_t total;
};

// output rows of module m (q, k, v, o, gate, up, down) and their sum
int module_rows(const Dims& D, int m) {
  const int r[7] = {D.qd, D.kvd, D.kvd, D.h, D.f, D.f, D.h};
  return r[m];
}
int module_rows_total(const Dims& D) {
  int t = 0;
  for (int m = 0; m < 7; ++m) t += module_rows(D, m);
  return t;
}

// decode attention partials: one per chunk of the longest prefix
int dec_splits(int max_n) { return decode_attention_splits(max_n); }

// Slots of the page-check table for `ids` page ids: a power of two, at least twice the ids.
uint32_t ptab_slots_for(long ids) {
  uint32_t s = 2;
  while (s < 2 * ids) s <<= 1;
  return s;
}

Plan make_plan(const Dims& D, const crf_request* reqs, int n_req) {
  Plan p;
  for (int l = 0; l < D.N; ++l) {
    int m = 0;
    for (int i = 0; i < n_req; ++i)
      if (reqs[i].s <= l && l < reqs[i].e) m += reqs[i].n_tokens;
    p.M = std::max(p.M, m);
  }
  for (int i = 0; i < n_req; ++i) {
    p.max_n = std::max(p.max_n, reqs[i].n_tokens);
    if (reqs[i].final_hidden_out) ++p.dec_rows;
  }
  const size_t M = static_cast<size_t>(p.M);
  size_t o = 0;
  auto take = [&](size_t bytes) {
    const size_t at = o;
    o = align256(o + bytes);
    return at;
  };
  p.off_g0 = take(M * D.h * 2);
  p.off_g1 = take(M * D.h * 2);
  p.off_x1 = take(M * D.h * 2);
  p.off_xn = take(M * D.h * 2);
  p.off_q = take(M * D.qd * 2);
  p.off_o = take(M * D.qd * 2);
  p.off_mlp = take(M * D.f * 2);
  p.off_xa = take(M * kXaCols * 2);
  p.off_bx = take(static_cast<size_t>(module_rows_total(D)) * kBxCols * 2);
  p.off_rope = take(static_cast<size_t>(p.max_n) * (D.d / 2) * sizeof(float2));
  p.off_dx0 = take(static_cast<size_t>(n_req) * D.h * 2);
  long ids = 0;
  for (int i = 0; i < n_req; ++i) ids += (reqs[i].n_tokens + kPage - 1) / kPage;
  p.ptab_slots = ptab_slots_for(ids);
  int layers = 0;
  for (int l = 0; l < D.N; ++l) {
    bool any = false;
    for (int i = 0; i < n_req; ++i) any |= reqs[i].s <= l && l < reqs[i].e;
    layers += any ? 1 : 0;
  }
  p.flag_words = static_cast<size_t>(layers) * 4 * ((p.M + 255) / 256) + kMaxReq;
  p.off_abort = take((1 + p.flag_words) * sizeof(int));
  p.off_ptab = take(static_cast<size_t>(p.ptab_slots) * sizeof(int));
  p.splits = dec_splits(p.max_n);
  // decode scratch per row, fp32: x, xn, x1, q, k, v, o, xa (7 slots), gu, m, norm partials,
  // attention partials
  const size_t dec_row = static_cast<size_t>(3 * D.h + 2 * D.qd + 2 * D.kvd + 7 * kRankPad + 3 * D.f + norm_up_slices(D.h)) * 4 +
                         static_cast<size_t>(D.hq) * p.splits * (D.d + 2) * 4;
  p.dec_bytes = align256(dec_row * std::max(1, p.dec_rows));
  p.off_dec = take(p.dec_rows ? p.dec_bytes : 0);
  p.total = o;
  return p;
}

// ---------------------------------------------------------------- request checks
crf_status check_model_layers(const crf_model* model, int l0, int l1, const Dims& D) {
  for (int l = l0; l < l1; ++l) {
    const crf_layer_weights& w = model->layers[l];
    for (int m = 0; m < CRF_NUM_MODULES; ++m)
      if (!w.W[m] || !aligned16(w.W[m])) return fail(CRF_EINVAL, "layer %d weight %d null or misaligned", l, m);
    if (!w.ln1 || !w.ln2) return fail(CRF_EINVAL, "layer %d norm gain is null", l);
    if (D.bias)
      for (int j = 0; j < 3; ++j)
        if (!w.bias[j] || !aligned16(w.bias[j]))
          return fail(CRF_EINVAL, "layer %d qkv bias %d null or misaligned", l, j);
  }
  return CRF_OK;
}

crf_status check_adapter_layers(const crf_adapter* a, int l0, int l1) {
  for (int l = l0; l < l1; ++l)
    for (int m = 0; m < CRF_NUM_MODULES; ++m) {
      if (!(a->dims.module_mask & (1u << m))) continue;
      const void* A = a->A[l * 7 + m];
      const void* B = a->B[l * 7 + m];
      if (!A || !B || !aligned16(A) || !aligned16(B))
        return fail(CRF_EINVAL, "adapter layer %d module %d factor null or misaligned", l, m);
    }
  return CRF_OK;
}

// ---------------------------------------------------------------- one layer
struct LayerCtx {
  const Dims* D;
  crf_ctx* ctx;
  const crf_model* model;
  const crf_adapter* ad;
  const crf_kv_pool* pool;
  cudaStream_t st;
  uint8_t* ws;
  const Plan* plan;
  float scale;
  const int* abort;  // the call's abort word (set by the page-table check)
  int* xa_flags;     // this layer's XA ready words (4 projections x row blocks), zero
};

bool adapted(const crf_adapter* a, int m) { return (a->dims.module_mask >> m) & 1u; }

crf_status run_layer(const LayerCtx& c, int l, const __nv_bfloat16* X_in, __nv_bfloat16* X_out,
                     int M, const ReqTable& rt) {
  const Dims& D = *c.D;
  const crf_layer_weights& w = c.model->layers[l];
  const Plan& p = *c.plan;
  uint8_t* ws = c.ws;
  auto* X1 = reinterpret_cast<__nv_bfloat16*>(ws + p.off_x1);
  auto* XN = reinterpret_cast<__nv_bfloat16*>(ws + p.off_xn);
  auto* Q = reinterpret_cast<__nv_bfloat16*>(ws + p.off_q);
  auto* O = reinterpret_cast<__nv_bfloat16*>(ws + p.off_o);
  auto* MLP = reinterpret_cast<__nv_bfloat16*>(ws + p.off_mlp);
  auto* XA = reinterpret_cast<__nv_bfloat16*>(ws + p.off_xa);
  auto* rope = reinterpret_cast<const float2*>(ws + p.off_rope);
  // one ready word per 256-row block for each of the layer's four projection launches
  int* flags = c.xa_flags;
  const int flag_stride = (p.M + 255) / 256;
  // BX = [B | B] rows of every module of layer l under its XA slot (up follows gate when both are
  // adapted, so one K block carries the stacked gate|up pair), built by the RMSNorm launches:
  // q, k, v, o with the first, gate, up, down with the second
  __nv_bfloat16* BX[7];
  BextDesc bext[2]{};
  {
    auto* bx = reinterpret_cast<__nv_bfloat16*>(ws + p.off_bx);
    for (int m = 0; m < 7; ++m) {
      BX[m] = bx;
      const int rows = module_rows(D, m);
      bx += static_cast<size_t>(rows) * kBxCols;
      // a stacked gate|up tile reads both modules' rows: an unadapted one's are zeros
      const bool need = adapted(c.ad, m) || ((m == CRF_MOD_GATE || m == CRF_MOD_UP) &&
                                              (adapted(c.ad, CRF_MOD_GATE) || adapted(c.ad, CRF_MOD_UP)));
      if (!need) continue;
      BextDesc& d = bext[m < CRF_MOD_GATE ? 0 : 1];
      d.B[d.n] = adapted(c.ad, m) ? static_cast<const __nv_bfloat16*>(c.ad->B[l * 7 + m]) : nullptr;
      d.out[d.n] = BX[m];
      d.rows[d.n] = rows;
      d.col_off[d.n] = (m == CRF_MOD_UP && adapted(c.ad, CRF_MOD_GATE)) ? 32 : 0;
      ++d.n;
    }
    bext[0].rank = bext[1].rank = c.ad->dims.rank;
  }
  // the unmerged adapter of the listed modules, slots in list order (Eq. S3)
  auto set_lora = [&](GemmDesc& g, const int* mods, int nm, int* slot_of) {
    g.n_slots = 0;
    for (int s = 0; s < nm; ++s) {
      slot_of[s] = -1;
      if (!adapted(c.ad, mods[s])) continue;
      slot_of[s] = g.n_slots;
      g.LA[g.n_slots++] = c.ad->A[l * 7 + mods[s]];
    }
    if (!g.n_slots) return;
    g.XA = XA;
    g.rank = c.ad->dims.rank;
    g.scale = c.scale;
    g.xa_flags = flags;
    flags += flag_stride;
  };

  // 1. RMSNorm before attention
  {
    ProfScope ps(c.ctx, kPNorm, c.st);
    CRF_CUDA(launch_rmsnorm(X_in, static_cast<const __nv_bfloat16*>(w.ln1), XN, M, D.h, D.eps, c.st,
                            bext[0].n ? &bext[0] : nullptr));
  }

  // 2-3. q/k/v projections (+ LoRA, bias, RoPE; K/V into the pages of layer l)
  {
    GemmDesc g;
    std::memset(&g, 0, sizeof(g));
    g.A = XN;
    g.M = M;
    g.K = D.h;
    g.lda = D.h;
    g.ngroups = 3;
    g.nseg = 1;
    const int mods[3] = {CRF_MOD_Q, CRF_MOD_K, CRF_MOD_V};
    int slot[3];
    set_lora(g, mods, 3, slot);
    const int rows[3] = {D.qd, D.kvd, D.kvd};
    for (int m = 0; m < 3; ++m) {
      g.B[m] = w.W[m];
      g.B_rows[m] = rows[m];
      g.ldb[m] = D.h;
      g.group_cols[m] = rows[m];
      if (slot[m] >= 0) {
        g.BX[m] = BX[m];
        g.ext_on[m] = 1;
        g.ext_steps[m] = 2;
        g.xa_base[m] = 32 * slot[m];
      }
      g.bias[m] = D.bias ? w.bias[m] : nullptr;
    }
    g.epi = kEpiQkv;
    g.rope = rope;
    g.head_dim = D.d;
    g.n_kv_heads = D.hkv;
    g.qbuf = Q;
    g.ldq = D.qd;
    g.kpages = c.pool->k_pages[l];
    g.vpages = c.pool->v_pages[l];
    g.req = rt;
    g.status = c.ctx->status_dev;
    g.abort = c.abort;
    ProfScope ps(c.ctx, kPQkv, c.st);
    CRF_CUDA(launch_gemm(g, c.ctx->num_sms, c.st));
  }

  // 4. causal GQA attention over the pages of layer l
  {
    AttnDesc a;
    a.q = Q;
    a.ldq = D.qd;
    a.kpages = static_cast<const __nv_bfloat16*>(c.pool->k_pages[l]);
    a.vpages = static_cast<const __nv_bfloat16*>(c.pool->v_pages[l]);
    a.out = O;
    a.ldo = D.qd;
    a.n_q_heads = D.hq;
    a.n_kv_heads = D.hkv;
    a.head_dim = D.d;
    a.req = rt;
    a.status = c.ctx->status_dev;
    a.abort = c.abort;
    ProfScope ps(c.ctx, kPAttn, c.st);
    CRF_CUDA(launch_attention_tc(a, c.pool->num_pages, M, c.st));
  }

  // 5-6. output projection + residual: X1 = X_in + O W_o^T (+ LoRA)
  auto proj_resid = [&](int m, const void* A, int K, const void* resid, void* out) -> cudaError_t {
    GemmDesc g;
    std::memset(&g, 0, sizeof(g));
    g.A = A;
    g.M = M;
    g.K = K;
    g.lda = K;
    g.ngroups = 1;
    g.nseg = 1;
    g.B[0] = w.W[m];
    g.B_rows[0] = D.h;
    g.ldb[0] = K;
    g.group_cols[0] = D.h;
    int slot[1];
    set_lora(g, &m, 1, slot);
    if (slot[0] >= 0) {
      g.BX[0] = BX[m];
      g.ext_on[0] = 1;
      g.ext_steps[0] = 2;
      g.xa_base[0] = 0;
    }
    g.epi = kEpiResid;
    g.out = out;
    g.ldo = D.h;
    g.resid = resid;
    g.ld_resid = D.h;
    g.status = c.ctx->status_dev;
    g.abort = c.abort;
    ProfScope ps(c.ctx, m == CRF_MOD_O ? kPO : kPDown, c.st);
    return launch_gemm(g, c.ctx->num_sms, c.st);
  };
  CRF_CUDA(proj_resid(CRF_MOD_O, O, D.qd, X_in, X1));

  // 7. RMSNorm before the MLP
  {
    ProfScope ps(c.ctx, kPNorm, c.st);
    CRF_CUDA(launch_rmsnorm(X1, static_cast<const __nv_bfloat16*>(w.ln2), XN, M, D.h, D.eps, c.st,
                            bext[1].n ? &bext[1] : nullptr));
  }

  // 8-9. gate|up projections with SwiGLU epilogue
  {
    GemmDesc g;
    std::memset(&g, 0, sizeof(g));
    g.A = XN;
    g.M = M;
    g.K = D.h;
    g.lda = D.h;
    g.ngroups = 1;
    g.nseg = 2;
    const int mods[2] = {CRF_MOD_GATE, CRF_MOD_UP};
    int slot[2];
    set_lora(g, mods, 2, slot);
    for (int s = 0; s < 2; ++s) {
      g.B[s] = w.W[mods[s]];
      g.B_rows[s] = D.f;
      g.ldb[s] = D.h;
      g.BX[s] = BX[mods[s]];  // all-zero rows for a module without adapter
    }
    if (g.n_slots) {
      // one K block carries both slots; each segment's B rows sit under its own slot only
      g.ext_on[0] = 1;
      g.ext_steps[0] = 2 * g.n_slots;
      g.xa_base[0] = 0;
    }
    g.group_cols[0] = D.f;
    g.epi = kEpiSwiGLU;
    g.out = MLP;
    g.ldo = D.f;
    g.status = c.ctx->status_dev;
    g.abort = c.abort;
    ProfScope ps(c.ctx, kPGateUp, c.st);
    CRF_CUDA(launch_gemm(g, c.ctx->num_sms, c.st));
  }

  // 10-11. down projection + residual: X_out = X1 + MLP W_d^T (+ LoRA)
  CRF_CUDA(proj_resid(CRF_MOD_DOWN, MLP, D.f, X1, X_out));
  return CRF_OK;
}

// ---------------------------------------------------------------- decode rows
// Carry the last prefix row of every listed request through layers [e_i, N) against each
// layer's cached K/V at positions < n_i - 1 (fp32 rows). Rows are ordered by window end, so
// the rows active at a layer are a prefix of the batch and each layer's weights are read once
// for all of them (GEMV launches of up to 8 rows).
struct DecodeRow {
  int e;            // first layer to run
  int pos;          // position of the row (= n - 1)
  const int32_t* page_table;
  const __nv_bfloat16* start;  // bf16 [h], or null when the row starts from `token`'s embedding
  void* out;        // bf16 [h], or null (the final fp32 rows stay in the decode scratch)
  const int32_t* token = nullptr;  // device, the row's input token (generation steps)
};

// Generation steps (crf_decode_step) write each layer's k, v of the row into its page slot and
// take RoPE angles from a table of the rows' own positions; the first-step rows of a window do
// neither (their positions are in the window's full table, and the historical cache stays).
struct DecodeOpts {
  bool write_kv = false;
  const float2* rope_by_row = nullptr;
};

crf_status decode_rows(const LayerCtx& c, std::vector<DecodeRow> rows, const DecodeOpts& opt = DecodeOpts()) {
  const Dims& D = *c.D;
  const Plan& p = *c.plan;
  const int R = static_cast<int>(rows.size());
  if (R == 0) return CRF_OK;
  std::stable_sort(rows.begin(), rows.end(), [](const DecodeRow& a, const DecodeRow& b) { return a.e < b.e; });
  const int l0 = rows[0].e;
  const size_t Rs = static_cast<size_t>(R);
  const int rank = c.ad->dims.rank;
  float* x = reinterpret_cast<float*>(c.ws + p.off_dec);
  float* xn = x + Rs * D.h;
  float* x1 = xn + Rs * D.h;
  float* q = x1 + Rs * D.h;
  float* k = q + Rs * D.qd;
  float* v = k + Rs * D.kvd;
  float* o = v + Rs * D.kvd;
  float* xa = o + Rs * D.qd;  // one [R, rank] slot per module: q, k, v, o, gate, up, down
  float* gu = xa + 7 * Rs * kRankPad;
  float* m = gu + Rs * 2 * D.f;
  float* npart = m + Rs * D.f;  // [R, slices] partial sums of squares of the norms
  float* part = npart + Rs * norm_up_slices(D.h);
  int* ncount = reinterpret_cast<int*>(c.ws + p.off_abort) + 1 + (p.flag_words - kMaxReq);
  auto xa_of = [&](int mod) { return xa + static_cast<size_t>(mod) * Rs * kRankPad; };
  auto up_of = [&](int l, int mod) {
    RowUp u{};
    if (adapted(c.ad, mod)) {
      u.B = static_cast<const __nv_bfloat16*>(c.ad->B[l * 7 + mod]);
      u.xa = xa_of(mod);
    }
    return u;
  };
  // kernels per layer: 2 norms (with the pending up products), 4 GEMV passes per 8 rows, RoPE
  // (with the q|k|v up products), 2 attention, SwiGLU (with the gate|up up products), the K/V
  // write of a generation step; then the last layer's down up product and a conversion per row
  int launches = 0;
  for (const auto& r : rows) launches += (r.start ? 1 : 0) + (r.out ? 1 : 0);
  bool any_token = false;
  for (const auto& r : rows) any_token |= r.token != nullptr;
  launches += any_token ? 1 : 0;
  for (int l = l0; l < D.N; ++l) {
    int nr = 0;
    for (const auto& r : rows) nr += r.e <= l;
    launches += 6 + (opt.write_kv ? 1 : 0) + 4 * ((nr + 7) / 8);
  }
  if (l0 < D.N && adapted(c.ad, CRF_MOD_DOWN)) ++launches;
  ProfScope ps(c.ctx, kPDecode, c.st, launches);
  TokenRows tr{};
  for (int i = 0; i < R; ++i) {
    if (rows[i].token) {
      tr.token[i] = rows[i].token;
    } else {
      CRF_CUDA(launch_bf16_to_f32(rows[i].start, x + i * static_cast<size_t>(D.h), D.h, c.st));
    }
  }
  if (any_token) {
    // token rows are the whole batch (a generation step), so one launch covers them
    for (int i = 0; i < R; ++i)
      if (!rows[i].token) return fail(CRF_EINVAL, "decode rows mix token and hidden starts");
    CRF_CUDA(launch_embed_rows_f32(static_cast<const __nv_bfloat16*>(c.model->embed), tr, R, x, D.h, D.V,
                                   c.ctx->status_dev, c.st));
  }
  // one weight pass per group of up to 8 rows: the modules' base rows (y = W in + bias + resid)
  // and, as segments of their own, their LoRA A rows (xa = (alpha/r) A in, Eq. S3)
  auto proj = [&](int l, int nr, const int* mods, int nm, const float* in, int in_dim, float* const* ys,
                  const int* outs, const float* resid, int resid_ld) -> cudaError_t {
    for (int r0 = 0; r0 < nr; r0 += 8) {
      GemvDesc g{};
      g.abort = c.abort;
      g.in_dim = in_dim;
      g.x = in + static_cast<size_t>(r0) * in_dim;
      g.rows = std::min(8, nr - r0);
      for (int s = 0; s < nm; ++s) {
        const int mod = mods[s];
        GemvSeg& sg = g.seg[g.nseg++];
        sg.W = static_cast<const __nv_bfloat16*>(c.model->layers[l].W[mod]);
        sg.out_dim = outs[s];
        sg.scale = 1.f;
        sg.bias = (mod < 3 && D.bias) ? static_cast<const __nv_bfloat16*>(c.model->layers[l].bias[mod])
                                      : nullptr;
        sg.y = ys[s] + static_cast<size_t>(r0) * outs[s];
        sg.resid = resid ? resid + static_cast<size_t>(r0) * resid_ld : nullptr;
      }
      for (int s = 0; s < nm; ++s) {
        const int mod = mods[s];
        if (!adapted(c.ad, mod)) continue;
        GemvSeg& sg = g.seg[g.nseg++];
        sg.W = static_cast<const __nv_bfloat16*>(c.ad->A[l * 7 + mod]);
        sg.out_dim = rank;
        sg.scale = c.scale;
        sg.y = xa_of(mod) + static_cast<size_t>(r0) * rank;
      }
      cudaError_t e = launch_gemv(g, c.ctx->num_sms, c.st, nr);
      if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
  };
  const int m_qkv[3] = {CRF_MOD_Q, CRF_MOD_K, CRF_MOD_V};
  const int o_qkv[3] = {D.qd, D.kvd, D.kvd};
  float* const y_qkv[3] = {q, k, v};
  const int m_o[1] = {CRF_MOD_O}, o_o[1] = {D.h};
  float* const y_o[1] = {x1};
  const int m_gu[2] = {CRF_MOD_GATE, CRF_MOD_UP}, o_gu[2] = {D.f, D.f};
  float* const y_gu[2] = {gu, gu + Rs * D.f};
  const int m_d[1] = {CRF_MOD_DOWN}, o_d[1] = {D.h};
  float* const y_d[1] = {x};
  RowPositions rp{};
  for (int i = 0; i < R; ++i) rp.pos[i] = rows[i].pos;
  int nr_prev = 0;  // rows that carry the previous layer's pending down up product
  {
    // the layer loop is a chain of short kernels only: each may become resident and prefetch its
    // weights while the one before it finishes
    PdlScope pdl;
    for (int l = l0; l < D.N; ++l) {
      int nr = 0;
      while (nr < R && rows[nr].e <= l) ++nr;
      const crf_layer_weights& w = c.model->layers[l];
      // x += the previous layer's down up product (rows active there), xn = RMSNorm(x)
      CRF_CUDA(launch_norm_up_rows(x, D.h, nr, l > l0 ? up_of(l - 1, CRF_MOD_DOWN) : RowUp{}, nr_prev, rank,
                                   static_cast<const __nv_bfloat16*>(w.ln1), D.eps, xn, npart, ncount, c.st));
      CRF_CUDA(proj(l, nr, m_qkv, 3, xn, D.h, y_qkv, o_qkv, nullptr, 0));
      const RowUp up_qkv[3] = {up_of(l, CRF_MOD_Q), up_of(l, CRF_MOD_K), up_of(l, CRF_MOD_V)};
      CRF_CUDA(launch_rope_up_rows(q, D.hq, k, D.hkv, v, nr, D.d, up_qkv, rank,
                                   opt.rope_by_row ? opt.rope_by_row
                                                   : reinterpret_cast<const float2*>(c.ws + p.off_rope),
                                   rp, opt.rope_by_row != nullptr, c.st));
      DecodeAttnDesc a;
      std::memset(&a, 0, sizeof(a));
      a.q = q;
      a.k_self = k;
      a.v_self = v;
      a.kpages = static_cast<const __nv_bfloat16*>(c.pool->k_pages[l]);
      a.vpages = static_cast<const __nv_bfloat16*>(c.pool->v_pages[l]);
      for (int i = 0; i < nr; ++i) {
        a.page_table[i] = rows[i].page_table;
        a.pos[i] = rows[i].pos;
      }
      a.out = o;
      a.part = part;
      a.rows = nr;
      a.n_q_heads = D.hq;
      a.n_kv_heads = D.hkv;
      a.head_dim = D.d;
      a.splits = p.splits;
      a.abort = c.abort;
      CRF_CUDA(launch_decode_attention(a, c.pool->num_pages, c.ctx->num_sms, c.ctx->status_dev, c.st));
      if (opt.write_kv) {
        RowPages pg{};
        for (int i = 0; i < nr; ++i) {
          pg.page_table[i] = rows[i].page_table;
          pg.pos[i] = rows[i].pos;
        }
        pg.num_pages = c.pool->num_pages;
        CRF_CUDA(launch_kv_write_rows(k, v, c.pool->k_pages[l], c.pool->v_pages[l], pg, nr, D.hkv, D.d,
                                      c.ctx->status_dev, c.abort, c.st));
      }
      // x1 = x + o W_o^T, then x1 += the o up product and xn = RMSNorm(x1)
      CRF_CUDA(proj(l, nr, m_o, 1, o, D.qd, y_o, o_o, x, D.h));
      CRF_CUDA(launch_norm_up_rows(x1, D.h, nr, up_of(l, CRF_MOD_O), nr, rank,
                                   static_cast<const __nv_bfloat16*>(w.ln2), D.eps, xn, npart, ncount, c.st));
      CRF_CUDA(proj(l, nr, m_gu, 2, xn, D.h, y_gu, o_gu, nullptr, 0));
      // gate rows then up rows: SwiGLU over [nr, f] with the up half Rs * f further on
      CRF_CUDA(launch_swiglu_up_rows(gu, gu + Rs * D.f, m, nr, D.f, up_of(l, CRF_MOD_GATE), up_of(l, CRF_MOD_UP),
                                     rank, c.st));
      // x = x1 + m W_d^T; its up product is added by the next layer's norm (or below)
      CRF_CUDA(proj(l, nr, m_d, 1, m, D.f, y_d, o_d, x1, D.h));
      nr_prev = nr;
    }
    if (l0 < D.N) CRF_CUDA(launch_rows_up(x, D.h, nr_prev, up_of(D.N - 1, CRF_MOD_DOWN), rank, c.st));
  }
  for (int i = 0; i < R; ++i)
    if (rows[i].out)
      CRF_CUDA(launch_f32_to_bf16(x + i * static_cast<size_t>(D.h),
                                  static_cast<__nv_bfloat16*>(rows[i].out), D.h, c.st, c.abort));
  return CRF_OK;
}

// Page ids are checked on the device by the first kernel of every call that uses them. Only a
// CRF_DEBUG build run with CRF_DEBUG_DEVICE_CHECKS_ONLY=1 skips that check, so that the per-use
// checks of that build alone stand between a bad id and the pool (the way its tests exercise them).
bool device_page_check() {
  if (!kDebugBuild) return true;
  const char* e = std::getenv("CRF_DEBUG_DEVICE_CHECKS_ONLY");
  return !(e && e[0] == '1');
}

// Opens a call on `st`: clears the call's abort word and the `flag_words` ready words after it,
// and checks every page id of the listed tables (in [0, num_pages), no page twice). Enqueued
// work only: the host does not wait.
crf_status open_call(crf_ctx* ctx, const PageCheck& pc, int num_pages, uint8_t* ws, size_t off_abort,
                     size_t flag_words, size_t off_ptab, uint32_t ptab_slots, cudaStream_t st) {
  int* abort = reinterpret_cast<int*>(ws + off_abort);
  ProfScope ps(ctx, kPCheck, st, device_page_check() ? 1 : 0);
  CRF_CUDA(cudaMemsetAsync(abort, 0, (1 + flag_words) * sizeof(int), st));
  if (!device_page_check()) return CRF_OK;
  int* table = reinterpret_cast<int*>(ws + off_ptab);
  CRF_CUDA(cudaMemsetAsync(table, 0xff, static_cast<size_t>(ptab_slots) * sizeof(int), st));
  CRF_CUDA(launch_validate_pages(pc, num_pages, table, ptab_slots - 1, abort, ctx->status_dev, st));
  return CRF_OK;
}

crf_status validate_requests(const crf_ctx* ctx, const crf_model* model, const crf_adapter* cur,
                             const crf_kv_pool* pool, const crf_request* reqs, int n_req,
                             const Dims& D) {
  if (n_req < 1 || n_req > CRF_MAX_REQUESTS)
    return fail(CRF_EINVAL, "n_req %d outside [1, %d]", n_req, CRF_MAX_REQUESTS);
  if (!pool || !pool->k_pages || !pool->v_pages || pool->num_pages < 1)
    return fail(CRF_EINVAL, "kv pool missing");
  for (int i = 0; i < n_req; ++i) {
    const crf_request& r = reqs[i];
    if (r.n_tokens < 1) return fail(CRF_EINVAL, "request %d: n_tokens must be >= 1", i);
    if (r.s < 0 || r.s > r.e || r.e > D.N)
      return fail(CRF_EINVAL, "request %d: window [%d,%d) outside [0,%d]", i, r.s, r.e, D.N);
    if (r.s == r.e && !r.final_hidden_out)
      return fail(CRF_EINVAL, "request %d: empty window without final_hidden_out", i);
    if (!r.page_table) return fail(CRF_EINVAL, "request %d: page_table is null", i);
    if (r.s == 0 && !r.tokens) return fail(CRF_EINVAL, "request %d: tokens required when s == 0", i);
    if (r.s > 0 && !r.hidden_in) return fail(CRF_EINVAL, "request %d: hidden_in required when s > 0", i);
    if (r.s == 0 && !model->embed) return fail(CRF_EINVAL, "model embedding is null");
    if (r.hidden_in && !aligned16(r.hidden_in)) return fail(CRF_EINVAL, "request %d: hidden_in misaligned", i);
    if (r.hidden_out)
      for (int j = 0; j < r.e - r.s; ++j)
        if (!r.hidden_out[j] || !aligned16(r.hidden_out[j]))
          return fail(CRF_EINVAL, "request %d: hidden_out[%d] null or misaligned", i, j);
    const int l_end = r.final_hidden_out ? D.N : r.e;
    crf_status s = check_model_layers(model, r.s, l_end, D);
    if (s != CRF_OK) return s;
    s = check_adapter_layers(cur, r.s, l_end);
    if (s != CRF_OK) return s;
    for (int l = r.s; l < l_end; ++l)
      if (!pool->k_pages[l] || !pool->v_pages[l] || !aligned16(pool->k_pages[l]) ||
          !aligned16(pool->v_pages[l]))
        return fail(CRF_EINVAL, "kv pool layer %d null or misaligned", l);
  }
  (void)ctx;
  return CRF_OK;
}

// Workspace of one generation step: the decode-row scratch, the rows' RoPE angles, the final
// normalised rows and (when the caller passes no buffer) the logits.
struct StepPlan {
  Plan p;
  size_t off_angles, off_norm, off_logits, total;
};  // p.off_abort / p.off_ptab / p.ptab_slots: the page check of the rows' tables

StepPlan make_step_plan(const Dims& D, const crf_decode_row* rows, int n) {
  StepPlan sp;
  Plan& p = sp.p;
  p.dec_rows = n;
  p.max_n = 1;
  for (int i = 0; i < n; ++i) p.max_n = std::max(p.max_n, rows[i].pos + 1);
  p.splits = dec_splits(p.max_n);
  const size_t dec_row = static_cast<size_t>(3 * D.h + 2 * D.qd + 2 * D.kvd + 7 * kRankPad + 3 * D.f + norm_up_slices(D.h)) * 4 +
                         static_cast<size_t>(D.hq) * p.splits * (D.d + 2) * 4;
  p.dec_bytes = align256(dec_row * std::max(1, n));
  size_t o = 0;
  auto take = [&](size_t bytes) {
    const size_t at = o;
    o = align256(o + bytes);
    return at;
  };
  p.off_dec = take(p.dec_bytes);
  p.off_rope = 0;
  sp.off_angles = take(static_cast<size_t>(n) * (D.d / 2) * sizeof(float2));
  sp.off_norm = take(static_cast<size_t>(n) * D.h * 4);
  sp.off_logits = take(static_cast<size_t>(n) * D.V * 4);
  long ids = 0;
  for (int i = 0; i < n; ++i) ids += rows[i].pos / kPage + 1;
  p.ptab_slots = ptab_slots_for(ids);
  p.off_abort = take((1 + p.flag_words) * sizeof(int));
  p.off_ptab = take(static_cast<size_t>(p.ptab_slots) * sizeof(int));
  sp.total = p.total = o;
  return sp;
}

crf_status validate_decode_rows(const crf_kv_pool* pool, const crf_decode_row* rows, int n) {
  if (n < 1 || n > CRF_MAX_REQUESTS) return fail(CRF_EINVAL, "n_rows %d outside [1, %d]", n, CRF_MAX_REQUESTS);
  if (!pool || !pool->k_pages || !pool->v_pages || pool->num_pages < 1) return fail(CRF_EINVAL, "kv pool missing");
  for (int i = 0; i < n; ++i) {
    const crf_decode_row& r = rows[i];
    if (r.pos < 0) return fail(CRF_EINVAL, "row %d: negative position", i);
    if (!r.page_table || !r.token) return fail(CRF_EINVAL, "row %d: page_table or token is null", i);
  }
  return CRF_OK;
}

}  // namespace

namespace crf {
// Records `msg` as this thread's crf_last_error() text (used by other translation units).
void set_last_error(const char* msg) { g_err = msg ? msg : ""; }
}  // namespace crf

// ====================================================================== ABI
extern "C" {

const char* crf_last_error(void) { return g_err.c_str(); }

crf_status crf_create(crf_ctx** out, int device) {
  if (!out) return fail(CRF_EINVAL, "out is null");
  *out = nullptr;
  int count = 0;
  CRF_CUDA(cudaGetDeviceCount(&count));
  if (device < 0 || device >= count) return fail(CRF_EINVAL, "device %d out of range", device);
  CRF_CUDA(cudaSetDevice(device));
  cudaDeviceProp prop;
  CRF_CUDA(cudaGetDeviceProperties(&prop, device));
  if (prop.major != 10 || prop.minor != 3)
    return fail(CRF_EUNSUPPORTED, "device is sm_%d%d; this library is built for sm_103a", prop.major,
                prop.minor);
  crf_ctx* c = new crf_ctx;
  c->device = device;
  c->num_sms = prop.multiProcessorCount;
  c->status_dev = nullptr;
  cudaError_t e = cudaMalloc(&c->status_dev, sizeof(int));
  if (e == cudaSuccess) e = cudaMemset(c->status_dev, 0, sizeof(int));
  if (e != cudaSuccess) {
    if (c->status_dev) cudaFree(c->status_dev);
    delete c;
    return fail(CRF_ECUDA, "status word: %s", cudaGetErrorString(e));
  }
  *out = c;
  return CRF_OK;
}

crf_status crf_destroy(crf_ctx* ctx) {
  if (!ctx) return fail(CRF_EINVAL, "ctx is null");
  for (cudaEvent_t e : ctx->ev) cudaEventDestroy(e);
  cudaFree(ctx->status_dev);
  delete ctx;
  return CRF_OK;
}

crf_status crf_check(crf_ctx* ctx, void* stream) {
  if (!ctx) return fail(CRF_EINVAL, "ctx is null");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  CRF_CUDA(cudaStreamSynchronize(st));
  int status = 0;
  CRF_CUDA(cudaMemcpy(&status, ctx->status_dev, sizeof(int), cudaMemcpyDeviceToHost));
  if (status) {
    CRF_CUDA(cudaMemset(ctx->status_dev, 0, sizeof(int)));
    if (status & kStatusPages)
      return fail(CRF_EINVAL, "a page table held an id outside the pool or a page twice; that call wrote "
                  "nothing outside its workspace (status 0x%x)", status);
    if (status & kStatusBounds)
      return fail(CRF_EINVAL, "a device-side bounds check failed: a token id outside the vocabulary%s "
                  "(status 0x%x)", kDebugBuild ? " or a page id outside the pool" : "", status);
    return fail(CRF_ETIMEOUT, "a kernel abandoned a bounded wait (status 0x%x)", status);
  }
  return CRF_OK;
}

crf_status crf_selftest_timeout(crf_ctx* ctx, void* stream) {
  if (!ctx) return fail(CRF_EINVAL, "ctx is null");
  CRF_CUDA(cudaSetDevice(ctx->device));
  CRF_CUDA(launch_wait_selftest(ctx->status_dev, static_cast<cudaStream_t>(stream)));
  return CRF_OK;
}

crf_status crf_workspace_size(crf_ctx* ctx, const crf_model* model, const crf_lora_dims* lora,
                              const crf_request* reqs, int n_req, size_t* bytes) {
  if (!ctx || !model || !lora || !reqs || !bytes) return fail(CRF_EINVAL, "null argument");
  crf_status s = check_dims(model->dims);
  if (s != CRF_OK) return s;
  s = check_lora(*lora);
  if (s != CRF_OK) return s;
  if (n_req < 1 || n_req > CRF_MAX_REQUESTS) return fail(CRF_EINVAL, "n_req out of range");
  const Dims D = dims_of(model->dims);
  for (int i = 0; i < n_req; ++i)
    if (reqs[i].n_tokens < 1 || reqs[i].s < 0 || reqs[i].s > reqs[i].e || reqs[i].e > D.N)
      return fail(CRF_EINVAL, "request %d malformed", i);
  *bytes = make_plan(D, reqs, n_req).total;
  return CRF_OK;
}

crf_status crf_recompute_window(crf_ctx* ctx, const crf_model* model, const crf_adapter* cur,
                                const crf_kv_pool* pool, const crf_request* reqs, int n_req,
                                void* workspace, size_t ws_bytes, void* stream) {
  if (!ctx || !model || !cur || !pool || !reqs) return fail(CRF_EINVAL, "null argument");
  if (!model->layers) return fail(CRF_EINVAL, "model layers missing");
  if (!cur->A || !cur->B) return fail(CRF_EINVAL, "adapter tables missing");
  crf_status s = check_dims(model->dims);
  if (s != CRF_OK) return s;
  s = check_lora(cur->dims);
  if (s != CRF_OK) return s;
  CRF_CUDA(cudaSetDevice(ctx->device));
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const Dims D = dims_of(model->dims);
  s = validate_requests(ctx, model, cur, pool, reqs, n_req, D);
  if (s != CRF_OK) return s;
  const Plan plan = make_plan(D, reqs, n_req);
  if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 255))
    return fail(CRF_EINVAL, "workspace null or not 256-byte aligned");
  if (ws_bytes < plan.total)
    return fail(CRF_ENOMEM, "workspace %zu bytes, %zu needed", ws_bytes, plan.total);

  uint8_t* ws = static_cast<uint8_t*>(workspace);
  LayerCtx c;
  c.D = &D;
  c.ctx = ctx;
  c.model = model;
  c.ad = cur;
  c.pool = pool;
  c.st = st;
  c.ws = ws;
  c.plan = &plan;
  c.scale = cur->dims.alpha / cur->dims.rank;
  c.abort = reinterpret_cast<const int*>(ws + plan.off_abort);
  {
    PageCheck pc{};
    pc.n = n_req;
    pc.first[0] = 0;
    for (int i = 0; i < n_req; ++i) {
      pc.pt[i] = reqs[i].page_table;
      pc.first[i + 1] = pc.first[i] + (reqs[i].n_tokens + kPage - 1) / kPage;
    }
    s = open_call(ctx, pc, pool->num_pages, ws, plan.off_abort, plan.flag_words, plan.off_ptab,
                  plan.ptab_slots, st);
    if (s != CRF_OK) return s;
  }

  {
    ProfScope ps(ctx, kPRope, st);
    CRF_CUDA(launch_rope_table(reinterpret_cast<float2*>(ws + plan.off_rope), plan.max_n, D.d, D.theta, st));
  }

  __nv_bfloat16* G[2] = {reinterpret_cast<__nv_bfloat16*>(ws + plan.off_g0),
                         reinterpret_cast<__nv_bfloat16*>(ws + plan.off_g1)};
  auto* dx0 = reinterpret_cast<__nv_bfloat16*>(ws + plan.off_dx0);
  const size_t row_bytes = static_cast<size_t>(D.h) * 2;
  std::vector<const __nv_bfloat16*> curp(n_req, nullptr);  // current hidden rows per request
  for (int i = 0; i < n_req; ++i)
    if (reqs[i].s > 0) curp[i] = static_cast<const __nv_bfloat16*>(reqs[i].hidden_in);

  int lmin = D.N, lmax = 0;
  for (int i = 0; i < n_req; ++i)
    if (reqs[i].s < reqs[i].e) {
      lmin = std::min(lmin, reqs[i].s);
      lmax = std::max(lmax, reqs[i].e);
    }
  int layer_seq = 0;  // layers run so far: each owns a slice of the ready words
  for (int l = lmin; l < lmax; ++l) {
    std::vector<int> act;
    for (int i = 0; i < n_req; ++i)
      if (reqs[i].s <= l && l < reqs[i].e) act.push_back(i);
    if (act.empty()) continue;
    ReqTable rt;
    std::memset(&rt, 0, sizeof(rt));
    rt.num_pages = pool->num_pages;
    int M = 0;
    for (int i : act) {
      rt.row0[rt.n] = M;
      rt.len[rt.n] = reqs[i].n_tokens;
      rt.page_table[rt.n] = reqs[i].page_table;
      ++rt.n;
      M += reqs[i].n_tokens;
    }
    const bool single = act.size() == 1;
    const int i0 = act[0];
    // input rows
    const __nv_bfloat16* X_in = nullptr;
    int in_buf = -1;
    if (single && curp[i0] && !(reqs[i0].s == l && l == 0)) {
      X_in = curp[i0];
    } else {
      // in place already?
      for (int b = 0; b < 2 && !X_in; ++b) {
        bool all = true;
        for (int k = 0; k < rt.n; ++k)
          all &= curp[act[k]] == G[b] + static_cast<size_t>(rt.row0[k]) * D.h;
        if (all) {
          X_in = G[b];
          in_buf = b;
        }
      }
      if (!X_in) {
        // gather into the buffer not holding any current rows
        int b = 0;
        for (int k = 0; k < rt.n; ++k) {
          const auto* cp = curp[act[k]];
          if (cp >= G[0] && cp < G[0] + static_cast<size_t>(plan.M) * D.h) b = 1;
        }
        for (int k = 0; k < rt.n; ++k) {
          const int i = act[k];
          __nv_bfloat16* dst = G[b] + static_cast<size_t>(rt.row0[k]) * D.h;
          if (reqs[i].s == l && l == 0) {
            ProfScope ps(ctx, kPEmbed, st);
            CRF_CUDA(launch_embed(static_cast<const __nv_bfloat16*>(model->embed), reqs[i].tokens, dst,
                                  reqs[i].n_tokens, D.h, D.V, ctx->status_dev, st));
          } else {
            ProfScope ps(ctx, kPCopy, st, 0);
            CRF_CUDA(cudaMemcpyAsync(dst, curp[i], reqs[i].n_tokens * row_bytes,
                                     cudaMemcpyDeviceToDevice, st));
          }
        }
        X_in = G[b];
        in_buf = b;
      }
    }
    // output rows
    __nv_bfloat16* X_out;
    if (single && reqs[i0].hidden_out) {
      X_out = static_cast<__nv_bfloat16*>(reqs[i0].hidden_out[l - reqs[i0].s]);
    } else {
      int b = in_buf >= 0 ? 1 - in_buf : 0;
      X_out = G[b];
    }
    c.xa_flags = reinterpret_cast<int*>(ws + plan.off_abort) + 1 +
                 static_cast<size_t>(layer_seq++) * 4 * ((plan.M + 255) / 256);
    s = run_layer(c, l, X_in, X_out, M, rt);
    if (s != CRF_OK) return s;
    for (int k = 0; k < rt.n; ++k) {
      const int i = act[k];
      const bool copy_out = !single && reqs[i].hidden_out;
      ProfScope ps(ctx, kPCopy, st, copy_out ? 1 : 0);
      curp[i] = X_out + static_cast<size_t>(rt.row0[k]) * D.h;
      if (copy_out)
        CRF_CUDA(launch_copy_bf16(static_cast<__nv_bfloat16*>(reqs[i].hidden_out[l - reqs[i].s]), curp[i],
                                  static_cast<size_t>(reqs[i].n_tokens) * D.h, c.abort, st));
      if (l == reqs[i].e - 1 && reqs[i].final_hidden_out)
        CRF_CUDA(cudaMemcpyAsync(dx0 + static_cast<size_t>(i) * D.h,
                                 curp[i] + static_cast<size_t>(reqs[i].n_tokens - 1) * D.h, row_bytes,
                                 cudaMemcpyDeviceToDevice, st));
    }
  }

  // first-step state: the last prefix row through layers e..N-1 on the historical cache
  std::vector<DecodeRow> dec;
  for (int i = 0; i < n_req; ++i) {
    const crf_request& r = reqs[i];
    if (!r.final_hidden_out) continue;
    __nv_bfloat16* start = dx0 + static_cast<size_t>(i) * D.h;
    if (r.s == r.e) {
      ProfScope ps(ctx, r.s == 0 ? kPEmbed : kPCopy, st, r.s == 0 ? 1 : 0);
      if (r.s == 0) {
        CRF_CUDA(launch_embed(static_cast<const __nv_bfloat16*>(model->embed), r.tokens + (r.n_tokens - 1),
                              start, 1, D.h, D.V, ctx->status_dev, st));
      } else {
        CRF_CUDA(cudaMemcpyAsync(start,
                                 static_cast<const __nv_bfloat16*>(r.hidden_in) +
                                     static_cast<size_t>(r.n_tokens - 1) * D.h,
                                 row_bytes, cudaMemcpyDeviceToDevice, st));
      }
    }
    if (r.e == D.N) {
      ProfScope ps(ctx, kPCopy, st, 1);
      CRF_CUDA(launch_copy_bf16(static_cast<__nv_bfloat16*>(r.final_hidden_out), start, D.h, c.abort, st));
    } else {
      dec.push_back({r.e, r.n_tokens - 1, r.page_table, start, r.final_hidden_out});
    }
  }
  s = decode_rows(c, dec);
  if (s != CRF_OK) return s;
  CRF_CUDA(cudaGetLastError());
  return CRF_OK;
}

crf_status crf_decode_workspace_size(crf_ctx* ctx, const crf_model* model, const crf_lora_dims* lora,
                                     const crf_decode_row* rows, int n_rows, size_t* bytes) {
  if (!ctx || !model || !lora || !rows || !bytes) return fail(CRF_EINVAL, "null argument");
  crf_status s = check_dims(model->dims);
  if (s != CRF_OK) return s;
  s = check_lora(*lora);
  if (s != CRF_OK) return s;
  if (n_rows < 1 || n_rows > CRF_MAX_REQUESTS) return fail(CRF_EINVAL, "n_rows out of range");
  for (int i = 0; i < n_rows; ++i)
    if (rows[i].pos < 0) return fail(CRF_EINVAL, "row %d: negative position", i);
  *bytes = make_step_plan(dims_of(model->dims), rows, n_rows).total;
  return CRF_OK;
}

crf_status crf_decode_step(crf_ctx* ctx, const crf_model* model, const crf_adapter* cur,
                           const crf_kv_pool* pool, const crf_decode_row* rows, int n_rows,
                           int32_t* next_tokens, float* logits, void* workspace, size_t ws_bytes,
                           void* stream) {
  if (!ctx || !model || !cur || !pool || !rows || !next_tokens) return fail(CRF_EINVAL, "null argument");
  if (!model->layers) return fail(CRF_EINVAL, "model layers missing");
  if (!model->embed || !model->final_norm || !model->lm_head)
    return fail(CRF_EINVAL, "model embedding, final norm or LM head is null");
  if (!cur->A || !cur->B) return fail(CRF_EINVAL, "adapter tables missing");
  crf_status s = check_dims(model->dims);
  if (s != CRF_OK) return s;
  s = check_lora(cur->dims);
  if (s != CRF_OK) return s;
  CRF_CUDA(cudaSetDevice(ctx->device));
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const Dims D = dims_of(model->dims);
  s = check_model_layers(model, 0, D.N, D);
  if (s != CRF_OK) return s;
  s = check_adapter_layers(cur, 0, D.N);
  if (s != CRF_OK) return s;
  for (int l = 0; l < D.N; ++l)
    if (!pool || !pool->k_pages || !pool->v_pages || !pool->k_pages[l] || !pool->v_pages[l] ||
        !aligned16(pool->k_pages[l]) || !aligned16(pool->v_pages[l]))
      return fail(CRF_EINVAL, "kv pool layer %d null or misaligned", l);
  s = validate_decode_rows(pool, rows, n_rows);
  if (s != CRF_OK) return s;
  const StepPlan sp = make_step_plan(D, rows, n_rows);
  if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 255))
    return fail(CRF_EINVAL, "workspace null or not 256-byte aligned");
  if (ws_bytes < sp.total) return fail(CRF_ENOMEM, "workspace %zu bytes, %zu needed", ws_bytes, sp.total);

  uint8_t* ws = static_cast<uint8_t*>(workspace);
  LayerCtx c;
  c.D = &D;
  c.ctx = ctx;
  c.model = model;
  c.ad = cur;
  c.pool = pool;
  c.st = st;
  c.ws = ws;
  c.plan = &sp.p;
  c.scale = cur->dims.alpha / cur->dims.rank;
  c.abort = reinterpret_cast<const int*>(ws + sp.p.off_abort);
  {
    PageCheck pc{};
    pc.n = n_rows;
    pc.first[0] = 0;
    for (int i = 0; i < n_rows; ++i) {
      pc.pt[i] = rows[i].page_table;
      pc.first[i + 1] = pc.first[i] + rows[i].pos / kPage + 1;
    }
    s = open_call(ctx, pc, pool->num_pages, ws, sp.p.off_abort, sp.p.flag_words, sp.p.off_ptab, sp.p.ptab_slots,
                  st);
    if (s != CRF_OK) return s;
  }
  RowPositions rp{};
  std::vector<DecodeRow> dec;
  for (int i = 0; i < n_rows; ++i) {
    rp.pos[i] = rows[i].pos;
    DecodeRow d{};
    d.e = 0;
    d.pos = rows[i].pos;
    d.page_table = rows[i].page_table;
    d.token = rows[i].token;
    dec.push_back(d);
  }
  auto* angles = reinterpret_cast<float2*>(ws + sp.off_angles);
  {
    ProfScope ps(ctx, kPRope, st);
    CRF_CUDA(launch_rope_table_rows(angles, rp, n_rows, D.d, D.theta, st));
  }
  DecodeOpts opt;
  opt.write_kv = true;
  opt.rope_by_row = angles;
  s = decode_rows(c, dec, opt);
  if (s != CRF_OK) return s;
  // final norm, LM head, greedy token: the fp32 rows are the head of the decode scratch
  float* x = reinterpret_cast<float*>(ws + sp.p.off_dec);
  float* hn = reinterpret_cast<float*>(ws + sp.off_norm);
  float* z = logits ? logits : reinterpret_cast<float*>(ws + sp.off_logits);
  {
    ProfScope ps(ctx, kPLmHead, st, 3);
    CRF_CUDA(launch_rmsnorm_f32(x, static_cast<const __nv_bfloat16*>(model->final_norm), hn, n_rows, D.h, D.eps, st));
    CRF_CUDA(launch_lm_head(static_cast<const __nv_bfloat16*>(model->lm_head), hn, n_rows, D.V, D.h, z,
                            ctx->num_sms, st, c.abort));
    CRF_CUDA(launch_argmax_rows(z, n_rows, D.V, next_tokens, st, c.abort));
  }
  return CRF_OK;
}

crf_status crf_drift_workspace_size(crf_ctx* ctx, const crf_model_dims* dims,
                                    const crf_lora_dims* lora, size_t* bytes) {
  if (!ctx || !dims || !lora || !bytes) return fail(CRF_EINVAL, "null argument");
  crf_status s = check_lora(*lora);
  if (s != CRF_OK) return s;
  if (dims->n_layers < 1) return fail(CRF_EINVAL, "n_layers must be positive");
  int nm = 0;
  for (int m = 0; m < 7; ++m) nm += (lora->module_mask >> m) & 1;
  *bytes = align256(drift_workspace_bytes(ctx->num_sms, lora->rank, dims->n_layers * nm));
  return CRF_OK;
}

crf_status crf_drift(crf_ctx* ctx, const crf_model_dims* dims, const crf_adapter* cur,
                     const crf_adapter* const* anchors, float* out_sq, void* workspace,
                     size_t ws_bytes, void* stream) {
  if (!ctx || !dims || !cur || !anchors || !out_sq) return fail(CRF_EINVAL, "null argument");
  if (dims->n_layers < 1) return fail(CRF_EINVAL, "n_layers must be positive");
  crf_status s = check_lora(cur->dims);
  if (s != CRF_OK) return s;
  if (!cur->A || !cur->B) return fail(CRF_EINVAL, "adapter tables missing");
  const Dims D = dims_of(*dims);
  if (D.h % 8 || D.f % 8 || D.qd % 8 || D.kvd % 8)
    return fail(CRF_EUNSUPPORTED, "drift needs every projection's widths to be multiples of 8");
  std::vector<DriftItem> items;
  for (int l = 0; l < D.N; ++l) {
    const crf_adapter* an = anchors[l];
    if (!an || !an->A || !an->B) return fail(CRF_EINVAL, "anchor %d missing", l);
    if (an->dims.rank != cur->dims.rank || an->dims.module_mask != cur->dims.module_mask)
      return fail(CRF_ESHAPE, "anchor %d has different LoRA dims", l);
    for (int m = 0; m < 7; ++m) {
      if (!adapted(cur, m)) continue;
      DriftItem it;
      it.A0 = static_cast<const __nv_bfloat16*>(an->A[l * 7 + m]);
      it.B0 = static_cast<const __nv_bfloat16*>(an->B[l * 7 + m]);
      it.A1 = static_cast<const __nv_bfloat16*>(cur->A[l * 7 + m]);
      it.B1 = static_cast<const __nv_bfloat16*>(cur->B[l * 7 + m]);
      if (!it.A0 || !it.B0 || !it.A1 || !it.B1)
        return fail(CRF_EINVAL, "layer %d module %d factor is null", l, m);
      if (!aligned16(it.A0) || !aligned16(it.B0) || !aligned16(it.A1) || !aligned16(it.B1))
        return fail(CRF_EINVAL, "layer %d module %d factor misaligned (16 bytes)", l, m);
      module_shape(D, m, it.out_dim, it.in_dim);
      it.out_index = l * 7 + m;
      items.push_back(it);
    }
  }
  size_t need = 0;
  s = crf_drift_workspace_size(ctx, dims, &cur->dims, &need);
  if (s != CRF_OK) return s;
  if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 255) || ws_bytes < need)
    return fail(CRF_ENOMEM, "drift workspace null, misaligned or %zu < %zu bytes", ws_bytes, need);
  CRF_CUDA(cudaSetDevice(ctx->device));
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (items.empty()) {
    CRF_CUDA(cudaMemsetAsync(out_sq, 0, static_cast<size_t>(D.N) * 7 * 2 * sizeof(float), st));
    return CRF_OK;
  }
  ProfScope ps(ctx, kPDrift, st, drift_launches(static_cast<int>(items.size())));
  CRF_CUDA(launch_drift(items.data(), static_cast<int>(items.size()), cur->dims.rank, D.N * 7,
                        static_cast<int>(cur->dims.module_mask), workspace, ctx->num_sms, out_sq,
                        ctx->status_dev, st));
  return CRF_OK;
}

// ---------------------------------------------------------------- KL
static int kl_splits(const crf_ctx* ctx, int n_rows, int vocab) {
  return kl_split_count(ctx->num_sms, n_rows, vocab);
}

crf_status crf_kl_workspace_size(crf_ctx* ctx, int n_rows, int vocab, int hidden, size_t* bytes) {
  if (!ctx || !bytes || n_rows < 1 || vocab < 1 || hidden < 0)
    return fail(CRF_EINVAL, "bad argument");
  const int sp = kl_splits(ctx, n_rows, vocab);
  size_t o = align256(static_cast<size_t>(n_rows) * sp * 5 * sizeof(float));
  if (hidden > 0) {
    o += align256(static_cast<size_t>(2 * n_rows) * hidden * sizeof(float)) * 2;
    o += align256(static_cast<size_t>(2 * n_rows) * vocab * sizeof(float));
  }
  *bytes = o;
  return CRF_OK;
}

crf_status crf_kl(crf_ctx* ctx, const crf_model* model, const void* ref, const void* cur,
                  int n_rows, int vocab, float* out_kl, float* logits_out, void* workspace,
                  size_t ws_bytes, void* stream) {
  if (!ctx || !ref || !cur || !out_kl) return fail(CRF_EINVAL, "null argument");
  if (n_rows < 1 || vocab < 1) return fail(CRF_EINVAL, "n_rows and vocab must be positive");
  const int hidden = model ? model->dims.hidden : 0;
  if (model) {
    if (model->dims.vocab != vocab) return fail(CRF_ESHAPE, "vocab %d != model vocab %d", vocab, model->dims.vocab);
    if (!model->lm_head || !model->final_norm) return fail(CRF_EINVAL, "model LM head or final norm is null");
    if (hidden < 1 || hidden % 8) return fail(CRF_EUNSUPPORTED, "hidden must be a positive multiple of 8");
  }
  size_t need = 0;
  crf_status s = crf_kl_workspace_size(ctx, n_rows, vocab, hidden, &need);
  if (s != CRF_OK) return s;
  if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 255) || ws_bytes < need)
    return fail(CRF_ENOMEM, "KL workspace null, misaligned or %zu < %zu", ws_bytes, need);
  CRF_CUDA(cudaSetDevice(ctx->device));
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  const int sp = kl_splits(ctx, n_rows, vocab);
  float* part = reinterpret_cast<float*>(ws);
  size_t o = align256(static_cast<size_t>(n_rows) * sp * 5 * sizeof(float));
  const float* zr = static_cast<const float*>(ref);
  const float* zc = static_cast<const float*>(cur);
  if (model) {
    float* hf = reinterpret_cast<float*>(ws + o);
    o += align256(static_cast<size_t>(2 * n_rows) * hidden * sizeof(float));
    float* hn = reinterpret_cast<float*>(ws + o);
    o += align256(static_cast<size_t>(2 * n_rows) * hidden * sizeof(float));
    float* logits = logits_out ? logits_out : reinterpret_cast<float*>(ws + o);
    ProfScope ps(ctx, kPLmHead, st, 4);
    CRF_CUDA(launch_bf16_to_f32(static_cast<const __nv_bfloat16*>(ref), hf, n_rows * hidden, st));
    CRF_CUDA(launch_bf16_to_f32(static_cast<const __nv_bfloat16*>(cur), hf + static_cast<size_t>(n_rows) * hidden,
                                n_rows * hidden, st));
    CRF_CUDA(launch_rmsnorm_f32(hf, static_cast<const __nv_bfloat16*>(model->final_norm), hn, 2 * n_rows,
                                hidden, model->dims.rms_eps, st));
    CRF_CUDA(launch_lm_head(static_cast<const __nv_bfloat16*>(model->lm_head), hn, 2 * n_rows, vocab,
                            hidden, logits, ctx->num_sms, st));
    zr = logits;
    zc = logits + static_cast<size_t>(n_rows) * vocab;
  }
  {
    ProfScope ps(ctx, kPKl, st, 2);
    CRF_CUDA(launch_kl(zr, zc, n_rows, vocab, out_kl, part, sp, st));
  }
  return CRF_OK;
}

// ---------------------------------------------------------------- profiling
crf_status crf_profile_enable(crf_ctx* ctx, int on, int max_launches) {
  if (!ctx) return fail(CRF_EINVAL, "ctx is null");
  if (on && max_launches < 1) return fail(CRF_EINVAL, "max_launches must be positive");
  CRF_CUDA(cudaSetDevice(ctx->device));
  if (on) {
    const size_t want = static_cast<size_t>(2) * max_launches;
    while (ctx->ev.size() < want) {
      cudaEvent_t e;
      CRF_CUDA(cudaEventCreate(&e));
      ctx->ev.push_back(e);
    }
  }
  ctx->prof_on = on != 0;
  ctx->ev_used = 0;
  ctx->rec.clear();
  ctx->dropped = 0;
  return CRF_OK;
}

crf_status crf_profile_read(crf_ctx* ctx, int max_kinds, char* names, double* total_ms,
                            int* launches, int* n_kinds, int* dropped) {
  if (!ctx || !names || !total_ms || !launches || !n_kinds) return fail(CRF_EINVAL, "null argument");
  double ms[kPNumKinds] = {0};
  int cnt[kPNumKinds] = {0};
  bool seen[kPNumKinds] = {false};
  for (const auto& r : ctx->rec) {
    CRF_CUDA(cudaEventSynchronize(ctx->ev[r.idx + 1]));
    float t = 0.f;
    CRF_CUDA(cudaEventElapsedTime(&t, ctx->ev[r.idx], ctx->ev[r.idx + 1]));
    ms[r.kind] += t;
    cnt[r.kind] += r.kernels;
    seen[r.kind] = true;
  }
  int k = 0;
  for (int i = 0; i < kPNumKinds && k < max_kinds; ++i) {
    if (!seen[i]) continue;
    std::snprintf(names + 32 * k, 32, "%s", kProfNames[i]);
    total_ms[k] = ms[i];
    launches[k] = cnt[i];
    ++k;
  }
  *n_kinds = k;
  if (dropped) *dropped = ctx->dropped;
  ctx->ev_used = 0;
  ctx->rec.clear();
  ctx->dropped = 0;
  return CRF_OK;
}

}  // extern "C"
