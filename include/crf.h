/*
 * crf.h -- C ABI of the GB300 bounded KV-cache recomputation library
 * (CacheReforge, arXiv 2609.30884).
 *
 * The library executes the data-parallel hot path of stale-KV-cache recovery
 * under an evolving LoRA adapter:
 *
 *   crf_recompute_window  Section 4.2 "Executable restart": feed the retained
 *                         boundary state H_{s-1} (the token embedding when
 *                         s = 0; H_{-1} in Section S1.1) to layers s..e-1 over
 *                         the complete prefix under the current adapter, and
 *                         overwrite exactly those layers' K/V (Eq. 1 cache,
 *                         Eq. S1 per-layer maps F_l / G_l, Eq. S3 projections).
 *                         Optionally continues the last prefix row through
 *                         layers e..N-1 against the historical cache, which
 *                         gives the first-step next-token state used for
 *                         fidelity (Section 3.1, Section S2.1).
 *   crf_drift             Eq. 8: per (layer, module) squared displacement of
 *                         the current adapter from each layer's anchor.
 *   crf_kl                Section S2.1: forward KL(p* || p) at the first
 *                         generated-token step, fresh logits as reference.
 *   crf_decode_step       one generated token per request on the recovered
 *                         (mixed-version) paged cache: the step that consumes
 *                         the refreshed cache (Section 3.1, first generated
 *                         tokens); greedy next token and optional logits.
 *
 * Conventions (every entry point):
 *   - Device pointers are CUDA device memory on the context's device; host
 *     arrays (the per-layer pointer tables) are read during the call only.
 *     The caller owns every buffer. The library keeps no pointer after it
 *     returns and allocates no device memory inside these calls: temporaries
 *     live in the caller's workspace (see crf_workspace_size).
 *   - `stream` is a cudaStream_t (NULL = legacy default stream). Work is
 *     enqueued on it; results are valid once the stream has synchronised.
 *   - Every argument the host can see is validated before anything is
 *     launched. A non-OK status from that validation (CRF_EINVAL,
 *     CRF_ESHAPE, CRF_EUNSUPPORTED, CRF_ENOMEM) means nothing was enqueued
 *     and nothing was written. A CRF_ECUDA from a failed launch can leave the
 *     call's earlier kernels enqueued; their outputs are then undefined.
 *     crf_last_error() returns a message in either case (thread-local).
 *   - Page tables live in device memory and the host never reads them: no
 *     call waits on its stream (crf_check alone synchronises). The first
 *     kernel of crf_recompute_window and crf_decode_step checks every page
 *     id (inside [0, num_pages), no page twice across the call's tables);
 *     a failure makes every later kernel of that call return at once, so the
 *     call writes nothing outside its workspace (pool pages, checkpoints,
 *     final rows, logits, tokens), and the next crf_check returns CRF_EINVAL.
 *   - A context is used by one host thread at a time: its device status word
 *     and timing state are shared by its calls. Separate contexts may run
 *     concurrently.
 *   - A kernel that gives up on a bounded internal wait records it in the
 *     context; crf_check() reports it as CRF_ETIMEOUT. An asynchronous CUDA
 *     error is reported as CRF_ECUDA by the next call.
 *   - Ids read from device memory are checked where they are used. A token id
 *     outside [0, vocab) is read as token 0 and recorded; crf_check() then
 *     returns CRF_EINVAL. A library built with CRF_DEBUG defined
 *     (libcrf_debug.so) also checks every page id again at each device-side
 *     use, reads or writes page 0 in place of a bad id and records it the
 *     same way.
 *   - Tensors are row-major, bf16 unless stated. Weights are [out, in].
 */
#ifndef CRF_H
#define CRF_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define CRF_API __attribute__((visibility("default")))
#else
#define CRF_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum crf_status {
  CRF_OK = 0,
  CRF_EINVAL = 1,        /* bad argument (null pointer, window out of range, ...) */
  CRF_ESHAPE = 2,        /* shapes inconsistent with each other or with the buffers */
  CRF_EUNSUPPORTED = 3,  /* valid but not implemented (head_dim, rank, alignment, ...) */
  CRF_ENOMEM = 4,        /* workspace too small */
  CRF_ECUDA = 5,         /* CUDA runtime / driver error */
  CRF_ETIMEOUT = 6       /* a kernel abandoned a bounded wait */
} crf_status;

/* Projection index order used by every per-module table. */
enum {
  CRF_MOD_Q = 0, CRF_MOD_K = 1, CRF_MOD_V = 2, CRF_MOD_O = 3,
  CRF_MOD_GATE = 4, CRF_MOD_UP = 5, CRF_MOD_DOWN = 6, CRF_NUM_MODULES = 7
};

#define CRF_PAGE_SIZE 16   /* tokens per KV page */
#define CRF_MAX_REQUESTS 32

/* Decoder shape (Qwen2.5 family, Section 5.1): pre-norm RMSNorm, rotate-half
 * RoPE, grouped-query causal attention, SwiGLU MLP. head_dim must be 64 or
 * 128; n_q_heads a multiple of n_kv_heads. */
typedef struct crf_model_dims {
  int n_layers, hidden, n_q_heads, n_kv_heads, head_dim, ffn, vocab;
  float rms_eps, rope_theta;
  int qkv_bias;          /* 1: q/k/v projections carry a bias */
} crf_model_dims;

/* LoRA adapter shape: every adapted module m (bit m of module_mask) uses
 * W_m + (alpha / rank) * B_m A_m, kept unmerged. rank must be 4, 8 or 16. */
typedef struct crf_lora_dims {
  int rank;
  float alpha;
  uint32_t module_mask;
} crf_lora_dims;

/* Base weights of one layer (device pointers, bf16):
 *   W[m]    [out_m, in_m]   q:[Hq*d,h] k,v:[Hkv*d,h] o:[h,Hq*d] gate,up:[f,h] down:[h,f]
 *   bias[j] [out_j] for q,k,v (j = 0..2), used iff dims.qkv_bias
 * Every W[m] and bias[j] starts on a 16-byte boundary (CRF_EINVAL otherwise).
 *   ln1/ln2 [h] RMSNorm gains before attention / before the MLP. */
typedef struct crf_layer_weights {
  const void* W[CRF_NUM_MODULES];
  const void* bias[3];
  const void* ln1;
  const void* ln2;
} crf_layer_weights;

typedef struct crf_model {
  crf_model_dims dims;
  const crf_layer_weights* layers;  /* host array [n_layers] */
  const void* embed;                /* [vocab, h]; read when a window starts at layer 0 */
  const void* final_norm;           /* [h]; read by crf_kl with a model */
  const void* lm_head;              /* [vocab, h]; read by crf_kl with a model */
} crf_model;

/* One adapter version theta_t. A/B are host arrays [n_layers * 7] of device
 * pointers, entry l*7+m: A [rank, in_m], B [out_m, rank] (bf16); NULL for
 * modules outside module_mask. */
typedef struct crf_adapter {
  crf_lora_dims dims;
  const void* const* A;
  const void* const* B;
} crf_adapter;

/* Paged KV pool shared by all requests: per layer one K and one V pool,
 * bf16 [num_pages][n_kv_heads][16][head_dim], keys stored after rotation.
 * Token t of a request lives at page page_table[t / 16], slot t % 16. */
typedef struct crf_kv_pool {
  void* const* k_pages;   /* host array [n_layers] of device pointers */
  void* const* v_pages;   /* host array [n_layers] of device pointers */
  int num_pages;
} crf_kv_pool;

/* One cached prefix to refresh over the window [s, e) (0 <= s <= e <= N).
 *   page_table        device int32 [ceil(n_tokens/16)], distinct ids < num_pages
 *   tokens            device int32 [n_tokens]; required iff s == 0; ids in [0, vocab)
 *   hidden_in         device [n_tokens, h] = H_{s-1}; required iff s > 0
 *   hidden_out        NULL, or host array [e-s] of device [n_tokens, h]
 *                     buffers receiving H_s..H_{e-1} (refreshed checkpoints)
 *   final_hidden_out  NULL, or device [h]: the last prefix row carried
 *                     through layers e..N-1 against those layers' cached K/V
 *                     (reads the pool, writes nothing to it). s == e is
 *                     allowed only with final_hidden_out (direct reuse).
 * Pages of different requests must not overlap. */
typedef struct crf_request {
  int n_tokens, s, e;
  const int32_t* page_table;
  const int32_t* tokens;
  const void* hidden_in;
  void* const* hidden_out;
  void* final_hidden_out;
} crf_request;

typedef struct crf_ctx crf_ctx;

/* Create a context bound to CUDA device `device` (allocates a small status
 * word and queries device properties). */
CRF_API crf_status crf_create(crf_ctx** out, int device);
CRF_API crf_status crf_destroy(crf_ctx* ctx);

/* Message for the last non-OK status returned on this thread. */
CRF_API const char* crf_last_error(void);

/* Synchronise `stream`, then report what the kernels recorded since the last
 * check: a rejected page table or a failed device-side bounds check
 * (CRF_EINVAL, which takes precedence) or an abandoned bounded wait
 * (CRF_ETIMEOUT); else a pending CUDA error (CRF_ECUDA). The record is
 * cleared. */
CRF_API crf_status crf_check(crf_ctx* ctx, void* stream);

/* Failure-path self-test (no counterpart in the paper): launches one block on
 * `stream` whose wait on a barrier that nothing completes runs out after the
 * library's bounded-wait limit (2 s), exactly as a stalled kernel of the hot
 * path would; the next crf_check then returns CRF_ETIMEOUT and clears the
 * report, and the context stays usable. No fault is raised on the GPU. */
CRF_API crf_status crf_selftest_timeout(crf_ctx* ctx, void* stream);

/* Workspace bytes crf_recompute_window needs for these requests. */
CRF_API crf_status crf_workspace_size(crf_ctx* ctx, const crf_model* model, const crf_lora_dims* lora,
                              const crf_request* reqs, int n_req, size_t* bytes);

/* Bounded recomputation of every request's window (Section 4.2), batched:
 * at each layer the rows of all requests whose window covers it run as one
 * set of GEMMs; attention, RoPE and the page writes are per request.
 * `workspace` is device memory of at least crf_workspace_size bytes, 256-byte
 * aligned. */
CRF_API crf_status crf_recompute_window(crf_ctx* ctx, const crf_model* model, const crf_adapter* cur,
                                const crf_kv_pool* pool, const crf_request* reqs, int n_req,
                                void* workspace, size_t ws_bytes, void* stream);

/* One generation step for each row (the decoding that consumes the recovered
 * cache, Section 2.1; the first generated token is where Section S2.1 measures
 * KL and top-1): the token at position `pos` (the number
 * of positions already cached for that request) is embedded and carried through
 * layers 0..N-1 under `cur`; at every layer it attends to the cached keys and
 * values at positions 0..pos-1 of its page table plus its own, and its post-RoPE
 * K and V are written into slot pos % 16 of page page_table[pos / 16] of that
 * layer (so the next step sees them). The final row goes through the final norm
 * and the LM head; next_tokens[i] = argmax of row i's logits (lowest index
 * among equal maxima).
 *   page_table: device int32 [pos / 16 + 1]; pages must be distinct across rows.
 *   token:      device int32, one entry: the input token id of the row, in [0, vocab).
 * next_tokens: device int32 [n_rows]. logits: NULL or device fp32 [n_rows][vocab].
 * The model needs embed, final_norm and lm_head; 1 <= n_rows <= CRF_MAX_REQUESTS.
 * `workspace` >= crf_decode_workspace_size bytes, 256-byte aligned. */
typedef struct {
  int pos;
  const int32_t* page_table;
  const int32_t* token;
} crf_decode_row;
CRF_API crf_status crf_decode_workspace_size(crf_ctx* ctx, const crf_model* model, const crf_lora_dims* lora,
                                     const crf_decode_row* rows, int n_rows, size_t* bytes);
CRF_API crf_status crf_decode_step(crf_ctx* ctx, const crf_model* model, const crf_adapter* cur,
                           const crf_kv_pool* pool, const crf_decode_row* rows, int n_rows,
                           int32_t* next_tokens, float* logits, void* workspace, size_t ws_bytes,
                           void* stream);

/* Eq. 8 drift. anchors: host array [n_layers] of adapters (anchors[l] is the
 * version that produced layer l's cache; all of the same lora dims as cur).
 * out_sq: device fp32 [n_layers][7][2]: {||B1 A1 - B0 A0||_F^2 (unscaled),
 * ||A1 - A0||_F^2 + ||B1 - B0||_F^2}, zeros for modules not in the mask.
 * Every projection width (hidden, ffn, query and key/value widths) must be a
 * multiple of 8 (CRF_EUNSUPPORTED otherwise); every factor 16-byte aligned.
 * `workspace` >= crf_drift_workspace_size bytes. */
CRF_API crf_status crf_drift_workspace_size(crf_ctx* ctx, const crf_model_dims* dims,
                                    const crf_lora_dims* lora, size_t* bytes);
CRF_API crf_status crf_drift(crf_ctx* ctx, const crf_model_dims* dims, const crf_adapter* cur,
                     const crf_adapter* const* anchors, float* out_sq, void* workspace,
                     size_t ws_bytes, void* stream);

/* Forward KL(p* || p), p* = softmax(z_ref), p = softmax(z_cur), one value per row.
 * With model == NULL, ref/cur are device fp32 logits [n_rows, vocab].
 * With a model, ref/cur are device bf16 final hidden rows [n_rows, h]; the
 * logits z = lm_head * (rmsnorm(h) * final_norm) are formed first (model->dims.vocab
 * must equal `vocab`) and, if logits_out != NULL, stored there as fp32
 * [2 * n_rows, vocab] (ref rows first). out_kl: device fp32 [n_rows].
 * `workspace` >= crf_kl_workspace_size bytes. */
CRF_API crf_status crf_kl_workspace_size(crf_ctx* ctx, int n_rows, int vocab, int hidden, size_t* bytes);
CRF_API crf_status crf_kl(crf_ctx* ctx, const crf_model* model, const void* ref, const void* cur,
                  int n_rows, int vocab, float* out_kl, float* logits_out, void* workspace,
                  size_t ws_bytes, void* stream);

/* Allocation-free first-step KL from logits (no counterpart in the paper; an
 * interface for callers that cannot allocate device memory when they need the
 * number, such as a serving loop under a fixed device-memory budget or a C
 * host without its own device allocator).
 * Same arithmetic as crf_kl with model == NULL (the same vocabulary splits,
 * reduced in the same order), but its scratch is a fixed device array inside
 * the library (160 KiB, held by every GPU that loads it until the process
 * exits) instead of a caller workspace, so the call allocates nothing.
 * z_ref, z_cur: device fp32 [n_rows, vocab]; out_kl: device fp32 [n_rows].
 * n_rows must be 1..32 (CRF_EUNSUPPORTED beyond). `device` is made current for
 * the call and restored after. The first call on a device (and the first after
 * that device's context is recreated, e.g. after cudaDeviceReset) looks up the
 * array's device address; make that first call before any stream capture.
 * All calls share the one array: calls whose kernels overlap on the GPU
 * (different streams, or different host threads) race and must be serialised
 * by the caller. */
CRF_API crf_status crf_kl_logits_noalloc(int device, const float* z_ref, const float* z_cur,
                                         int n_rows, int vocab, float* out_kl, void* stream);

/* Per-kernel timing, for measurement: while enabled, every kernel launch and
 * device copy the library issues is bracketed by CUDA events recorded on the
 * caller's stream (the events are created here, up to `max_launches` launches
 * between reads; later launches are counted as dropped).
 * crf_profile_read synchronises those events and returns, per kernel kind,
 * its name (NUL-terminated, at most 31 chars, in names[i*32]), total device
 * milliseconds and number of kernel launches; then it clears the record.
 * Kinds with no launches are omitted. *n_kinds receives the number written. */
CRF_API crf_status crf_profile_enable(crf_ctx* ctx, int on, int max_launches);
CRF_API crf_status crf_profile_read(crf_ctx* ctx, int max_kinds, char* names, double* total_ms,
                                    int* launches, int* n_kinds, int* dropped);

#ifdef __cplusplus
}
#endif
#endif /* CRF_H */
