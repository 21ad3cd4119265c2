/*
 * kvr.h -- C ABI of libkvr: KV-cache reuse attention for GB300 (sm_103a).
 *
 * Paper: "Can I Buy Your KV Cache?" (arXiv 2606.13361).  A publisher computes
 * a document's per-layer K/V once (Sec. 3.1, Algorithm 1, SaveKV); consumers
 * load that artifact and continue from it without re-running prefill (Sec. 3.2,
 * Algorithm 2, GenerateFromKV).  Because attention is causal the continuation
 * rows equal the matching rows of a prefill over prefix||suffix (Sec. 3.3,
 * Claim 1).  This library is the attention part of both paths on one GPU:
 * loading the artifact into a paged cache, the per-token QK-norm + RoPE +
 * cache append, the reuse attention for continuation/decode tokens of many
 * consumers sharing one prefix, and the full causal prefill attention that
 * reuse replaces.
 *
 * Conventions shared by every call:
 *  - Tensors are bf16, row-major, innermost dimension contiguous, 16-byte
 *    aligned: q/q_out/out [T][n_q_heads][head_dim], k/v [T][n_kv_heads][head_dim],
 *    artifact [layers][2 (K then V)][n_kv_heads][L][head_dim].
 *  - Device pointers are CUDA device addresses on the current device.  The
 *    caller owns every buffer (including the pool given to kvr_create); the
 *    library owns only its page tables and bookkeeping.
 *  - Calls taking a stream enqueue work on it and return without waiting,
 *    unless stated.  Argument, metadata and position errors are detected on
 *    the host before anything is enqueued.  Faults found by a kernel (a wait
 *    that ran past its time limit, an index out of range) are recorded in a
 *    device error word and reported by kvr_sync_status.  The library never
 *    aborts the process and never traps on the device.
 *  - A context is not thread-safe; use one per host thread or serialise.
 *  - kvr_last_error() returns a message for the last failing call on the
 *    calling thread.
 */
#ifndef KVR_H_
#define KVR_H_

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define KVR_API __attribute__((visibility("default")))
#else
#define KVR_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaStream_t; NULL selects the legacy default stream. */
typedef struct CUstream_st* kvr_stream;

typedef enum kvr_status {
  KVR_OK = 0,
  KVR_ERR_INVALID_ARG = 1,   /* null pointer, bad size, unknown handle */
  KVR_ERR_META_MISMATCH = 2, /* artifact (model id, dtype) differ from the context's
                                (Sec. 3.1: the consumer must reject mismatches;
                                Algorithm 2's assert) */
  KVR_ERR_POSITION = 3,      /* start position != cached length: the "shifted"
                                failure of Sec. 3.2 is refused, not computed */
  KVR_ERR_OOM = 4,           /* page pool, sequence slots or workspace exhausted */
  KVR_ERR_UNSUPPORTED = 5,   /* shape or option the library does not handle */
  KVR_ERR_TIMEOUT = 6,       /* a device-side wait gave up (see kvr_sync_status) */
  KVR_ERR_CUDA = 7,          /* a CUDA runtime call failed */
  KVR_ERR_DEVICE = 8         /* a device-side bounds check fired */
} kvr_status;

/* KVR_DTYPE_BF16: the cache type (the only one a context runs in).
 * KVR_DTYPE_Q8: an artifact encoding, not a cache type -- per-tensor symmetric
 * int8 codes of a bf16 cache (Sec. 5 "Quantizing the artifact"); see
 * kvr_export_kv_q8. */
enum { KVR_DTYPE_BF16 = 1, KVR_DTYPE_Q8 = 2 };
enum { KVR_PAGE_TOKENS = 128 }; /* tokens per cache page (= attention key tile) */
enum { KVR_MAX_BATCH = 512 };   /* sequences per append/attention call */

/* Model shape.  Sec. 2 "Prefill and the KV cache": per layer, K and V of shape
 * (heads, seq, head_dim).  head_dim is 64 or 128; n_q_heads is a multiple of
 * n_kv_heads with group size G = n_q_heads / n_kv_heads in {1, 2, 4, 8, 16}.
 * rope_theta and rms_eps parametrise the per-head RMSNorm and rotate-half RoPE
 * of the append step.  max_positions bounds every sequence's length. */
typedef struct kvr_model_desc {
  uint32_t layers;
  uint32_t n_q_heads;
  uint32_t n_kv_heads;
  uint32_t head_dim;
  uint32_t dtype;          /* KVR_DTYPE_BF16 */
  uint32_t max_positions;
  double rope_theta;
  double rms_eps;
  uint64_t model_id;
} kvr_model_desc;

/* Artifact metadata m = (model id, dtype, L) of Sec. 3.1 / Algorithm 1. */
typedef struct kvr_artifact_meta {
  uint64_t model_id;
  uint32_t dtype;
  uint32_t L;
} kvr_artifact_meta;

/* Attention options.  num_splits: 0 picks a split of each query block's keys
 * over several CTAs to fill the GPU (results then merged in a fixed split
 * order); 1 runs every query block's keys in one pass, in key order from key 0,
 * which makes reuse rows bitwise equal to the same rows of kvr_prefill_attn
 * (the Claim 1 check).  Values above 1 request that many splits (capped). */
typedef struct kvr_attn_opts {
  int32_t num_splits;
  int32_t reserved;
} kvr_attn_opts;

typedef struct kvr_ctx kvr_ctx;
typedef int32_t kvr_seq; /* sequence handle (>= 0) */

/* ---- sizes (pure host arithmetic, no GPU needed) ---- */

/* Bytes of an artifact of L positions: layers * 2 * n_kv_heads * L * head_dim * 2
 * (Sec. 5 "Artifact size": linear in L, 147,456 B/token for Qwen3-4B). 0 on bad desc. */
KVR_API size_t kvr_artifact_bytes(const kvr_model_desc* desc, uint32_t L);
/* Bytes of one cache page (KVR_PAGE_TOKENS positions of every layer's K and V). */
KVR_API size_t kvr_page_bytes(const kvr_model_desc* desc);
/* Bytes of an int8 (KVR_DTYPE_Q8) artifact of L positions: fp32 scales
 * [layers][2] (K then V of each layer), zero-padded to a multiple of 16 bytes,
 * then int8 codes [layers][2][n_kv_heads][L][head_dim].  0 for a bad desc. */
KVR_API size_t kvr_artifact_bytes_q8(const kvr_model_desc* desc, uint32_t L);
/* Pool bytes kvr_create needs for max_seqs sequences, n_pages pages and a
 * split-attention workspace of workspace_bytes (0 = default 256 MiB). */
KVR_API size_t kvr_pool_bytes(const kvr_model_desc* desc, uint32_t max_seqs, uint32_t n_pages,
                      size_t workspace_bytes);
KVR_API const char* kvr_status_string(kvr_status s);
KVR_API const char* kvr_last_error(void);
/* Library version, major * 10000 + minor * 100 + patch. */
KVR_API int kvr_version(void);

/* ---- context ---- */

/* Create a context on the current device over the caller's device buffer
 * `pool` (pool_bytes, 256-byte aligned, owned by the caller and kept alive
 * until kvr_destroy).  The pool holds the device page tables, a RoPE cos/sin
 * table (built on the host in fp64, stored fp32), the split workspace, the
 * area where long-context decode calls merge their cluster partials, and the
 * cache pages.  Uploads are enqueued on `stream`.  Calls on one context share
 * the workspace and the merge area: order them on the GPU (one stream, or
 * events between streams); calls that run at the same time race on them. */
KVR_API kvr_status kvr_create(const kvr_model_desc* desc, void* pool, size_t pool_bytes,
                      uint32_t max_seqs, size_t workspace_bytes, kvr_stream stream,
                      kvr_ctx** out);
KVR_API kvr_status kvr_destroy(kvr_ctx* ctx);
/* Pages still free in the pool. */
KVR_API kvr_status kvr_free_pages(const kvr_ctx* ctx, uint32_t* n_free);
/* Number of kernels this context has launched so far (append, attention,
 * split combine and page-table updates); copies are not counted. */
KVR_API kvr_status kvr_launch_count(const kvr_ctx* ctx, uint64_t* n);
/* Synchronise `stream`, then read and clear the device error word.  Returns
 * KVR_ERR_TIMEOUT or KVR_ERR_DEVICE if a kernel recorded one since the last
 * call, else KVR_OK (or KVR_ERR_CUDA). */
KVR_API kvr_status kvr_sync_status(kvr_ctx* ctx, kvr_stream stream);
/* Failure-detection self-test (no counterpart in the paper): launches one CTA
 * whose thread waits, through the same bounded mbarrier wait every kernel of
 * the library uses, on a barrier phase that nothing completes.  After the wait
 * limit (about 2 s) the kernel records a timeout in the context's error word
 * and exits normally: the GPU neither faults nor hangs, the context stays
 * usable, and the next kvr_sync_status returns KVR_ERR_TIMEOUT (clearing the
 * word).  KVR_ERR_INVALID_ARG for a null ctx. */
KVR_API kvr_status kvr_selftest_wait_timeout(kvr_ctx* ctx, kvr_stream stream);

/* ---- sequences ---- */

/* An empty sequence (length 0): the publisher's context or a fresh prefill. */
KVR_API kvr_status kvr_seq_open(kvr_ctx* ctx, kvr_seq* out);
/* A consumer of `parent`: shares its full pages read-only and copies its last
 * partial page (copy enqueued on `stream`), so the child continues at position
 * parent length (Sec. 3.2, positions L, L+1, ...) without touching the parent. */
KVR_API kvr_status kvr_seq_fork(kvr_ctx* ctx, kvr_seq parent, kvr_stream stream, kvr_seq* out);
KVR_API kvr_status kvr_seq_close(kvr_ctx* ctx, kvr_seq seq);
/* Committed length (positions 0..len-1 are cached for every layer). */
KVR_API kvr_status kvr_seq_length(const kvr_ctx* ctx, kvr_seq seq, uint32_t* len);
/* Make room for n_tokens[b] more positions after each sequence's length
 * (allocates pages; enqueues the page-table upload on `stream`).  The append
 * call reserves on its own when needed; reserving ahead keeps page-table
 * uploads out of a captured CUDA graph. */
KVR_API kvr_status kvr_seq_reserve(kvr_ctx* ctx, int n_seqs, const kvr_seq* seqs,
                           const int32_t* n_tokens, kvr_stream stream);
/* After the last layer's append: length += n_tokens[b]. */
KVR_API kvr_status kvr_seq_advance(kvr_ctx* ctx, int n_seqs, const kvr_seq* seqs,
                           const int32_t* n_tokens);

/* ---- artifact I/O (Algorithm 1 store / Algorithm 2 deserialize) ---- */

/* Place an artifact [layers][2][n_kv_heads][L][head_dim] (host memory if
 * on_device == 0, else device) into a new sequence of length L, bit for bit
 * (Sec. 3.3: deserialisation is value-preserving).  Rejects a metadata
 * (model id, dtype) that differs from the context's with KVR_ERR_META_MISMATCH
 * (Sec. 3.1, Algorithm 2's assert).  Copies are enqueued on `stream`; a host
 * artifact must stay valid until the stream reaches them.
 * meta->dtype == KVR_DTYPE_Q8 loads an int8 artifact (kvr_artifact_bytes_q8
 * layout) of the same model: one kernel dequantises every code into the bf16
 * cache as bf16(code * s), an fp32 product rounded once (Sec. 5 "Quantizing
 * the artifact": lossy, so such a cache is no longer bitwise the publisher's).
 * An int8 artifact is read in place by that kernel: it must be device memory
 * or pinned host memory (KVR_ERR_UNSUPPORTED for pageable host memory) and
 * 16-byte aligned (KVR_ERR_INVALID_ARG). */
KVR_API kvr_status kvr_load_kv(kvr_ctx* ctx, const kvr_artifact_meta* meta, const void* artifact,
                       int on_device, kvr_stream stream, kvr_seq* out);
/* kvr_load_kv of an int8 (KVR_DTYPE_Q8) artifact that also keeps its codes
 * resident (Sec. 5's int8 artifact, dequantised inside the reuse kernel's tile
 * load): the sequence gets the bf16 cache of kvr_load_kv -- which every other
 * kernel reads -- plus an int8 copy of each of its full pages (one more page
 * each from the pool, shared by forks like the bf16 pages).  Reuse attention
 * on the decode path (<= 8 query rows per KV head: kvr_decode_step, and
 * kvr_reuse_attn with num_splits = 0) reads those pages' int8 copies, half the
 * bytes: the codes become exact f16 values in shared memory and the per-tensor
 * scales multiply the scores (s_K) and the probabilities (s_V), so these keys
 * enter attention as code * s exactly, without the bf16 rounding of the
 * dequantising load.  Results agree with the plain load's within the bf16
 * attention tolerance, not bit for bit; q enters those products as f16
 * (saturated beyond +-65504).
 * Errors as kvr_load_kv and kvr_export_kv_q8's buffer rules; KVR_ERR_OOM when
 * the pool lacks the extra pages; KVR_ERR_UNSUPPORTED for a pool too large for
 * the int8 row space (2 x page rows >= 2^31). */
KVR_API kvr_status kvr_load_kv_q8_resident(kvr_ctx* ctx, const kvr_artifact_meta* meta, const void* artifact,
                                   int on_device, kvr_stream stream, kvr_seq* out);
/* Write positions 0..len-1 of `seq` as an artifact (same layout) and its
 * metadata (Algorithm 1: store (K, V) per layer with m = (model, dtype, L)). */
KVR_API kvr_status kvr_export_kv(kvr_ctx* ctx, kvr_seq seq, void* artifact, int on_device,
                         kvr_stream stream, kvr_artifact_meta* meta_out);
/* Algorithm 1 with the Sec. 5 int8 artifact: write positions 0..len-1 of `seq`
 * as per-tensor symmetric int8 (kvr_artifact_bytes_q8 layout) and meta_out
 * with dtype KVR_DTYPE_Q8.  A tensor is one layer's K or one layer's V over
 * all KV heads and positions; its scale s = max|x| / 127 and each code
 * round-half-even(x / s) clamped to [-127, 127] (0 when s = 0), with s and
 * x / s IEEE fp32 operations.  Two kernels (max |x| per tensor, then the
 * codes) write the artifact in place: device memory, or pinned host memory
 * (KVR_ERR_UNSUPPORTED for pageable), 16-byte aligned.  Uses the first
 * 8 * layers bytes of the context's workspace on `stream`.  An empty
 * sequence writes nothing. */
KVR_API kvr_status kvr_export_kv_q8(kvr_ctx* ctx, kvr_seq seq, void* artifact, int on_device,
                            kvr_stream stream, kvr_artifact_meta* meta_out);

/* Self-describing artifact container for storage and transfer (Algorithm 1
 * publishes (K, V) with m = (model, dtype, L); Algorithm 2 checks m before
 * loading).  A container is a KVR_ARTIFACT_HEADER_BYTES header followed by the
 * artifact bytes of kvr_artifact_bytes(desc, L) (kvr_artifact_bytes_q8 for a
 * KVR_DTYPE_Q8 artifact), in the layouts above.  Header
 * (little-endian, 64 bytes): magic "KVRA", uint32 version (1), uint64 model_id,
 * uint32 dtype, uint32 L, uint32 layers, uint32 n_kv_heads, uint32 head_dim,
 * uint32 reserved (0), uint64 payload bytes, 16 bytes reserved (0). */
#define KVR_ARTIFACT_HEADER_BYTES 64

/* Fill `header` (host memory, KVR_ARTIFACT_HEADER_BYTES writable bytes, owned
 * by the caller) for an artifact of `meta` produced under `desc` (for instance
 * the meta_out of kvr_export_kv).  Pure host code.  KVR_ERR_INVALID_ARG on null
 * pointers or a meta whose model id differs from desc or whose dtype is
 * neither desc's nor KVR_DTYPE_Q8. */
KVR_API kvr_status kvr_artifact_write_header(const kvr_model_desc* desc, const kvr_artifact_meta* meta,
                                     void* header);
/* Check a container header (host memory) against the model of `desc`: the
 * magic and version, then (model id, dtype) and the shape (layers, n_kv_heads,
 * head_dim) -- KVR_ERR_META_MISMATCH if any differs (Algorithm 2's assert;
 * a KVR_DTYPE_Q8 artifact of the same model is accepted),
 * KVR_ERR_INVALID_ARG for a malformed header or a payload size that does not
 * match L.  On success fills meta_out and *payload_bytes (either may be null).
 * Pure host code. */
KVR_API kvr_status kvr_artifact_read_header(const kvr_model_desc* desc, const void* header,
                                    kvr_artifact_meta* meta_out, uint64_t* payload_bytes);

/* ---- the hot path ---- */

/* Append step for one layer.  Sequence b contributes tokens cu_q[b]..cu_q[b+1]-1
 * of the packed inputs at positions start_pos[b] .. start_pos[b]+n_b-1, and
 * start_pos[b] must equal the sequence's committed length (else
 * KVR_ERR_POSITION: Sec. 3.2 requires positions L, L+1, ...).  Per token and
 * head: y = RMSNorm(x) * w over head_dim (eps = rms_eps), then rotate-half RoPE
 * at the token's position with base rope_theta, computed in fp32 and rounded to
 * bf16 once.  Normed+roped q goes to q_out [T][n_q_heads][head_dim]; normed+roped
 * k and the unchanged v go to the cache at those positions of `layer`.
 * q_pre [T][n_q_heads][d], k_pre and v [T][n_kv_heads][d], q_norm_w and k_norm_w [d];
 * cu_q_host and start_pos_host are host arrays of n_seqs+1 and n_seqs entries. */
KVR_API kvr_status kvr_append_kv(kvr_ctx* ctx, int layer, int n_seqs, const kvr_seq* seqs,
                         const int32_t* start_pos_host, const int32_t* cu_q_host,
                         const void* q_pre, const void* k_pre, const void* v,
                         const void* q_norm_w, const void* k_norm_w, void* q_out,
                         kvr_stream stream);

/* Reuse attention for one layer (Algorithm 2's forward over cached context).
 * Rows of sequence b are the tokens cu_q[b]..cu_q[b+1]-1 of q [T][n_q_heads][d]
 * (normed+roped, as written by kvr_append_kv) at positions len_b .. len_b+n_b-1,
 * len_b the committed length; each row attends causally to keys 0..its position
 * of its own sequence: the shared prefix and its own appended tokens (Sec. 3.2:
 * the mask spans all L+|q| positions).  Query head h reads KV head
 * h / (n_q_heads / n_kv_heads); scores are scaled by 1/sqrt(head_dim).
 * Sequences forked from one parent share its full prefix pages: each such key
 * tile is staged once per query block and serves every consumer row in it.
 * out [T][n_q_heads][d] bf16; lse [T][n_q_heads] fp32 natural-log sum of exp of
 * the scaled scores (may be NULL).  opts may be NULL (automatic splits). */
KVR_API kvr_status kvr_reuse_attn(kvr_ctx* ctx, int layer, int n_seqs, const kvr_seq* seqs,
                          const int32_t* cu_q_host, const void* q, void* out, float* lse,
                          const kvr_attn_opts* opts, kvr_stream stream);

/* One decode step of Algorithm 2 for one layer: kvr_append_kv followed by
 * kvr_reuse_attn over the same tokens, with the same arguments and results
 * (the cache, q_out if not NULL, out and lse are bitwise what the two calls
 * produce).  When every KV head serves at most 8 rows (tokens x GQA group) and
 * opts requests automatic splits, both run in one launch; otherwise the two
 * calls are made in turn and q_out must not be NULL. */
KVR_API kvr_status kvr_decode_step(kvr_ctx* ctx, int layer, int n_seqs, const kvr_seq* seqs,
                                   const int32_t* start_pos_host, const int32_t* cu_q_host,
                                   const void* q_pre, const void* k_pre, const void* v,
                                   const void* q_norm_w, const void* k_norm_w, void* q_out,
                                   void* out, float* lse, const kvr_attn_opts* opts,
                                   kvr_stream stream);

/* Full causal prefill attention for one layer (Sec. 1: prefill runs a forward
 * pass over all L tokens; Sec. 5 Table 1 cost (a)): rows len .. len+n_tokens-1
 * of `seq` against keys 0..row, q [n_tokens][n_q_heads][d].  For a fresh
 * sequence (len 0) that is the whole prefill over positions 0..n_tokens-1.
 * Same kernel and tile order as kvr_reuse_attn. */
KVR_API kvr_status kvr_prefill_attn(kvr_ctx* ctx, int layer, kvr_seq seq, int n_tokens,
                            const void* q, void* out, float* lse,
                            const kvr_attn_opts* opts, kvr_stream stream);

/* ---- reuse attention without allocation ----
 * The paper has no counterpart to this call; it serves callers that cannot
 * allocate device memory where they run attention (for example code running
 * under another framework's allocator that forbids side allocations, or a
 * runtime that reserved all device memory up front).  Same arguments, rows,
 * masking and results as kvr_reuse_attn (within its rounding; the split count
 * may differ), but the per-split partial results live in a fixed
 * KVR_NOALLOC_SCRATCH_BYTES array inside the library's device image instead of
 * the context's workspace.  Every GPU that loads the library holds that array
 * until the process exits; nothing is allocated per call (no cudaMalloc, no
 * cudaFree, no allocating library routine).
 *  - The first call on a device looks up the array's device address on that
 *    device (it must be the current device); make that first call before any
 *    stream capture.  A device reset (cudaDeviceReset, or the primary
 *    context released and created again) invalidates that address: the next
 *    call finds a different current context and looks it up again, so make
 *    that call, too, before any capture.
 *  - Splits: num_splits = 0 picks as many as the array holds (one pass when
 *    even two do not fit); an explicit count whose partials
 *    (num_splits * T * n_q_heads * (head_dim + 1) * 4 bytes) exceed the array
 *    is rejected with KVR_ERR_OOM.
 *  - All calls share the one array and it keeps the last call's contents; no
 *    part of it needs to start at zero (every partial a call reads back, the
 *    same call wrote).  Calls that overlap on the GPU (other streams, other
 *    threads, other contexts of this process on the same device) race on it:
 *    serialise them. */
#define KVR_NOALLOC_SCRATCH_BYTES ((size_t)16 << 20)
KVR_API kvr_status kvr_reuse_attn_noalloc(kvr_ctx* ctx, int layer, int n_seqs, const kvr_seq* seqs,
                                          const int32_t* cu_q_host, const void* q, void* out,
                                          float* lse, const kvr_attn_opts* opts, kvr_stream stream);

/* ---- a whole decoder layer (Table 1's costs are whole-model forwards) ---- */

/* The paper measures a whole Qwen3-4B forward (Sec. 5, Table 1) and names the
 * model, not its layer; these calls run the public Qwen3 decoder layer around
 * the hot path so that whole-layer prefill and reuse-step costs can be
 * measured: h1 = h + Wo . attn(QKnorm+RoPE(Wq x, Wk x), Wv x) with
 * x = RMSNorm(h); h_out = h1 + Wd . (silu(Wg x2) * (Wu x2)) with
 * x2 = RMSNorm(h1).  The model runs in bf16: every tensor between two
 * operations is bf16, computed in fp32 (projections are this library's
 * tcgen05 bf16 GEMM with fp32 accumulation, or its weight-streaming GEMV when
 * the batch has at most 8 tokens; the residual add is the GEMM's epilogue, one
 * rounding; SwiGLU is the gate/up GEMM's epilogue, from the bf16-rounded
 * gate and up values), and the norms are this library's kernels. */
typedef struct kvr_layer_desc {
  uint32_t hidden;        /* residual width (2560 for Qwen3-4B), multiple of 8 */
  uint32_t intermediate;  /* MLP width (9728 for Qwen3-4B), multiple of 8 */
} kvr_layer_desc;

/* One layer's weights, bf16, device memory, row-major [out][in] (the layout
 * of a Linear layer's weight), all 16-byte aligned.  Owned by the caller. */
typedef struct kvr_layer_weights {
  const void* input_norm; /* [hidden] */
  const void* wq;         /* [n_q_heads * head_dim][hidden] */
  const void* wk;         /* [n_kv_heads * head_dim][hidden] */
  const void* wv;         /* [n_kv_heads * head_dim][hidden] */
  const void* q_norm;     /* [head_dim] */
  const void* k_norm;     /* [head_dim] */
  const void* wo;         /* [hidden][n_q_heads * head_dim] */
  const void* post_norm;  /* [hidden] */
  const void* w_gate_up;  /* [2 * intermediate][hidden]: the gate rows, then the up rows */
  const void* w_down;     /* [hidden][intermediate] */
} kvr_layer_weights;

/* Scratch that kvr_layer_forward needs for up to max_tokens packed tokens
 * (activations plus the GEMM workspace); 0 for a bad desc. */
KVR_API size_t kvr_layer_workspace_bytes(const kvr_model_desc* desc, const kvr_layer_desc* ldesc,
                                         uint32_t max_tokens);

/* One layer for the packed tokens of n_seqs sequences (the kvr_append_kv
 * batch convention: tokens cu_q[b]..cu_q[b+1]-1 of sequence b at positions
 * start_pos[b].., start_pos[b] == the sequence's length), h_in / h_out
 * [T][hidden] bf16 device (h_out may not alias h_in).  The keys and values of
 * the new tokens are appended to the cache (call kvr_seq_advance after the
 * last layer, as with kvr_append_kv).  Attention: kvr_prefill_attn when the
 * batch is one sequence starting at position 0 (prefill from scratch, Table 1
 * cost (a)), else the reuse path of kvr_decode_step (a continuation step over
 * the cache, cost (b)).  `workspace` (device, 256-byte aligned,
 * kvr_layer_workspace_bytes(desc, ldesc, T) bytes at least) is overwritten.
 * Errors as kvr_append_kv / kvr_reuse_attn; KVR_ERR_CUDA when a launch
 * fails. */
KVR_API kvr_status kvr_layer_forward(kvr_ctx* ctx, int layer, const kvr_layer_desc* ldesc,
                                     const kvr_layer_weights* w, int n_seqs, const kvr_seq* seqs,
                                     const int32_t* start_pos_host, const int32_t* cu_q_host,
                                     const void* h_in, void* h_out, void* workspace,
                                     size_t workspace_bytes, kvr_stream stream);

/* ---- the layer's projections on their own ----
 * The GEMMs of kvr_layer_forward (Sec. 5 Table 1 times whole-model forwards;
 * these are the Qwen3 layer's linear maps), for testing and for callers that
 * run their own layer.  Always the tcgen05 GEMM, for any T >= 1.
 *   kvr_linear:        d[T][N] = bf16(x[T][K] w[N][K]^T (+ c[T][N]))
 *   kvr_linear_swiglu: a[T][I] = bf16(silu(g) * u), g = bf16(x W_gate^T),
 *                      u = bf16(x W_up^T), w_gate_up = [W_gate; W_up] ([2 I][K])
 * bf16 row-major device tensors owned by the caller, fp32 accumulation, one
 * rounding per output; c may be NULL.  `workspace` (device, 16-byte aligned,
 * may be NULL) is fp32 scratch for split-K: when the output tiles alone would
 * leave most SMs idle (short batches), K is split over several CTAs whose
 * partial sums (splits x T x N, or x 2 I, floats) are added in split order by
 * a second kernel; the split count is cut to what workspace_bytes holds (none
 * without a workspace).  K, N and I must be positive multiples of 8 and every
 * pointer 16-byte aligned (else KVR_ERR_INVALID_ARG, nothing enqueued).
 * Asynchronous on `stream`; a device-side wait that gives up is reported by
 * kvr_sync_status(ctx), whose error word the kernel uses. */
KVR_API kvr_status kvr_linear(kvr_ctx* ctx, int T, int N, int K, const void* x, const void* w, const void* c,
                              void* d, void* workspace, size_t workspace_bytes, kvr_stream stream);
KVR_API kvr_status kvr_linear_swiglu(kvr_ctx* ctx, int T, int I, int K, const void* x, const void* w_gate_up,
                                     void* a, void* workspace, size_t workspace_bytes, kvr_stream stream);

#ifdef __cplusplus
}
#endif

#endif /* KVR_H_ */
