// kvr_api.cu -- the C ABI of include/kvr.h: context over a caller-owned device
// pool (page tables, int8-copy tables and scales, RoPE table, split
// workspace, the decode kernels' cluster-partial area, pages), page allocator
// with shared (refcounted) prefix pages and their int8 copies, sequence
// bookkeeping, argument checks, the artifact container header, and the
// launches of the append, attention, decode, split-combine and artifact
// kernels.
//
// Paper: "Can I Buy Your KV Cache?" (arXiv 2606.13361).  Sec. 3.1/Algorithm 1
// (artifact = per-layer K, V + metadata), Sec. 3.2/Algorithm 2 (load, assert
// metadata, continue at positions L, L+1, ... under a full mask), Sec. 3.3
// Claim 1 (reuse rows == prefill rows).
#include <cudaTypedefs.h>

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <string>
#include <vector>

#include "kvr_artifact.cuh"
#include "kvr_internal.h"
#include "kvr_ptx.cuh"

using namespace kvr;

namespace {

thread_local std::string g_last_error;

kvr_status fail(kvr_status s, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return s;
}

kvr_status cuda_fail(cudaError_t e, const char* what) {
  return fail(KVR_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

#define KVR_CUDA(call)                                   \
  do {                                                   \
    cudaError_t e_ = (call);                             \
    if (e_ != cudaSuccess) return cuda_fail(e_, #call);  \
  } while (0)

constexpr size_t kAlign = 256;
constexpr size_t kPageAlign = 4096;
constexpr size_t kDefaultWorkspace = size_t(256) << 20;

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

bool desc_ok(const kvr_model_desc* d, const char** why) {
  if (!d) { *why = "null model desc"; return false; }
  if (d->layers == 0 || d->layers > 1024) { *why = "layers must be in [1, 1024]"; return false; }
  if (d->head_dim != 64 && d->head_dim != 128) { *why = "head_dim must be 64 or 128"; return false; }
  if (d->n_kv_heads == 0 || d->n_q_heads == 0 || d->n_q_heads % d->n_kv_heads) {
    *why = "n_q_heads must be a positive multiple of n_kv_heads"; return false;
  }
  const uint32_t G = d->n_q_heads / d->n_kv_heads;
  if (G != 1 && G != 2 && G != 4 && G != 8 && G != 16) { *why = "GQA group must be 1, 2, 4, 8 or 16"; return false; }
  if (d->dtype != KVR_DTYPE_BF16) { *why = "only KVR_DTYPE_BF16 is supported"; return false; }
  if (d->max_positions == 0 || d->max_positions > (1u << 24)) { *why = "max_positions must be in [1, 2^24]"; return false; }
  if (!(d->rope_theta > 1.0) || !(d->rms_eps >= 0.0)) { *why = "rope_theta must be > 1 and rms_eps >= 0"; return false; }
  return true;
}

struct Seq {
  bool used = false;
  bool root = true;        // opened or loaded (not forked)
  uint32_t len = 0;        // committed positions
  uint64_t family = 0;     // lineage id: forks share their root's id
  uint32_t n_shared = 0;   // for forks: leading pages identical to the root's
  std::vector<int32_t> pages;
  std::vector<int32_t> q8_pages;  // int8 copies of the first pages (int8-resident prefix)
};

}  // namespace

struct kvr_ctx {
  kvr_model_desc desc{};
  int device = 0;
  int num_sms = 148;
  char* pool = nullptr;
  size_t pool_bytes = 0;
  int* d_err = nullptr;
  uint32_t* d_amax = nullptr;  // [layers][2] max |x| scratch of kvr_export_kv_q8
  int32_t* d_page_table = nullptr;
  int32_t* d_q8_table = nullptr;   // [max_seqs][max_pages]: int8 copy of each page, or -1
  float* d_q8_scales = nullptr;    // [max_seqs][layers][2]: their per-tensor scales
  float* d_dpart = nullptr;  // decode cluster partials [Hkv][kDecodeMaxClusters][decode_part_floats(d)]
  int* d_dcnt = nullptr;     // their arrival counts [Hkv][kDecodeMaxSplits], zero between launches
  float2* d_rope = nullptr;
  float* d_ws = nullptr;
  size_t ws_bytes = 0;
  char* d_pages = nullptr;
  int64_t n_pages = 0;
  size_t page_bytes = 0;
  uint32_t max_seqs = 0, max_pages = 0;
  std::vector<int32_t> h_table;  // host mirror of the page tables
  std::vector<int32_t> h_q8_table;
  std::vector<Seq> seqs;
  std::vector<int32_t> page_ref;
  std::vector<int32_t> free_pages;
  uint64_t next_family = 1;
  CUtensorMap tm_kv{};
  CUtensorMap tm_kv32{};
  CUtensorMap tm_q8{};   // the page area as rows of head_dim bytes (int8 K copies)
  CUtensorMap tm_q8t{};  // the page area as rows of 128 bytes (int8 V copies, transposed)
  bool q8_ok = false;   // int8 row space fits a TMA coordinate
  int64_t n_pool_rows = 0;
  uint64_t launches = 0;  // kernels this context has launched
};

namespace kvr {

// For the layer driver (kvr_layer.cu): the context's model, its launch
// counter, and the thread's last-error message.
const kvr_model_desc* ctx_desc(const kvr_ctx* c) { return &c->desc; }
void ctx_add_launches(kvr_ctx* c, int n) { c->launches += static_cast<uint64_t>(n); }
int* ctx_err(kvr_ctx* c) { return c->d_err; }
kvr_status set_error(kvr_status s, const char* msg) {
  g_last_error = msg;
  return s;
}

}  // namespace kvr

namespace {

PFN_cuTensorMapEncodeTiled_v12000 get_encode() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

}  // namespace

namespace kvr {
int encode_bf16_2d(CUtensorMap* tm, const void* base, uint64_t inner, uint64_t rows, uint32_t box_inner,
                   uint32_t box_rows) {
  auto enc = get_encode();
  if (!enc) return static_cast<int>(CUDA_ERROR_NOT_SUPPORTED);
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(inner), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(inner) * 2};
  cuuint32_t box[2] = {box_inner, box_rows};
  cuuint32_t es[2] = {1, 1};
  return static_cast<int>(enc(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
                              es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE));
}
}  // namespace kvr

namespace {

// 2D map over rows of `d` bf16 (row stride d*2 bytes), box 64 x box_rows, 128B swizzle.
kvr_status encode_rows_map(CUtensorMap* tm, void* base, int64_t rows, int d, int box_rows) {
  auto enc = get_encode();
  if (!enc) return fail(KVR_ERR_CUDA, "cuTensorMapEncodeTiled is unavailable");
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(d) * 2};
  cuuint32_t box[2] = {64, static_cast<cuuint32_t>(box_rows)};
  cuuint32_t es[2] = {1, 1};
  CUresult r = enc(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, base, dims, strides, box, es,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(KVR_ERR_CUDA, "cuTensorMapEncodeTiled(rows) failed: %d", int(r));
  return KVR_OK;
}

// 2D map over the page area as rows of d bytes (int8 K codes), box (d, 32);
// 128B swizzle at d = 128 (rows of 128 bytes), none at d = 64.
kvr_status encode_q8_map(CUtensorMap* tm, void* base, int64_t rows, int d) {
  auto enc = get_encode();
  if (!enc) return fail(KVR_ERR_CUDA, "cuTensorMapEncodeTiled is unavailable");
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(d)};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(d), 32};
  cuuint32_t es[2] = {1, 1};
  CUresult r = enc(tm, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, base, dims, strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
                   d == 128 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(KVR_ERR_CUDA, "cuTensorMapEncodeTiled(q8) failed: %d", int(r));
  return KVR_OK;
}

// 2D map over the page area as rows of 128 bytes (int8 V codes stored
// transposed, [d][128 keys] per page block), box (32 keys, d rows), no swizzle.
kvr_status encode_q8t_map(CUtensorMap* tm, void* base, int64_t rows128, int d) {
  auto enc = get_encode();
  if (!enc) return fail(KVR_ERR_CUDA, "cuTensorMapEncodeTiled is unavailable");
  cuuint64_t dims[2] = {128, static_cast<cuuint64_t>(rows128)};
  cuuint64_t strides[1] = {128};
  cuuint32_t box[2] = {32, static_cast<cuuint32_t>(d)};
  cuuint32_t es[2] = {1, 1};
  CUresult r = enc(tm, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, base, dims, strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
                   CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(KVR_ERR_CUDA, "cuTensorMapEncodeTiled(q8t) failed: %d", int(r));
  return KVR_OK;
}

// 3D map over q [T][Hq][d], box (64, G, 128/G), 128B swizzle.
kvr_status encode_q_map(CUtensorMap* tm, const void* q, int T, int Hq, int d, int G) {
  auto enc = get_encode();
  if (!enc) return fail(KVR_ERR_CUDA, "cuTensorMapEncodeTiled is unavailable");
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(Hq), static_cast<cuuint64_t>(T)};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(d) * 2, static_cast<cuuint64_t>(Hq) * d * 2};
  cuuint32_t box[3] = {64, static_cast<cuuint32_t>(G), static_cast<cuuint32_t>(kBlockRows / G)};
  cuuint32_t es[3] = {1, 1, 1};
  CUresult r = enc(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(q), dims, strides, box, es,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(KVR_ERR_CUDA, "cuTensorMapEncodeTiled(q) failed: %d", int(r));
  return KVR_OK;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; }

Seq* get_seq(kvr_ctx* c, kvr_seq s) {
  if (!c || s < 0 || static_cast<uint32_t>(s) >= c->max_seqs || !c->seqs[s].used) return nullptr;
  return &c->seqs[s];
}

uint32_t shared_with_root(const kvr_ctx* c, const Seq& s) {
  (void)c;
  return s.root ? s.len / kPageTokens : s.n_shared;
}

// Page-table rows reach the device through a kernel whose parameters carry
// the values (copied at launch), so the update is ordered on the stream, never
// waits on the host, and can be captured in a CUDA graph.
constexpr int kTableChunk = 7168;
struct TableUpdate {
  int64_t offset;
  int32_t n;
  int32_t vals[kTableChunk];
};

// One thread waits on a phase of a fresh barrier that nothing arrives on; the
// bounded wait gives up after its limit and records the timeout in `err`.
__global__ void wait_timeout_kernel(int* err) {
  __shared__ uint64_t bar;
  __shared__ int abort_word;
  griddep_wait();
  griddep_launch_dependents();
  if (threadIdx.x != 0) return;
  abort_word = 0;
  mbar_init(&bar, 1);
  fence_barrier_init();
  (void)mbar_wait(&bar, 0, &abort_word, err);
}

__global__ void table_update_kernel(const __grid_constant__ TableUpdate u, int32_t* table) {
  griddep_wait();
  griddep_launch_dependents();
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < u.n; i += gridDim.x * blockDim.x)
    table[u.offset + i] = u.vals[i];
}

kvr_status upload_rows(kvr_ctx* c, uint32_t lo, uint32_t hi, cudaStream_t st) {
  if (lo > hi) return KVR_OK;
  const size_t off = static_cast<size_t>(lo) * c->max_pages;
  const size_t n = static_cast<size_t>(hi - lo + 1) * c->max_pages;
  thread_local static TableUpdate u;  // filled and launched (parameters copied) one chunk at a time
  for (size_t done = 0; done < n; done += kTableChunk) {
    const int m = static_cast<int>(std::min<size_t>(kTableChunk, n - done));
    u.offset = static_cast<int64_t>(off + done);
    u.n = m;
    std::memcpy(u.vals, c->h_table.data() + off + done, m * sizeof(int32_t));
    KVR_CUDA(launch_kernel(table_update_kernel, dim3((m + 255) / 256), dim3(256), 0, st, 0, u, c->d_page_table));
    ++c->launches;
  }
  return KVR_OK;
}

// The int8-copy row of sequence s (its host mirror and the device table),
// through the same parameter-carrying kernel.
kvr_status upload_q8_row(kvr_ctx* c, kvr_seq s, cudaStream_t st) {
  int32_t* row = c->h_q8_table.data() + static_cast<size_t>(s) * c->max_pages;
  const Seq& q = c->seqs[s];
  for (uint32_t i = 0; i < c->max_pages; ++i) row[i] = i < q.q8_pages.size() ? q.q8_pages[i] : -1;
  thread_local static TableUpdate u;
  for (size_t done = 0; done < c->max_pages; done += kTableChunk) {
    const int m = static_cast<int>(std::min<size_t>(kTableChunk, c->max_pages - done));
    u.offset = static_cast<int64_t>(static_cast<size_t>(s) * c->max_pages + done);
    u.n = m;
    std::memcpy(u.vals, row + done, m * sizeof(int32_t));
    KVR_CUDA(launch_kernel(table_update_kernel, dim3((m + 255) / 256), dim3(256), 0, st, 0, u, c->d_q8_table));
    ++c->launches;
  }
  return KVR_OK;
}

void write_row(kvr_ctx* c, kvr_seq s) {
  int32_t* row = c->h_table.data() + static_cast<size_t>(s) * c->max_pages;
  const Seq& q = c->seqs[s];
  for (uint32_t i = 0; i < c->max_pages; ++i) row[i] = i < q.pages.size() ? q.pages[i] : -1;
}

int32_t alloc_page(kvr_ctx* c) {
  if (c->free_pages.empty()) return -1;
  int32_t p = c->free_pages.back();
  c->free_pages.pop_back();
  c->page_ref[p] = 1;
  return p;
}

void release_page(kvr_ctx* c, int32_t p) {
  if (--c->page_ref[p] == 0) c->free_pages.push_back(p);
}

int find_free_slot(kvr_ctx* c) {
  for (uint32_t i = 0; i < c->max_seqs; ++i)
    if (!c->seqs[i].used) return static_cast<int>(i);
  return -1;
}

// Grow each sequence's pages to hold `need[b]` positions; all-or-nothing.
// A new page is zero-filled unless the calling operation writes all of its
// positions (`writes`: positions len..need-1 of every layer are about to be
// written).  Attention multiplies whole key tiles: a position past a
// sequence's end enters P V with p = 0, and 0 x (stale bits that read as NaN
// or Inf) would poison the row, so such positions must hold finite values.
kvr_status ensure_capacity(kvr_ctx* c, int n, const kvr_seq* seqs, const uint32_t* need,
                           cudaStream_t st, bool writes = true) {
  size_t extra = 0;
  for (int b = 0; b < n; ++b) {
    const Seq& q = c->seqs[seqs[b]];
    const size_t want = (static_cast<size_t>(need[b]) + kPageTokens - 1) / kPageTokens;
    if (need[b] > c->desc.max_positions)
      return fail(KVR_ERR_INVALID_ARG, "sequence %d would pass max_positions (%u > %u)", seqs[b],
                  need[b], c->desc.max_positions);
    if (want > q.pages.size()) extra += want - q.pages.size();
  }
  if (extra == 0) return KVR_OK;
  if (extra > c->free_pages.size())
    return fail(KVR_ERR_OOM, "page pool exhausted: need %zu pages, %zu free", extra, c->free_pages.size());
  uint32_t lo = UINT32_MAX, hi = 0;
  for (int b = 0; b < n; ++b) {
    Seq& q = c->seqs[seqs[b]];
    const size_t want = (static_cast<size_t>(need[b]) + kPageTokens - 1) / kPageTokens;
    if (want <= q.pages.size()) continue;
    while (q.pages.size() < want) {
      const uint32_t pi = static_cast<uint32_t>(q.pages.size());
      const int32_t pg = alloc_page(c);
      q.pages.push_back(pg);
      const bool covered = writes && pi * kPageTokens >= q.len && (pi + 1) * kPageTokens <= need[b];
      if (!covered) KVR_CUDA(cudaMemsetAsync(c->d_pages + static_cast<size_t>(pg) * c->page_bytes, 0, c->page_bytes, st));
    }
    write_row(c, seqs[b]);
    lo = std::min(lo, static_cast<uint32_t>(seqs[b]));
    hi = std::max(hi, static_cast<uint32_t>(seqs[b]));
  }
  return upload_rows(c, lo, hi, st);
}

// Validate a batch and fill the kernel-side description.  Sequences with no
// tokens are dropped.  Rows of sequence b sit at positions start_b.. where
// start_b is its committed length.
kvr_status build_batch(kvr_ctx* c, int n_seqs, const kvr_seq* seqs, const int32_t* cu_q,
                       const int32_t* start_pos, BatchDesc* bd, std::vector<kvr_seq>* kept,
                       std::vector<uint32_t>* need) {
  if (n_seqs < 0 || n_seqs > kMaxBatch)
    return fail(KVR_ERR_INVALID_ARG, "n_seqs must be in [0, %d]", kMaxBatch);
  if (n_seqs > 0 && (!seqs || !cu_q)) return fail(KVR_ERR_INVALID_ARG, "null seqs or cu_q");
  if (n_seqs > 0 && cu_q[0] != 0) return fail(KVR_ERR_INVALID_ARG, "cu_q[0] must be 0");
  bd->n_seqs = 0;
  bd->T = n_seqs > 0 ? cu_q[n_seqs] : 0;
  bd->max_pages = static_cast<int>(c->max_pages);
  bd->page_table = c->d_page_table;
  bd->shared_pages = 0;
  bd->cu_q[0] = 0;
  for (int b = 0; b < n_seqs; ++b) {
    if (cu_q[b + 1] < cu_q[b]) return fail(KVR_ERR_INVALID_ARG, "cu_q must be non-decreasing");
    Seq* q = get_seq(c, seqs[b]);
    if (!q) return fail(KVR_ERR_INVALID_ARG, "unknown sequence handle %d", seqs[b]);
    for (int e = 0; e < b; ++e)
      if (seqs[e] == seqs[b]) return fail(KVR_ERR_INVALID_ARG, "sequence %d appears twice", seqs[b]);
    if (start_pos && static_cast<uint32_t>(start_pos[b]) != q->len)
      return fail(KVR_ERR_POSITION,
                  "sequence %d: start position %d != cached length %u (continuation tokens must take "
                  "positions L, L+1, ...)",
                  seqs[b], start_pos[b], q->len);
    const int nb = cu_q[b + 1] - cu_q[b];
    if (nb == 0) continue;
    const int k = bd->n_seqs++;
    bd->slot[k] = seqs[b];
    bd->start[k] = static_cast<int32_t>(q->len);
    bd->cu_q[k + 1] = cu_q[b + 1];
    kept->push_back(seqs[b]);
    need->push_back(q->len + static_cast<uint32_t>(nb));
  }
  if (bd->T > 0 && static_cast<int64_t>(bd->T) * c->desc.n_q_heads * c->desc.head_dim > (int64_t(1) << 40))
    return fail(KVR_ERR_INVALID_ARG, "batch too large");
  // Leading pages common to the whole batch: forks of one root share its full pages.
  if (bd->n_seqs > 1) {
    const Seq& s0 = c->seqs[bd->slot[0]];
    uint32_t sh = shared_with_root(c, s0);
    for (int k = 1; k < bd->n_seqs && sh > 0; ++k) {
      const Seq& s = c->seqs[bd->slot[k]];
      if (s.family != s0.family) sh = 0;
      else sh = std::min(sh, shared_with_root(c, s));
    }
    bd->shared_pages = static_cast<int>(sh);
  }
  return KVR_OK;
}

// Query blocks per attention CTA.  Two halve the K/V bytes staged per MMA
// (the kernel is bound by that staging rate) and pay off when the query
// blocks alone fill the GPU.  Split-heavy batches keep one: their fixed
// per-CTA costs and split partials dominate, and with many consumers a pair of
// blocks walks the union of both blocks' own suffix tiles, each visible to few
// rows (measured slower for 256 decode rows per KV head); with one block both
// softmax warpgroups share each key tile.  An explicit single split (the
// bitwise reuse == prefill mode) always takes two, so that a row runs the same
// arithmetic whatever the batch around it.
int attention_q_tiles(int n_rb, int hkv, int num_sms, const kvr_attn_opts* opts) {
  if (opts && opts->num_splits == 1) return kQTiles;
  return n_rb * hkv >= num_sms ? kQTiles : 1;
}

kvr_status run_attention(kvr_ctx* c, int layer, BatchDesc& bd, const std::vector<uint32_t>& need,
                         const void* q, void* out, float* lse, const kvr_attn_opts* opts,
                         cudaStream_t st) {
  const kvr_model_desc& d = c->desc;
  if (layer < 0 || static_cast<uint32_t>(layer) >= d.layers)
    return fail(KVR_ERR_INVALID_ARG, "layer %d out of range", layer);
  if (bd.T == 0) return KVR_OK;
  if (!q || !out) return fail(KVR_ERR_INVALID_ARG, "null q or out");
  if (!aligned16(q) || !aligned16(out)) return fail(KVR_ERR_INVALID_ARG, "q and out must be 16-byte aligned");
  for (int k = 0; k < bd.n_seqs; ++k) {
    const Seq& s = c->seqs[bd.slot[k]];
    if (s.pages.size() * kPageTokens < need[k])
      return fail(KVR_ERR_POSITION,
                  "sequence %d: rows reach position %u but only %zu positions were appended/reserved",
                  bd.slot[k], need[k] - 1, s.pages.size() * kPageTokens);
  }
  const int G = static_cast<int>(d.n_q_heads / d.n_kv_heads);
  const int TB = kBlockRows / G;
  const float scale_log2 = static_cast<float>(1.4426950408889634 / std::sqrt(static_cast<double>(d.head_dim)));
  // Few rows per KV head (decode of one or two consumers): the CUDA-core kernel
  // with an in-kernel split merge.  An explicit split count keeps the tcgen05
  // kernel (the bitwise reuse == prefill mode uses num_splits = 1).
  if ((!opts || opts->num_splits == 0) && bd.T * G <= kDecodeMaxRows) {
    DecodeArgs da{};
    da.tm_kv32 = c->tm_kv32;
    da.tm_q8 = c->tm_q8;
    da.tm_q8t = c->tm_q8t;
    da.q8_table = c->d_q8_table;
    da.q8_scales = c->d_q8_scales;
    for (int k = 0; k < bd.n_seqs && k < kDecodeMaxRows; ++k)
      da.q8_n[k] = static_cast<int>(c->seqs[bd.slot[k]].q8_pages.size());
    da.q = static_cast<const uint16_t*>(q);
    da.out = static_cast<uint16_t*>(out);
    da.lse = lse;
    da.err = c->d_err;
    da.layer = layer;
    da.layers = static_cast<int>(d.layers);
    da.Hq = static_cast<int>(d.n_q_heads);
    da.Hkv = static_cast<int>(d.n_kv_heads);
    da.G = G;
    da.scale_log2 = scale_log2;
    da.n_pool_rows = c->n_pool_rows;
    da.pages = c->d_pages;
    // the splits of a KV head form one cluster; all heads' clusters resident at once
    const SmallBatch sb = small_batch(bd);
    bool q8 = false;
    for (int k = 0; k < sb.n_seqs && k < kDecodeMaxRows; ++k) q8 = q8 || da.q8_n[k] > 0;
    da.n_splits = decode_splits(static_cast<int>(d.head_dim), da.Hkv, decode_units(sb), q8, &da.n_clusters,
                                &da.n_warps);
    da.part = c->d_dpart;
    da.cnt = c->d_dcnt;
    cudaError_t e = launch_decode(da, sb, static_cast<int>(d.head_dim), false, st);
    if (e != cudaSuccess) return cuda_fail(e, "decode attention launch");
    ++c->launches;
    return KVR_OK;
  }
  AttnArgs a{};
  kvr_status s = encode_q_map(&a.tm_q, q, bd.T, static_cast<int>(d.n_q_heads), static_cast<int>(d.head_dim), G);
  if (s != KVR_OK) return s;
  a.tm_kv = c->tm_kv;
  a.layer = layer;
  a.layers = static_cast<int>(d.layers);
  a.Hq = static_cast<int>(d.n_q_heads);
  a.Hkv = static_cast<int>(d.n_kv_heads);
  a.G = G;
  a.n_rb = (bd.T + TB - 1) / TB;
  a.scale_log2 = scale_log2;
  a.out = static_cast<uint16_t*>(out);
  a.lse = lse;
  a.err = c->d_err;
  a.n_pool_rows = c->n_pool_rows;
  // Key splits: enough CTAs to cover the SMs when query blocks are few.
  uint32_t max_need = 0;
  for (uint32_t v : need) max_need = std::max(max_need, v);
  const int tiles = static_cast<int>((max_need + kPageTokens - 1) / kPageTokens);
  a.q_tiles = attention_q_tiles(a.n_rb, a.Hkv, c->num_sms, opts);
  const int units = (a.n_rb + a.q_tiles - 1) / a.q_tiles * a.Hkv;  // attention CTAs per split
  int S = 1;
  if (!opts || opts->num_splits == 0) {
    if (units < c->num_sms) S = std::min(std::max(1, c->num_sms / units), std::max(1, tiles / 2));
  } else if (opts->num_splits > 0) {
    S = std::min(opts->num_splits, std::max(1, tiles));
  } else {
    return fail(KVR_ERR_INVALID_ARG, "num_splits must be >= 0");
  }
  S = std::min(S, 64);
  const size_t per_split = static_cast<size_t>(bd.T) * d.n_q_heads * (d.head_dim + 1) * sizeof(float);
  if (S > 1 && per_split * S > c->ws_bytes) S = std::max<int>(1, static_cast<int>(c->ws_bytes / per_split));
  if (opts && opts->num_splits > 1 && S < std::min(opts->num_splits, std::max(1, tiles)))
    return fail(KVR_ERR_OOM, "workspace too small for %d splits", opts->num_splits);
  a.n_splits = S;
  if (S > 1) {
    a.part_o = c->d_ws;
    a.part_lse = c->d_ws + static_cast<size_t>(S) * bd.T * d.n_q_heads * d.head_dim;
  }
  cudaError_t e = launch_attention(a, bd, static_cast<int>(d.head_dim), st);
  if (e != cudaSuccess) return cuda_fail(e, "attention launch");
  ++c->launches;
  if (S > 1) {
    ++c->launches;
    e = launch_combine(a.part_o, a.part_lse, S, bd.T, a.Hq, static_cast<int>(d.head_dim),
                       static_cast<uint16_t*>(out), lse, st);
    if (e != cudaSuccess) return cuda_fail(e, "combine launch");
  }
  return KVR_OK;
}

// Scale block of an int8 artifact: fp32 [layers][2], padded to 16 bytes.
size_t q8_scale_bytes(const kvr_model_desc& d) { return align_up(static_cast<size_t>(d.layers) * 8, 16); }

size_t payload_bytes_of(const kvr_model_desc* d, uint32_t dtype, uint32_t L) {
  return dtype == KVR_DTYPE_Q8 ? kvr_artifact_bytes_q8(d, L) : kvr_artifact_bytes(d, L);
}

// The address the artifact kernels use for `p`: device memory as is, pinned
// host memory through its device mapping; null for pageable host memory,
// which no kernel touches (the copy engine moves it).
kvr_status artifact_view(const void* p, int on_device, char** view) {
  cudaPointerAttributes attr{};
  KVR_CUDA(cudaPointerGetAttributes(&attr, p));
  const bool dev = attr.type == cudaMemoryTypeDevice || attr.type == cudaMemoryTypeManaged;
  if ((on_device != 0) != dev)
    return fail(KVR_ERR_INVALID_ARG, "on_device=%d does not match the artifact pointer", on_device);
  *view = dev ? static_cast<char*>(const_cast<void*>(p))
              : (attr.type == cudaMemoryTypeHost ? static_cast<char*>(attr.devicePointer) : nullptr);
  return KVR_OK;
}

kvr_status q8_view_ok(const char* view) {
  if (!view) return fail(KVR_ERR_UNSUPPORTED, "an int8 artifact in host memory must be pinned (cudaHostAlloc / pin_memory)");
  if (!aligned16(view)) return fail(KVR_ERR_INVALID_ARG, "an int8 artifact must be 16-byte aligned");
  return KVR_OK;
}

// ---- artifact container header: explicit little-endian fields ----
void put_u32(uint8_t* p, uint32_t v) {
  for (int i = 0; i < 4; ++i) p[i] = static_cast<uint8_t>(v >> (8 * i));
}
void put_u64(uint8_t* p, uint64_t v) {
  for (int i = 0; i < 8; ++i) p[i] = static_cast<uint8_t>(v >> (8 * i));
}
uint32_t get_u32(const uint8_t* p) {
  uint32_t v = 0;
  for (int i = 0; i < 4; ++i) v |= static_cast<uint32_t>(p[i]) << (8 * i);
  return v;
}
uint64_t get_u64(const uint8_t* p) {
  uint64_t v = 0;
  for (int i = 0; i < 8; ++i) v |= static_cast<uint64_t>(p[i]) << (8 * i);
  return v;
}
const uint8_t kArtifactMagic[4] = {'K', 'V', 'R', 'A'};
constexpr uint32_t kArtifactVersion = 1;

}  // namespace

extern "C" {

size_t kvr_artifact_bytes(const kvr_model_desc* d, uint32_t L) {
  const char* why;
  if (!desc_ok(d, &why)) return 0;
  return static_cast<size_t>(d->layers) * 2 * d->n_kv_heads * L * d->head_dim * 2;
}

size_t kvr_artifact_bytes_q8(const kvr_model_desc* d, uint32_t L) {
  const char* why;
  if (!desc_ok(d, &why)) return 0;
  return q8_scale_bytes(*d) + static_cast<size_t>(d->layers) * 2 * d->n_kv_heads * L * d->head_dim;
}

size_t kvr_page_bytes(const kvr_model_desc* d) {
  const char* why;
  if (!desc_ok(d, &why)) return 0;
  return static_cast<size_t>(d->layers) * 2 * d->n_kv_heads * kPageTokens * d->head_dim * 2;
}

kvr_status kvr_artifact_write_header(const kvr_model_desc* d, const kvr_artifact_meta* meta, void* header) {
  const char* why;
  if (!d || !meta || !header) return fail(KVR_ERR_INVALID_ARG, "null argument");
  if (!desc_ok(d, &why)) return fail(KVR_ERR_INVALID_ARG, "bad model desc: %s", why);
  if (meta->model_id != d->model_id || (meta->dtype != d->dtype && meta->dtype != KVR_DTYPE_Q8))
    return fail(KVR_ERR_INVALID_ARG, "artifact metadata does not belong to this model");
  uint8_t* h = static_cast<uint8_t*>(header);
  std::memset(h, 0, KVR_ARTIFACT_HEADER_BYTES);
  std::memcpy(h, kArtifactMagic, 4);
  put_u32(h + 4, kArtifactVersion);
  put_u64(h + 8, meta->model_id);
  put_u32(h + 16, meta->dtype);
  put_u32(h + 20, meta->L);
  put_u32(h + 24, d->layers);
  put_u32(h + 28, d->n_kv_heads);
  put_u32(h + 32, d->head_dim);
  put_u64(h + 40, payload_bytes_of(d, meta->dtype, meta->L));
  return KVR_OK;
}

kvr_status kvr_artifact_read_header(const kvr_model_desc* d, const void* header, kvr_artifact_meta* meta_out,
                                    uint64_t* payload_bytes) {
  const char* why;
  if (!d || !header) return fail(KVR_ERR_INVALID_ARG, "null argument");
  if (!desc_ok(d, &why)) return fail(KVR_ERR_INVALID_ARG, "bad model desc: %s", why);
  const uint8_t* h = static_cast<const uint8_t*>(header);
  if (std::memcmp(h, kArtifactMagic, 4) != 0) return fail(KVR_ERR_INVALID_ARG, "not a kvr artifact (bad magic)");
  if (get_u32(h + 4) != kArtifactVersion)
    return fail(KVR_ERR_INVALID_ARG, "artifact container version %u is not supported", get_u32(h + 4));
  kvr_artifact_meta m;
  m.model_id = get_u64(h + 8);
  m.dtype = get_u32(h + 16);
  m.L = get_u32(h + 20);
  if (m.model_id != d->model_id || (m.dtype != d->dtype && m.dtype != KVR_DTYPE_Q8))
    return fail(KVR_ERR_META_MISMATCH, "artifact is for model %llu dtype %u, context is model %llu dtype %u",
                static_cast<unsigned long long>(m.model_id), m.dtype,
                static_cast<unsigned long long>(d->model_id), d->dtype);
  if (get_u32(h + 24) != d->layers || get_u32(h + 28) != d->n_kv_heads || get_u32(h + 32) != d->head_dim)
    return fail(KVR_ERR_META_MISMATCH, "artifact shape (%u layers, %u KV heads, d %u) differs from the model's",
                get_u32(h + 24), get_u32(h + 28), get_u32(h + 32));
  const uint64_t payload = get_u64(h + 40);
  if (payload != payload_bytes_of(d, m.dtype, m.L))
    return fail(KVR_ERR_INVALID_ARG, "payload of %llu bytes does not match L = %u",
                static_cast<unsigned long long>(payload), m.L);
  if (meta_out) *meta_out = m;
  if (payload_bytes) *payload_bytes = payload;
  return KVR_OK;
}

static size_t header_bytes(const kvr_model_desc* d, uint32_t max_seqs, size_t ws) {
  const uint32_t max_pages = (d->max_positions + kPageTokens - 1) / kPageTokens;
  size_t off = kAlign;  // error word
  off += align_up(static_cast<size_t>(d->layers) * 2 * sizeof(uint32_t), kAlign);
  off += align_up(static_cast<size_t>(max_seqs) * max_pages * sizeof(int32_t), kAlign);
  off += align_up(static_cast<size_t>(max_seqs) * max_pages * sizeof(int32_t), kAlign);  // int8-copy table
  off += align_up(static_cast<size_t>(max_seqs) * d->layers * 2 * sizeof(float), kAlign);  // their scales
  off += align_up(static_cast<size_t>(d->n_kv_heads) * kDecodeMaxClusters * decode_part_floats(d->head_dim) *
                      sizeof(float), kAlign);  // decode cluster partials
  off += align_up(static_cast<size_t>(d->n_kv_heads) * kDecodeMaxSplits * sizeof(int), kAlign);  // their counts
  off += align_up(static_cast<size_t>(d->max_positions) * (d->head_dim / 2) * sizeof(float2), kAlign);
  off += align_up(ws, kAlign);
  return align_up(off, kPageAlign);
}

size_t kvr_pool_bytes(const kvr_model_desc* d, uint32_t max_seqs, uint32_t n_pages, size_t ws) {
  const char* why;
  if (!desc_ok(d, &why) || max_seqs == 0) return 0;
  if (ws == 0) ws = kDefaultWorkspace;
  return header_bytes(d, max_seqs, ws) + static_cast<size_t>(n_pages) * kvr_page_bytes(d);
}

const char* kvr_status_string(kvr_status s) {
  switch (s) {
    case KVR_OK: return "ok";
    case KVR_ERR_INVALID_ARG: return "invalid argument";
    case KVR_ERR_META_MISMATCH: return "artifact metadata does not match the model";
    case KVR_ERR_POSITION: return "position does not continue the cached length";
    case KVR_ERR_OOM: return "out of pages, sequence slots or workspace";
    case KVR_ERR_UNSUPPORTED: return "unsupported";
    case KVR_ERR_TIMEOUT: return "device wait timed out";
    case KVR_ERR_CUDA: return "CUDA error";
    case KVR_ERR_DEVICE: return "device bounds check failed";
  }
  return "unknown status";
}

const char* kvr_last_error(void) { return g_last_error.c_str(); }

int kvr_version(void) { return 100; }

kvr_status kvr_create(const kvr_model_desc* desc, void* pool, size_t pool_bytes, uint32_t max_seqs,
                      size_t workspace_bytes, kvr_stream stream, kvr_ctx** out) {
  const char* why = nullptr;
  if (!out) return fail(KVR_ERR_INVALID_ARG, "null out");
  *out = nullptr;
  if (!desc_ok(desc, &why)) return fail(KVR_ERR_INVALID_ARG, "%s", why);
  if (!pool || (reinterpret_cast<uintptr_t>(pool) % kAlign))
    return fail(KVR_ERR_INVALID_ARG, "pool must be a non-null 256-byte aligned device pointer");
  if (max_seqs == 0 || max_seqs > (1u << 20)) return fail(KVR_ERR_INVALID_ARG, "max_seqs must be in [1, 2^20]");
  if (workspace_bytes == 0) workspace_bytes = kDefaultWorkspace;
  const size_t page_bytes = kvr_page_bytes(desc);
  const size_t head = header_bytes(desc, max_seqs, workspace_bytes);
  if (pool_bytes < head + page_bytes)
    return fail(KVR_ERR_OOM, "pool too small: %zu bytes, need at least %zu", pool_bytes, head + page_bytes);
  cudaPointerAttributes attr{};
  KVR_CUDA(cudaPointerGetAttributes(&attr, pool));
  if (attr.type != cudaMemoryTypeDevice) return fail(KVR_ERR_INVALID_ARG, "pool must be device memory");
  int dev = 0;
  KVR_CUDA(cudaGetDevice(&dev));
  if (attr.device != dev) return fail(KVR_ERR_INVALID_ARG, "pool lives on device %d, current device is %d", attr.device, dev);
  int major = 0, minor = 0;
  KVR_CUDA(cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev));
  KVR_CUDA(cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev));
  if (major != 10 || minor != 3)
    return fail(KVR_ERR_UNSUPPORTED, "this library is built for sm_103a (GB300); device is sm_%d%d", major, minor);

  kvr_ctx* c = new kvr_ctx();
  c->desc = *desc;
  c->device = dev;
  KVR_CUDA(cudaDeviceGetAttribute(&c->num_sms, cudaDevAttrMultiProcessorCount, dev));
  c->pool = static_cast<char*>(pool);
  c->pool_bytes = pool_bytes;
  c->max_seqs = max_seqs;
  c->max_pages = (desc->max_positions + kPageTokens - 1) / kPageTokens;
  c->page_bytes = page_bytes;
  size_t off = 0;
  c->d_err = reinterpret_cast<int*>(c->pool + off);
  off += kAlign;
  c->d_amax = reinterpret_cast<uint32_t*>(c->pool + off);
  off += align_up(static_cast<size_t>(desc->layers) * 2 * sizeof(uint32_t), kAlign);
  c->d_page_table = reinterpret_cast<int32_t*>(c->pool + off);
  off += align_up(static_cast<size_t>(max_seqs) * c->max_pages * sizeof(int32_t), kAlign);
  c->d_q8_table = reinterpret_cast<int32_t*>(c->pool + off);
  off += align_up(static_cast<size_t>(max_seqs) * c->max_pages * sizeof(int32_t), kAlign);
  c->d_q8_scales = reinterpret_cast<float*>(c->pool + off);
  off += align_up(static_cast<size_t>(max_seqs) * desc->layers * 2 * sizeof(float), kAlign);
  c->d_dpart = reinterpret_cast<float*>(c->pool + off);
  off += align_up(static_cast<size_t>(desc->n_kv_heads) * kDecodeMaxClusters *
                      decode_part_floats(static_cast<int>(desc->head_dim)) * sizeof(float),
                  kAlign);
  c->d_dcnt = reinterpret_cast<int*>(c->pool + off);
  off += align_up(static_cast<size_t>(desc->n_kv_heads) * kDecodeMaxSplits * sizeof(int), kAlign);
  c->d_rope = reinterpret_cast<float2*>(c->pool + off);
  off += align_up(static_cast<size_t>(desc->max_positions) * (desc->head_dim / 2) * sizeof(float2), kAlign);
  c->d_ws = reinterpret_cast<float*>(c->pool + off);
  c->ws_bytes = workspace_bytes;
  off += align_up(workspace_bytes, kAlign);
  off = align_up(off, kPageAlign);
  c->d_pages = c->pool + off;
  c->n_pages = static_cast<int64_t>((pool_bytes - off) / page_bytes);
  const int64_t rows_per_page = static_cast<int64_t>(desc->layers) * 2 * desc->n_kv_heads * kPageTokens;
  const int64_t max_rows = (int64_t(1) << 31) - 1;
  if (c->n_pages * rows_per_page > max_rows) c->n_pages = max_rows / rows_per_page;
  if (c->n_pages > (int64_t(1) << 30)) c->n_pages = int64_t(1) << 30;
  c->n_pool_rows = c->n_pages * rows_per_page;
  c->h_table.assign(static_cast<size_t>(max_seqs) * c->max_pages, -1);
  c->h_q8_table.assign(static_cast<size_t>(max_seqs) * c->max_pages, -1);
  c->seqs.resize(max_seqs);
  c->page_ref.assign(static_cast<size_t>(c->n_pages), 0);
  c->free_pages.reserve(static_cast<size_t>(c->n_pages));
  for (int64_t p = c->n_pages - 1; p >= 0; --p) c->free_pages.push_back(static_cast<int32_t>(p));

  kvr_status s = encode_rows_map(&c->tm_kv, c->d_pages, c->n_pool_rows, static_cast<int>(desc->head_dim), kPageTokens);
  if (s == KVR_OK) s = encode_rows_map(&c->tm_kv32, c->d_pages, c->n_pool_rows, static_cast<int>(desc->head_dim), 32);
  c->q8_ok = 2 * c->n_pool_rows <= (int64_t(1) << 31) - 1;
  if (s == KVR_OK && c->q8_ok)
    s = encode_q8_map(&c->tm_q8, c->d_pages, 2 * c->n_pool_rows, static_cast<int>(desc->head_dim));
  if (s == KVR_OK && c->q8_ok)  // pool bytes / 128 = n_pool_rows * d / 64 <= 2 n_pool_rows
    s = encode_q8t_map(&c->tm_q8t, c->d_pages, c->n_pool_rows * static_cast<int64_t>(desc->head_dim) / 64,
                       static_cast<int>(desc->head_dim));
  if (s != KVR_OK) { delete c; return s; }
  // RoPE table: angle = p * theta^(-2i/d) in fp64, cos/sin stored fp32.
  const int half = static_cast<int>(desc->head_dim / 2);
  std::vector<float2> rope(static_cast<size_t>(desc->max_positions) * half);
  std::vector<double> inv_freq(half);
  for (int i = 0; i < half; ++i)
    inv_freq[i] = std::pow(desc->rope_theta, -2.0 * i / static_cast<double>(desc->head_dim));
  for (uint32_t p = 0; p < desc->max_positions; ++p)
    for (int i = 0; i < half; ++i) {
      const double ang = static_cast<double>(p) * inv_freq[i];
      rope[static_cast<size_t>(p) * half + i] = make_float2(static_cast<float>(std::cos(ang)),
                                                            static_cast<float>(std::sin(ang)));
    }
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  cudaError_t e = cudaMemcpyAsync(c->d_rope, rope.data(), rope.size() * sizeof(float2), cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess) e = cudaMemsetAsync(c->d_err, 0, sizeof(int), st);
  if (e == cudaSuccess)
    e = cudaMemsetAsync(c->d_page_table, 0xff, static_cast<size_t>(max_seqs) * c->max_pages * sizeof(int32_t), st);
  if (e == cudaSuccess)
    e = cudaMemsetAsync(c->d_q8_table, 0xff, static_cast<size_t>(max_seqs) * c->max_pages * sizeof(int32_t), st);
  if (e == cudaSuccess)
    e = cudaMemsetAsync(c->d_dcnt, 0, static_cast<size_t>(desc->n_kv_heads) * kDecodeMaxSplits * sizeof(int), st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) { delete c; return cuda_fail(e, "context upload"); }
  *out = c;
  return KVR_OK;
}

kvr_status kvr_destroy(kvr_ctx* c) {
  if (!c) return fail(KVR_ERR_INVALID_ARG, "null ctx");
  delete c;
  return KVR_OK;
}

kvr_status kvr_free_pages(const kvr_ctx* c, uint32_t* n) {
  if (!c || !n) return fail(KVR_ERR_INVALID_ARG, "null argument");
  *n = static_cast<uint32_t>(c->free_pages.size());
  return KVR_OK;
}

kvr_status kvr_launch_count(const kvr_ctx* c, uint64_t* n) {
  if (!c || !n) return fail(KVR_ERR_INVALID_ARG, "null argument");
  *n = c->launches;
  return KVR_OK;
}

kvr_status kvr_sync_status(kvr_ctx* c, kvr_stream stream) {
  if (!c) return fail(KVR_ERR_INVALID_ARG, "null ctx");
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  KVR_CUDA(cudaStreamSynchronize(st));
  int h = 0;
  KVR_CUDA(cudaMemcpy(&h, c->d_err, sizeof(int), cudaMemcpyDeviceToHost));
  if (h == 0) return KVR_OK;
  KVR_CUDA(cudaMemset(c->d_err, 0, sizeof(int)));
  if (h & kDevErrTimeout) return fail(KVR_ERR_TIMEOUT, "a device-side wait passed its time limit (error word 0x%x)", h);
  return fail(KVR_ERR_DEVICE, "a device-side bounds check fired (error word 0x%x)", h);
}

kvr_status kvr_selftest_wait_timeout(kvr_ctx* c, kvr_stream stream) {
  if (!c) return fail(KVR_ERR_INVALID_ARG, "null ctx");
  KVR_CUDA(launch_kernel(wait_timeout_kernel, dim3(1), dim3(32), 0, reinterpret_cast<cudaStream_t>(stream), 0,
                         c->d_err));
  ++c->launches;
  return KVR_OK;
}

kvr_status kvr_seq_open(kvr_ctx* c, kvr_seq* out) {
  if (!c || !out) return fail(KVR_ERR_INVALID_ARG, "null argument");
  const int s = find_free_slot(c);
  if (s < 0) return fail(KVR_ERR_OOM, "no free sequence slot (max_seqs = %u)", c->max_seqs);
  Seq& q = c->seqs[s];
  q = Seq();
  q.used = true;
  q.root = true;
  q.family = c->next_family++;
  write_row(c, s);  // nothing to upload: an empty row is never read
  *out = s;
  return KVR_OK;
}

kvr_status kvr_seq_fork(kvr_ctx* c, kvr_seq parent, kvr_stream stream, kvr_seq* out) {
  if (!out) return fail(KVR_ERR_INVALID_ARG, "null out");
  Seq* p = get_seq(c, parent);
  if (!p) return fail(KVR_ERR_INVALID_ARG, "unknown parent sequence %d", parent);
  const uint32_t nfull = p->len / kPageTokens;
  const bool partial = (p->len % kPageTokens) != 0;
  if (partial && c->free_pages.empty()) return fail(KVR_ERR_OOM, "no free page for the forked tail");
  const int s = find_free_slot(c);
  if (s < 0) return fail(KVR_ERR_OOM, "no free sequence slot (max_seqs = %u)", c->max_seqs);
  p = &c->seqs[parent];
  Seq& q = c->seqs[s];
  q = Seq();
  q.used = true;
  q.root = false;
  q.len = p->len;
  q.family = p->family;
  q.n_shared = std::min(shared_with_root(c, *p), nfull);
  for (uint32_t i = 0; i < nfull; ++i) {
    q.pages.push_back(p->pages[i]);
    ++c->page_ref[p->pages[i]];
  }
  for (uint32_t i = 0; i < nfull && i < p->q8_pages.size(); ++i) {
    q.q8_pages.push_back(p->q8_pages[i]);
    ++c->page_ref[p->q8_pages[i]];
  }
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (!q.q8_pages.empty()) {
    const size_t nsc = static_cast<size_t>(c->desc.layers) * 2;
    cudaError_t e = cudaMemcpyAsync(c->d_q8_scales + static_cast<size_t>(s) * nsc,
                                    c->d_q8_scales + static_cast<size_t>(parent) * nsc, nsc * sizeof(float),
                                    cudaMemcpyDeviceToDevice, st);
    kvr_status r = e == cudaSuccess ? upload_q8_row(c, s, st) : cuda_fail(e, "fork scales");
    if (r != KVR_OK) {
      for (int32_t pg : q.pages) release_page(c, pg);
      for (int32_t pg : q.q8_pages) release_page(c, pg);
      q = Seq();
      return r;
    }
  }
  if (partial) {
    const int32_t np = alloc_page(c);
    q.pages.push_back(np);
    cudaError_t e = cudaMemcpyAsync(c->d_pages + static_cast<size_t>(np) * c->page_bytes,
                                    c->d_pages + static_cast<size_t>(p->pages[nfull]) * c->page_bytes,
                                    c->page_bytes, cudaMemcpyDeviceToDevice, st);
    if (e != cudaSuccess) {
      for (int32_t pg : q.pages) release_page(c, pg);
      for (int32_t pg : q.q8_pages) release_page(c, pg);
      q = Seq();
      return cuda_fail(e, "fork copy");
    }
  }
  write_row(c, s);
  kvr_status r = upload_rows(c, s, s, st);
  if (r != KVR_OK) return r;
  *out = s;
  return KVR_OK;
}

kvr_status kvr_seq_close(kvr_ctx* c, kvr_seq s) {
  Seq* q = get_seq(c, s);
  if (!q) return fail(KVR_ERR_INVALID_ARG, "unknown sequence %d", s);
  for (int32_t p : q->pages) release_page(c, p);
  for (int32_t p : q->q8_pages) release_page(c, p);
  *q = Seq();
  write_row(c, s);
  return KVR_OK;
}

kvr_status kvr_seq_length(const kvr_ctx* c, kvr_seq s, uint32_t* len) {
  if (!c || !len || s < 0 || static_cast<uint32_t>(s) >= c->max_seqs || !c->seqs[s].used)
    return fail(KVR_ERR_INVALID_ARG, "unknown sequence %d", s);
  *len = c->seqs[s].len;
  return KVR_OK;
}

kvr_status kvr_seq_reserve(kvr_ctx* c, int n, const kvr_seq* seqs, const int32_t* n_tokens, kvr_stream stream) {
  if (!c || n < 0 || (n > 0 && (!seqs || !n_tokens))) return fail(KVR_ERR_INVALID_ARG, "bad arguments");
  std::vector<uint32_t> need(n);
  for (int b = 0; b < n; ++b) {
    Seq* q = get_seq(c, seqs[b]);
    if (!q || n_tokens[b] < 0) return fail(KVR_ERR_INVALID_ARG, "bad sequence %d or count", seqs[b]);
    need[b] = q->len + static_cast<uint32_t>(n_tokens[b]);
  }
  return ensure_capacity(c, n, seqs, need.data(), reinterpret_cast<cudaStream_t>(stream), /*writes=*/false);
}

kvr_status kvr_seq_advance(kvr_ctx* c, int n, const kvr_seq* seqs, const int32_t* n_tokens) {
  if (!c || n < 0 || (n > 0 && (!seqs || !n_tokens))) return fail(KVR_ERR_INVALID_ARG, "bad arguments");
  for (int b = 0; b < n; ++b) {
    Seq* q = get_seq(c, seqs[b]);
    if (!q || n_tokens[b] < 0) return fail(KVR_ERR_INVALID_ARG, "bad sequence %d or count", seqs[b]);
    if (static_cast<size_t>(q->len) + n_tokens[b] > q->pages.size() * kPageTokens)
      return fail(KVR_ERR_POSITION, "sequence %d: advancing past the appended positions", seqs[b]);
  }
  for (int b = 0; b < n; ++b) c->seqs[seqs[b]].len += static_cast<uint32_t>(n_tokens[b]);
  return KVR_OK;
}

// Artifact [layers][2][Hkv][L][d] <-> pages: one 2D copy per page moves the
// page's positions of all (layer, K/V, head) rows at once.
static ArtifactArgs artifact_args(kvr_ctx* c, kvr_seq s, uint32_t L, char* view, bool q8) {
  ArtifactArgs a{};
  a.pages = c->d_pages;
  a.table = c->d_page_table + static_cast<size_t>(s) * c->max_pages;
  a.n_pages = c->n_pages;
  a.layers = static_cast<int>(c->desc.layers);
  a.Hkv = static_cast<int>(c->desc.n_kv_heads);
  a.d = static_cast<int>(c->desc.head_dim);
  a.L = static_cast<int>(L);
  if (q8) {
    a.scales = reinterpret_cast<float*>(view);
    a.codes = reinterpret_cast<int8_t*>(view + q8_scale_bytes(c->desc));
  } else {
    a.art = view;
  }
  a.amax = c->d_amax;
  a.err = c->d_err;
  return a;
}

// bf16 artifact <-> pages of sequence s.  Device or pinned host memory
// (`view` non-null and 16-byte aligned): one tile-copy kernel.  Pageable host
// memory: the copy engine, one 2-D copy per page.
static kvr_status copy_artifact(kvr_ctx* c, kvr_seq s, uint32_t L, char* art, char* view, bool to_pages,
                                cudaStream_t st) {
  if (L == 0) return KVR_OK;
  if (view && aligned16(view)) {
    const cudaError_t e = launch_artifact_copy(artifact_args(c, s, L, view, false), to_pages, st);
    if (e != cudaSuccess) return cuda_fail(e, "artifact copy");
    ++c->launches;
    return KVR_OK;
  }
  const Seq& q = c->seqs[s];
  const kvr_model_desc& d = c->desc;
  const size_t rowb = static_cast<size_t>(d.head_dim) * 2;
  const size_t height = static_cast<size_t>(d.layers) * 2 * d.n_kv_heads;
  for (uint32_t pi = 0; pi * kPageTokens < L; ++pi) {
    const uint32_t ntok = std::min<uint32_t>(kPageTokens, L - pi * kPageTokens);
    char* page = c->d_pages + static_cast<size_t>(q.pages[pi]) * c->page_bytes;
    char* a = art + static_cast<size_t>(pi) * kPageTokens * rowb;
    const size_t apitch = static_cast<size_t>(L) * rowb, ppitch = kPageTokens * rowb;
    cudaError_t e = to_pages
        ? cudaMemcpy2DAsync(page, ppitch, a, apitch, ntok * rowb, height, cudaMemcpyDefault, st)
        : cudaMemcpy2DAsync(a, apitch, page, ppitch, ntok * rowb, height, cudaMemcpyDefault, st);
    if (e != cudaSuccess) return cuda_fail(e, "artifact copy");
  }
  return KVR_OK;
}

kvr_status kvr_load_kv(kvr_ctx* c, const kvr_artifact_meta* meta, const void* artifact, int on_device,
                       kvr_stream stream, kvr_seq* out) {
  if (!c || !meta || !out) return fail(KVR_ERR_INVALID_ARG, "null argument");
  const bool q8 = meta->dtype == KVR_DTYPE_Q8;
  if (meta->model_id != c->desc.model_id || (meta->dtype != c->desc.dtype && !q8))
    return fail(KVR_ERR_META_MISMATCH,
                "artifact was produced for model %llu dtype %u; this context runs model %llu dtype %u",
                static_cast<unsigned long long>(meta->model_id), meta->dtype,
                static_cast<unsigned long long>(c->desc.model_id), c->desc.dtype);
  if (meta->L > c->desc.max_positions)
    return fail(KVR_ERR_INVALID_ARG, "artifact length %u exceeds max_positions %u", meta->L, c->desc.max_positions);
  if (meta->L > 0 && !artifact) return fail(KVR_ERR_INVALID_ARG, "null artifact");
  char* view = nullptr;
  if (meta->L > 0) {
    kvr_status r = artifact_view(artifact, on_device, &view);
    if (r == KVR_OK && q8) r = q8_view_ok(view);
    if (r != KVR_OK) return r;
  }
  kvr_seq s;
  kvr_status r = kvr_seq_open(c, &s);
  if (r != KVR_OK) return r;
  const uint32_t need = meta->L;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  r = ensure_capacity(c, 1, &s, &need, st);
  if (r != KVR_OK) { kvr_seq_close(c, s); return r; }
  if (q8) {
    const cudaError_t e = launch_q8_load(artifact_args(c, s, meta->L, view, true), st);
    if (e != cudaSuccess) { kvr_seq_close(c, s); return cuda_fail(e, "int8 artifact load"); }
    if (meta->L > 0) ++c->launches;
  } else {
    r = copy_artifact(c, s, meta->L, static_cast<char*>(const_cast<void*>(artifact)), view, true, st);
    if (r != KVR_OK) { kvr_seq_close(c, s); return r; }
  }
  c->seqs[s].len = meta->L;
  *out = s;
  return KVR_OK;
}

kvr_status kvr_load_kv_q8_resident(kvr_ctx* c, const kvr_artifact_meta* meta, const void* artifact, int on_device,
                                   kvr_stream stream, kvr_seq* out) {
  if (!c || !meta || !out) return fail(KVR_ERR_INVALID_ARG, "null argument");
  if (meta->dtype != KVR_DTYPE_Q8) return fail(KVR_ERR_INVALID_ARG, "an int8-resident load takes a KVR_DTYPE_Q8 artifact");
  if (!c->q8_ok) return fail(KVR_ERR_UNSUPPORTED, "the pool is too large for int8 copies (2 x rows >= 2^31)");
  const uint32_t nfull = meta->L / kPageTokens;
  if (nfull > c->free_pages.size() ||
      nfull + (meta->L + kPageTokens - 1) / kPageTokens > c->free_pages.size())
    return fail(KVR_ERR_OOM, "page pool exhausted: an int8-resident load of %u positions needs %u pages", meta->L,
                nfull + (meta->L + kPageTokens - 1) / kPageTokens);
  // the bf16 cache (every other kernel reads it) -- validates everything else
  kvr_seq s;
  kvr_status r = kvr_load_kv(c, meta, artifact, on_device, stream, &s);
  if (r != KVR_OK) return r;
  if (nfull > 0) {
    char* view = nullptr;
    r = artifact_view(artifact, on_device, &view);
    if (r != KVR_OK) { kvr_seq_close(c, s); return r; }
    Seq& q = c->seqs[s];
    for (uint32_t i = 0; i < nfull; ++i) q.q8_pages.push_back(alloc_page(c));
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    r = upload_q8_row(c, s, st);
    if (r == KVR_OK) {
      ArtifactArgs a = artifact_args(c, s, meta->L, view, true);
      a.table = c->d_q8_table + static_cast<size_t>(s) * c->max_pages;
      a.n_tiles = static_cast<int>(nfull);
      cudaError_t e = launch_q8_codes_to_pages(a, st);
      const size_t nsc = static_cast<size_t>(c->desc.layers) * 2;
      if (e == cudaSuccess)
        e = cudaMemcpyAsync(c->d_q8_scales + static_cast<size_t>(s) * nsc, view, nsc * sizeof(float),
                            cudaMemcpyDefault, st);
      if (e != cudaSuccess) r = cuda_fail(e, "int8 copy of the prefix");
      else ++c->launches;
    }
    if (r != KVR_OK) { kvr_seq_close(c, s); return r; }
  }
  *out = s;
  return KVR_OK;
}

kvr_status kvr_export_kv(kvr_ctx* c, kvr_seq s, void* artifact, int on_device, kvr_stream stream,
                         kvr_artifact_meta* meta_out) {
  Seq* q = get_seq(c, s);
  if (!q) return fail(KVR_ERR_INVALID_ARG, "unknown sequence %d", s);
  if (q->len > 0 && !artifact) return fail(KVR_ERR_INVALID_ARG, "null artifact");
  char* view = nullptr;
  if (q->len > 0) {
    kvr_status r = artifact_view(artifact, on_device, &view);
    if (r != KVR_OK) return r;
  }
  kvr_status r = copy_artifact(c, s, q->len, static_cast<char*>(artifact), view, false,
                               reinterpret_cast<cudaStream_t>(stream));
  if (r != KVR_OK) return r;
  if (meta_out) {
    meta_out->model_id = c->desc.model_id;
    meta_out->dtype = c->desc.dtype;
    meta_out->L = q->len;
  }
  return KVR_OK;
}

kvr_status kvr_export_kv_q8(kvr_ctx* c, kvr_seq s, void* artifact, int on_device, kvr_stream stream,
                            kvr_artifact_meta* meta_out) {
  Seq* q = get_seq(c, s);
  if (!q) return fail(KVR_ERR_INVALID_ARG, "unknown sequence %d", s);
  if (q->len > 0) {
    if (!artifact) return fail(KVR_ERR_INVALID_ARG, "null artifact");
    char* view = nullptr;
    kvr_status r = artifact_view(artifact, on_device, &view);
    if (r == KVR_OK) r = q8_view_ok(view);
    if (r != KVR_OK) return r;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    KVR_CUDA(cudaMemsetAsync(c->d_amax, 0, static_cast<size_t>(c->desc.layers) * 2 * sizeof(uint32_t), st));
    const cudaError_t e = launch_q8_export(artifact_args(c, s, q->len, view, true), st);
    if (e != cudaSuccess) return cuda_fail(e, "int8 artifact export");
    c->launches += 2;
  }
  if (meta_out) {
    meta_out->model_id = c->desc.model_id;
    meta_out->dtype = KVR_DTYPE_Q8;
    meta_out->L = q->len;
  }
  return KVR_OK;
}

kvr_status kvr_append_kv(kvr_ctx* c, int layer, int n_seqs, const kvr_seq* seqs, const int32_t* start_pos,
                         const int32_t* cu_q, const void* q_pre, const void* k_pre, const void* v,
                         const void* q_norm_w, const void* k_norm_w, void* q_out, kvr_stream stream) {
  if (!c) return fail(KVR_ERR_INVALID_ARG, "null ctx");
  if (layer < 0 || static_cast<uint32_t>(layer) >= c->desc.layers)
    return fail(KVR_ERR_INVALID_ARG, "layer %d out of range", layer);
  if (n_seqs > 0 && !start_pos) return fail(KVR_ERR_INVALID_ARG, "null start_pos");
  BatchDesc bd;
  std::vector<kvr_seq> kept;
  std::vector<uint32_t> need;
  kvr_status r = build_batch(c, n_seqs, seqs, cu_q, start_pos, &bd, &kept, &need);
  if (r != KVR_OK) return r;
  if (bd.T == 0) return KVR_OK;
  const void* ptrs[] = {q_pre, k_pre, v, q_norm_w, k_norm_w, q_out};
  for (const void* p : ptrs)
    if (!p || !aligned16(p)) return fail(KVR_ERR_INVALID_ARG, "tensor pointers must be non-null and 16-byte aligned");
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  r = ensure_capacity(c, static_cast<int>(kept.size()), kept.data(), need.data(), st);
  if (r != KVR_OK) return r;
  AppendArgs a{};
  a.q_pre = static_cast<const uint16_t*>(q_pre);
  a.k_pre = static_cast<const uint16_t*>(k_pre);
  a.v = static_cast<const uint16_t*>(v);
  a.q_w = static_cast<const uint16_t*>(q_norm_w);
  a.k_w = static_cast<const uint16_t*>(k_norm_w);
  a.q_out = static_cast<uint16_t*>(q_out);
  a.rope = c->d_rope;
  a.max_positions = static_cast<int>(c->desc.max_positions);
  a.eps = static_cast<float>(c->desc.rms_eps);
  a.layer = layer;
  a.Hq = static_cast<int>(c->desc.n_q_heads);
  a.geom.pages = c->d_pages;
  a.geom.n_pages = c->n_pages;
  a.geom.layers = static_cast<int>(c->desc.layers);
  a.geom.Hkv = static_cast<int>(c->desc.n_kv_heads);
  a.geom.d = static_cast<int>(c->desc.head_dim);
  a.err = c->d_err;
  cudaError_t e = launch_append(a, bd, static_cast<int>(c->desc.head_dim), static_cast<int>(c->desc.n_kv_heads), st);
  if (e != cudaSuccess) return cuda_fail(e, "append launch");
  ++c->launches;
  return KVR_OK;
}

kvr_status kvr_decode_step(kvr_ctx* c, int layer, int n_seqs, const kvr_seq* seqs, const int32_t* start_pos,
                           const int32_t* cu_q, const void* q_pre, const void* k_pre, const void* v,
                           const void* q_norm_w, const void* k_norm_w, void* q_out, void* out, float* lse,
                           const kvr_attn_opts* opts, kvr_stream stream) {
  if (!c) return fail(KVR_ERR_INVALID_ARG, "null ctx");
  if (layer < 0 || static_cast<uint32_t>(layer) >= c->desc.layers)
    return fail(KVR_ERR_INVALID_ARG, "layer %d out of range", layer);
  if (n_seqs > 0 && !start_pos) return fail(KVR_ERR_INVALID_ARG, "null start_pos");
  BatchDesc bd;
  std::vector<kvr_seq> kept;
  std::vector<uint32_t> need;
  kvr_status r = build_batch(c, n_seqs, seqs, cu_q, start_pos, &bd, &kept, &need);
  if (r != KVR_OK) return r;
  if (bd.T == 0) return KVR_OK;
  const void* ptrs[] = {q_pre, k_pre, v, q_norm_w, k_norm_w, out};
  for (const void* p : ptrs)
    if (!p || !aligned16(p)) return fail(KVR_ERR_INVALID_ARG, "tensor pointers must be non-null and 16-byte aligned");
  if (q_out && !aligned16(q_out)) return fail(KVR_ERR_INVALID_ARG, "q_out must be 16-byte aligned");
  const kvr_model_desc& d = c->desc;
  const int G = static_cast<int>(d.n_q_heads / d.n_kv_heads);
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if ((!opts || opts->num_splits == 0) && bd.T * G <= kDecodeMaxRows) {
    r = ensure_capacity(c, static_cast<int>(kept.size()), kept.data(), need.data(), st);
    if (r != KVR_OK) return r;
    DecodeArgs da{};
    da.tm_kv32 = c->tm_kv32;
    da.tm_q8 = c->tm_q8;
    da.tm_q8t = c->tm_q8t;
    da.q8_table = c->d_q8_table;
    da.q8_scales = c->d_q8_scales;
    for (int k = 0; k < bd.n_seqs && k < kDecodeMaxRows; ++k)
      da.q8_n[k] = static_cast<int>(c->seqs[bd.slot[k]].q8_pages.size());
    da.out = static_cast<uint16_t*>(out);
    da.lse = lse;
    da.err = c->d_err;
    da.layer = layer;
    da.layers = static_cast<int>(d.layers);
    da.Hq = static_cast<int>(d.n_q_heads);
    da.Hkv = static_cast<int>(d.n_kv_heads);
    da.G = G;
    da.scale_log2 = static_cast<float>(1.4426950408889634 / std::sqrt(static_cast<double>(d.head_dim)));
    da.n_pool_rows = c->n_pool_rows;
    da.q_pre = static_cast<const uint16_t*>(q_pre);
    da.k_pre = static_cast<const uint16_t*>(k_pre);
    da.v_new = static_cast<const uint16_t*>(v);
    da.q_w = static_cast<const uint16_t*>(q_norm_w);
    da.k_w = static_cast<const uint16_t*>(k_norm_w);
    da.rope = c->d_rope;
    da.max_positions = static_cast<int>(d.max_positions);
    da.eps = static_cast<float>(d.rms_eps);
    da.q_out = static_cast<uint16_t*>(q_out);
    da.pages = c->d_pages;
    const SmallBatch sb = small_batch(bd);
    bool q8 = false;
    for (int k = 0; k < sb.n_seqs && k < kDecodeMaxRows; ++k) q8 = q8 || da.q8_n[k] > 0;
    da.n_splits = decode_splits(static_cast<int>(d.head_dim), da.Hkv, decode_units(sb), q8, &da.n_clusters,
                                &da.n_warps);
    da.part = c->d_dpart;
    da.cnt = c->d_dcnt;
    cudaError_t e = launch_decode(da, sb, static_cast<int>(d.head_dim), true, st);
    if (e != cudaSuccess) return cuda_fail(e, "decode step launch");
    ++c->launches;
    return KVR_OK;
  }
  if (!q_out)
    return fail(KVR_ERR_INVALID_ARG, "q_out is required when the batch has more than %d rows per KV head",
                kDecodeMaxRows);
  r = kvr_append_kv(c, layer, n_seqs, seqs, start_pos, cu_q, q_pre, k_pre, v, q_norm_w, k_norm_w, q_out, stream);
  if (r != KVR_OK) return r;
  return kvr_reuse_attn(c, layer, n_seqs, seqs, cu_q, q_out, out, lse, opts, stream);
}

kvr_status kvr_reuse_attn(kvr_ctx* c, int layer, int n_seqs, const kvr_seq* seqs, const int32_t* cu_q,
                          const void* q, void* out, float* lse, const kvr_attn_opts* opts, kvr_stream stream) {
  if (!c) return fail(KVR_ERR_INVALID_ARG, "null ctx");
  BatchDesc bd;
  std::vector<kvr_seq> kept;
  std::vector<uint32_t> need;
  kvr_status r = build_batch(c, n_seqs, seqs, cu_q, nullptr, &bd, &kept, &need);
  if (r != KVR_OK) return r;
  return run_attention(c, layer, bd, need, q, out, lse, opts, reinterpret_cast<cudaStream_t>(stream));
}

kvr_status kvr_prefill_attn(kvr_ctx* c, int layer, kvr_seq seq, int n_tokens, const void* q, void* out,
                            float* lse, const kvr_attn_opts* opts, kvr_stream stream) {
  if (!c) return fail(KVR_ERR_INVALID_ARG, "null ctx");
  if (n_tokens < 0) return fail(KVR_ERR_INVALID_ARG, "n_tokens must be >= 0");
  const int32_t cu[2] = {0, n_tokens};
  BatchDesc bd;
  std::vector<kvr_seq> kept;
  std::vector<uint32_t> need;
  kvr_status r = build_batch(c, 1, &seq, cu, nullptr, &bd, &kept, &need);
  if (r != KVR_OK) return r;
  return run_attention(c, layer, bd, need, q, out, lse, opts, reinterpret_cast<cudaStream_t>(stream));
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Reuse attention without any allocation by the caller or the library.
//
// Some callers cannot allocate device memory at the point where they run
// attention: code executing under another framework's allocator that forbids
// side allocations, a runtime that reserved all device memory up front, or a
// context created with a small pool whose split workspace is too small for the
// batch at hand.  kvr_reuse_attn_noalloc keeps the per-split partial results in
// a fixed array that lives in the library's own device image (below): the
// driver reserves it once per device when the library's module loads and holds
// it until the process exits; nothing is allocated per call.
namespace {

constexpr size_t kNoAllocScratchBytes = KVR_NOALLOC_SCRATCH_BYTES;
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

std::mutex g_noalloc_mu;
struct NoAllocAddr {
  CUcontext ctx;  // the context the address was looked up in
  void* addr;
};
NoAllocAddr g_noalloc_addr[kMaxDevices] = {};

PFN_cuCtxGetCurrent_v4000 get_ctx_current() {
  static PFN_cuCtxGetCurrent_v4000 fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 4000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuCtxGetCurrent_v4000>(p);
  }
  return fn;
}

// Device address of the scratch array on `dev` (the current device).  In host
// code the array's name only stands for the symbol; its device address comes
// from cudaGetSymbolAddress, looked up on a device's first call and again
// whenever the device's current context is a different one (after a device
// reset the module, and with it the array, may sit at a new address).
kvr_status noalloc_scratch_ptr(int dev, float** out) {
  if (dev < 0 || dev >= kMaxDevices) return fail(KVR_ERR_UNSUPPORTED, "device ordinal %d out of range", dev);
  auto ctx_current = get_ctx_current();
  if (!ctx_current) return fail(KVR_ERR_CUDA, "cuCtxGetCurrent is unavailable");
  CUcontext cur = nullptr;
  if (ctx_current(&cur) != CUDA_SUCCESS || cur == nullptr)
    return fail(KVR_ERR_CUDA, "no current CUDA context on device %d", dev);
  std::lock_guard<std::mutex> lock(g_noalloc_mu);
  NoAllocAddr& slot = g_noalloc_addr[dev];
  if (slot.addr == nullptr || slot.ctx != cur) {
    void* p = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress(no-alloc scratch)");
    if (p == nullptr) return fail(KVR_ERR_CUDA, "no-alloc scratch has no device address");
    slot.ctx = cur;
    slot.addr = p;
  }
  *out = static_cast<float*>(slot.addr);
  return KVR_OK;
}

kvr_status run_attention_noalloc(kvr_ctx* c, int layer, BatchDesc& bd, const std::vector<uint32_t>& need,
                                 const void* q, void* out, float* lse, const kvr_attn_opts* opts,
                                 cudaStream_t st) {
  const kvr_model_desc& d = c->desc;
  if (layer < 0 || static_cast<uint32_t>(layer) >= d.layers)
    return fail(KVR_ERR_INVALID_ARG, "layer %d out of range", layer);
  if (bd.T == 0) return KVR_OK;
  if (!q || !out) return fail(KVR_ERR_INVALID_ARG, "null q or out");
  if (!aligned16(q) || !aligned16(out)) return fail(KVR_ERR_INVALID_ARG, "q and out must be 16-byte aligned");
  for (int k = 0; k < bd.n_seqs; ++k) {
    const Seq& s = c->seqs[bd.slot[k]];
    if (s.pages.size() * kPageTokens < need[k])
      return fail(KVR_ERR_POSITION,
                  "sequence %d: rows reach position %u but only %zu positions were appended/reserved",
                  bd.slot[k], need[k] - 1, s.pages.size() * kPageTokens);
  }
  int dev = -1;
  KVR_CUDA(cudaGetDevice(&dev));
  if (dev != c->device) return fail(KVR_ERR_INVALID_ARG, "current device %d is not the context's device %d", dev, c->device);
  const int G = static_cast<int>(d.n_q_heads / d.n_kv_heads);
  const int TB = kBlockRows / G;
  AttnArgs a{};
  kvr_status s = encode_q_map(&a.tm_q, q, bd.T, static_cast<int>(d.n_q_heads), static_cast<int>(d.head_dim), G);
  if (s != KVR_OK) return s;
  a.tm_kv = c->tm_kv;
  a.layer = layer;
  a.layers = static_cast<int>(d.layers);
  a.Hq = static_cast<int>(d.n_q_heads);
  a.Hkv = static_cast<int>(d.n_kv_heads);
  a.G = G;
  a.n_rb = (bd.T + TB - 1) / TB;
  a.scale_log2 = static_cast<float>(1.4426950408889634 / std::sqrt(static_cast<double>(d.head_dim)));
  a.out = static_cast<uint16_t*>(out);
  a.lse = lse;
  a.err = c->d_err;
  a.n_pool_rows = c->n_pool_rows;
  uint32_t max_need = 0;
  for (uint32_t v : need) max_need = std::max(max_need, v);
  const int tiles = static_cast<int>((max_need + kPageTokens - 1) / kPageTokens);
  a.q_tiles = attention_q_tiles(a.n_rb, a.Hkv, c->num_sms, opts);
  const int units = (a.n_rb + a.q_tiles - 1) / a.q_tiles * a.Hkv;  // attention CTAs per split
  const size_t per_split = static_cast<size_t>(bd.T) * d.n_q_heads * (d.head_dim + 1) * sizeof(float);
  int S = 1;
  if (!opts || opts->num_splits == 0) {
    if (units < c->num_sms) S = std::min(std::max(1, c->num_sms / units), std::max(1, tiles / 2));
    S = std::min(S, 64);
    // automatic choice: as many splits as the fixed scratch holds
    if (S > 1 && per_split * S > kNoAllocScratchBytes) S = static_cast<int>(kNoAllocScratchBytes / per_split);
    if (S < 2) S = 1;
  } else if (opts->num_splits > 0) {
    S = std::min(std::min(opts->num_splits, std::max(1, tiles)), 64);
    if (S > 1 && per_split * S > kNoAllocScratchBytes)
      return fail(KVR_ERR_OOM,
                  "%d splits of %d rows need %zu bytes of scratch; the no-alloc scratch holds %zu bytes "
                  "(use fewer splits, or kvr_reuse_attn)",
                  S, bd.T * a.Hq, per_split * S, kNoAllocScratchBytes);
  } else {
    return fail(KVR_ERR_INVALID_ARG, "num_splits must be >= 0");
  }
  a.n_splits = S;
  if (S > 1) {
    float* scratch = nullptr;
    s = noalloc_scratch_ptr(dev, &scratch);
    if (s != KVR_OK) return s;
    a.part_o = scratch;
    a.part_lse = scratch + static_cast<size_t>(S) * bd.T * d.n_q_heads * d.head_dim;
  }
  cudaError_t e = launch_attention(a, bd, static_cast<int>(d.head_dim), st);
  if (e != cudaSuccess) return cuda_fail(e, "attention launch");
  ++c->launches;
  if (S > 1) {
    ++c->launches;
    e = launch_combine(a.part_o, a.part_lse, S, bd.T, a.Hq, static_cast<int>(d.head_dim),
                       static_cast<uint16_t*>(out), lse, st);
    if (e != cudaSuccess) return cuda_fail(e, "combine launch");
  }
  return KVR_OK;
}

}  // namespace

extern "C" kvr_status kvr_reuse_attn_noalloc(kvr_ctx* c, int layer, int n_seqs, const kvr_seq* seqs,
                                             const int32_t* cu_q, const void* q, void* out, float* lse,
                                             const kvr_attn_opts* opts, kvr_stream stream) {
  if (!c) return fail(KVR_ERR_INVALID_ARG, "null ctx");
  BatchDesc bd;
  std::vector<kvr_seq> kept;
  std::vector<uint32_t> need;
  kvr_status r = build_batch(c, n_seqs, seqs, cu_q, nullptr, &bd, &kept, &need);
  if (r != KVR_OK) return r;
  return run_attention_noalloc(c, layer, bd, need, q, out, lse, opts, reinterpret_cast<cudaStream_t>(stream));
}
