// kvr_internal.h -- structures shared by the host runtime and the kernels.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>
#include <mutex>

#include "../../include/kvr.h"

namespace kvr {

constexpr int kPageTokens = KVR_PAGE_TOKENS;  // tokens per page == key tile (Bc)
constexpr int kMaxBatch = KVR_MAX_BATCH;
constexpr int kBlockRows = 128;               // packed query rows per Q tile (MMA M)
constexpr int kQTiles = 2;                    // most Q tiles per attention CTA (they share each K/V tile)

// Device error word bits (kvr_sync_status maps them to kvr_status).
enum : int {
  kDevErrTimeout = 1,  // an mbarrier wait passed its time limit
  kDevErrBounds = 2,   // a page index or position was out of range
};

// Physical layout of the pool's page area: page p holds, for every layer l,
// K and V (kv = 0/1) of kv head g for its 128 positions:
//   row(p, l, kv, g, slot) = (((p * layers + l) * 2 + kv) * Hkv + g) * 128 + slot
// each row head_dim bf16 contiguous.  This is the row space the TMA map sees.
struct PoolGeom {
  char* pages;         // base of page area (bf16 rows of head_dim)
  int64_t n_pages;
  int layers, Hkv, d;
};

__host__ __device__ inline int64_t kv_row(int64_t page, int layer, int kv, int g, int layers,
                                          int Hkv) {
  return ((((page * layers + layer) * 2 + kv) * Hkv + g) * (int64_t)kPageTokens);
}

// Per-call description of a batch of sequences (passed by value to kernels),
// sized for N sequences.
template <int N>
struct BatchDescT {
  int n_seqs;
  int T;                     // packed tokens
  int shared_pages;          // leading pages common to every sequence
  int max_pages;             // page-table row stride
  const int32_t* page_table; // device [max_seqs][max_pages]
  int32_t slot[N];           // page-table row of sequence b
  int32_t start[N];          // position of its first packed token
  int32_t cu_q[N + 1];
};
using BatchDesc = BatchDescT<kMaxBatch>;

struct AppendArgs {
  const uint16_t* q_pre;
  const uint16_t* k_pre;
  const uint16_t* v;
  const uint16_t* q_w;
  const uint16_t* k_w;
  uint16_t* q_out;
  const float2* rope;  // [max_positions][d/2] (cos, sin)
  int max_positions;
  float eps;
  int layer;
  int Hq;
  PoolGeom geom;
  int* err;
};

struct AttnArgs {
  CUtensorMap tm_q;   // 3D over q [T][Hq][d], box (64, G, 128/G), 128B swizzle
  CUtensorMap tm_kv;  // 2D over the page rows [rows][d], box (64, 128), 128B swizzle
  int layer, layers, Hq, Hkv, G;
  int n_rb;           // query blocks of 128/G tokens
  int q_tiles;        // query blocks per CTA: 1 or kQTiles
  int n_splits;
  float scale_log2;   // log2(e) / sqrt(d)
  uint16_t* out;      // [T][Hq][d] bf16 (n_splits == 1)
  float* lse;         // [T][Hq] or null
  float* part_o;      // [n_splits][T][Hq][d] fp32 (n_splits > 1)
  float* part_lse;    // [n_splits][T][Hq] log2-domain
  int* err;
  int64_t n_pool_rows;
};

// Few-rows reuse attention (decode): at most kDecodeMaxRows packed rows
// (tokens x GQA group) per KV head, split merge in-kernel; its batches have at
// most kDecodeMaxRows sequences and travel in a small descriptor.
constexpr int kDecodeMaxRows = 8;
// Long contexts: a KV head's splits may span up to kDecodeMaxClusters clusters
// of at most kDecodeMaxSplits CTAs; cluster partials meet in the pool header.
constexpr int kDecodeMaxClusters = 4;
constexpr int kDecodeMaxSplits = 16;
// floats of one cluster partial: values [rows][d], then (max, sum) per
// [owner CTA][row]
__host__ __device__ constexpr int decode_part_floats(int d) {
  return kDecodeMaxRows * d + kDecodeMaxSplits * kDecodeMaxRows * 2;
}
using SmallBatch = BatchDescT<kDecodeMaxRows>;

inline SmallBatch small_batch(const BatchDesc& b) {
  SmallBatch s{};
  s.n_seqs = b.n_seqs;
  s.T = b.T;
  s.shared_pages = b.shared_pages;
  s.max_pages = b.max_pages;
  s.page_table = b.page_table;
  for (int i = 0; i < b.n_seqs && i < kDecodeMaxRows; ++i) {
    s.slot[i] = b.slot[i];
    s.start[i] = b.start[i];
    s.cu_q[i] = b.cu_q[i];
  }
  s.cu_q[b.n_seqs < kDecodeMaxRows ? b.n_seqs : kDecodeMaxRows] = b.cu_q[b.n_seqs];
  return s;
}

struct DecodeArgs {
  CUtensorMap tm_kv32;  // 2D over the page rows, box (64, 32), 128B swizzle
  const uint16_t* q;    // [T][Hq][d] bf16 (normed + roped)
  uint16_t* out;        // [T][Hq][d] bf16
  float* lse;           // [T][Hq] or null
  int* err;
  int layer, layers, Hq, Hkv, G;
  int n_splits;         // CTAs per KV head = cluster size (decode_splits)
  int n_warps;          // warps per CTA: 12 (or 0) or 6 (decode_splits)
  float scale_log2;
  int64_t n_pool_rows;
  // fused append (decode step): pre-norm inputs of the new tokens; the kernel
  // norms and ropes them itself, writes k, v to the cache and q to q_out
  const uint16_t* q_pre;  // [T][Hq][d]
  const uint16_t* k_pre;  // [T][Hkv][d]
  const uint16_t* v_new;  // [T][Hkv][d]
  const uint16_t* q_w;    // [d]
  const uint16_t* k_w;    // [d]
  const float2* rope;     // [max_positions][d/2]
  int max_positions;
  float eps;
  uint16_t* q_out;        // [T][Hq][d] or null
  char* pages;            // page area (cache rows of d bf16)
  // int8-resident prefixes: the first q8_n[b] pages of batch sequence b also
  // have an int8 copy (page q8_table[slot][i]), read instead of the bf16
  // page; scales fp32 [slot][layer][K|V].  An int8 page holds, per (layer,
  // K|V, head) block of 128 * d bytes at the block's bf16 row index * d,
  // the codes + 128 (bytes x ^ 0x80): K as [128 keys][d], V transposed as
  // [d][128 keys]
  CUtensorMap tm_q8;      // K: rows of d bytes, box (d, 32), 128B swizzle at d = 128
  CUtensorMap tm_q8t;     // V: rows of 128 bytes, box (32, d), no swizzle
  const int32_t* q8_table;
  const float* q8_scales;
  int q8_n[kDecodeMaxRows];
  // clusters per KV head (>= 1).  With more than one, each cluster's owner
  // CTA k leaves its slice in part [Hkv][kDecodeMaxClusters][part floats] and
  // counts itself in cnt [Hkv][kDecodeMaxSplits]; the last of the clusters to
  // arrive merges them in cluster order and resets the count to 0.
  int n_clusters;
  float* part;
  int* cnt;
};

// Projections of the whole layer (kvr_gemm.cu): D_s[T][N_s] = X[T][K]
// W_s[N_s][K]^T for up to kMaxGemmSegs weight matrices sharing X, plus a
// residual C[T][N_0] on segment 0; or, with swiglu, one W = [W_gate; W_up]
// ([2 I][K]) and D_0[T][I] = silu(X W_gate^T) * (X W_up^T).
constexpr int kMaxGemmSegs = 3;
struct GemmSeg {
  CUtensorMap tm_w;  // W_s [N_s][K] bf16, box (64, BN / 2), 128B swizzle
  uint16_t* D;       // [T][N_s] bf16 (swiglu: [T][I])
  int N;             // output columns (swiglu: I)
};
struct GemmArgs {
  CUtensorMap tm_x;  // X [T][K] bf16, box (64, 128), 128B swizzle
  GemmSeg seg[kMaxGemmSegs];
  int nseg, T, K;
  const uint16_t* C;  // residual [T][seg[0].N] or null
  int swiglu, I;
  int* err;
  // split-K (short batches whose output tiles alone would leave most SMs
  // idle): ksplit CTAs per output tile each sum a contiguous range of K into
  // fp32 partials part[ks][T][P] (P = the segments' widths side by side, or
  // gate then up columns: 2 I), which gemm_reduce adds in split order before
  // the epilogue's arithmetic.  ksplit = 1: no partials.
  int ksplit;
  float* part;
};
// Output tile width for a batch of T rows (the W maps' box is (64, width / 2)).
int gemm_tile_n(int T);
// Splits of K for a GEMM of T rows, K columns of X and `tiles` output tiles
// (1 when the tiles fill the GPU), at most max_split.
int gemm_ksplit(int T, int K, int tiles, int num_sms, int max_split);
int gemm_tiles(const GemmArgs& g);
cudaError_t launch_gemm(const GemmArgs& g, int num_sms, cudaStream_t st);
// 2-D tensor map over a row-major bf16 matrix [rows][inner] (row pitch
// inner * 2 bytes), box (box_inner, box_rows), 128-byte swizzle, zero fill
// out of bounds.  Defined in kvr_api.cu; returns the driver's CUresult.
int encode_bf16_2d(CUtensorMap* tm, const void* base, uint64_t inner, uint64_t rows, uint32_t box_inner,
                   uint32_t box_rows);

// Launch with programmatic stream serialization (the kernel waits for the
// previous one with griddepcontrol.wait before touching global memory) and,
// when cluster_x > 0, thread-block clusters of cluster_x CTAs along x.
template <typename... KArgs, typename... Args>
inline cudaError_t launch_kernel(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                                 unsigned cluster_x, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  unsigned n = 0;
  attr[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[n].val.programmaticStreamSerializationAllowed = 1;
  ++n;
  if (cluster_x > 0) {
    attr[n].id = cudaLaunchAttributeClusterDimension;
    attr[n].val.clusterDim.x = cluster_x;
    attr[n].val.clusterDim.y = 1;
    attr[n].val.clusterDim.z = 1;
    ++n;
  }
  cfg.attrs = attr;
  cfg.numAttrs = n;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args&&>(args)...);
}

// One-time, per-device setup of a kernel's attributes (cudaFuncSetAttribute
// acts on the current device only, so a context on a second device needs its
// own).  `run(f)` calls f() once per device ordinal, with that device current,
// until it succeeds; concurrent first calls from several threads are
// serialised, later calls take the lock-free fast path.
constexpr int kMaxDevices = 64;
struct PerDeviceOnce {
  std::atomic<bool> done[kMaxDevices] = {};
  std::mutex mu;
  template <typename F>
  cudaError_t run(F&& f) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    if (done[dev].load(std::memory_order_acquire)) return cudaSuccess;
    std::lock_guard<std::mutex> lock(mu);
    if (done[dev].load(std::memory_order_relaxed)) return cudaSuccess;
    e = f();
    if (e == cudaSuccess) done[dev].store(true, std::memory_order_release);
    return e;
  }
};

// Stage timestamps for latency analysis, compiled in only when KVR_STAGE_TRACE
// is defined (paper_2606_13361_gb300/stage_trace.py builds such a library;
// the product library carries none of it): KVR_STAGE(buf, layer, slot) stores
// %globaltimer into buf[layer % 40][blockIdx.x % 160][slot].
constexpr int kStageSlots = 32;
#ifdef KVR_STAGE_TRACE
#define KVR_STAGE_BUFFER(name) __device__ unsigned long long name[40][160][kStageSlots]
#define KVR_STAGE(buf, layer, slot)                                   \
  do {                                                                \
    unsigned long long t_;                                            \
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t_));            \
    buf[(layer) % 40][blockIdx.x % 160][slot] = t_;                   \
  } while (0)
#else
#define KVR_STAGE(buf, layer, slot) ((void)0)
#endif

// Launchers (defined in the .cu files).  Return a cudaError_t.
cudaError_t launch_decode(const DecodeArgs& a, const SmallBatch& b, int d, bool fused, cudaStream_t st);
int decode_units(const SmallBatch& b);
int decode_splits(int d, int heads, int units, bool q8, int* clusters, int* warps);
cudaError_t launch_append(const AppendArgs& a, const BatchDesc& b, int d, int Hkv,
                          cudaStream_t st);
cudaError_t launch_attention(const AttnArgs& a, const BatchDesc& b, int d, cudaStream_t st);
cudaError_t launch_combine(const float* part_o, const float* part_lse, int n_splits, int T,
                           int Hq, int d, uint16_t* out, float* lse, cudaStream_t st);
int attention_smem_bytes(int d);

}  // namespace kvr
