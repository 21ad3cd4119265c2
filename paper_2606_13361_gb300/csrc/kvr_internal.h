// kvr_internal.h -- structures shared by the host runtime and the kernels.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/kvr.h"

namespace kvr {

constexpr int kPageTokens = KVR_PAGE_TOKENS;  // tokens per page == key tile (Bc)
constexpr int kMaxBatch = KVR_MAX_BATCH;
constexpr int kBlockRows = 128;               // packed query rows per CTA (MMA M)

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

// Per-call description of a batch of sequences (passed by value to kernels).
struct BatchDesc {
  int n_seqs;
  int T;                     // packed tokens
  int shared_pages;          // leading pages common to every sequence
  int max_pages;             // page-table row stride
  const int32_t* page_table; // device [max_seqs][max_pages]
  int32_t slot[kMaxBatch];   // page-table row of sequence b
  int32_t start[kMaxBatch];  // position of its first packed token
  int32_t cu_q[kMaxBatch + 1];
};

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
// (tokens x GQA group) per KV head, on CUDA cores, split merge in-kernel.
constexpr int kDecodeMaxRows = 8;

struct DecodeArgs {
  CUtensorMap tm_kv32;  // 2D over the page rows, box (64, 32), 128B swizzle
  const uint16_t* q;    // [T][Hq][d] bf16 (normed + roped)
  uint16_t* out;        // [T][Hq][d] bf16
  float* lse;           // [T][Hq] or null
  int* err;
  int layer, layers, Hq, Hkv, G;
  int n_splits;         // CTAs per KV head = cluster size (decode_splits)
  float scale_log2;
  int64_t n_pool_rows;
};

// Launchers (defined in the .cu files).  Return a cudaError_t.
cudaError_t launch_decode(const DecodeArgs& a, const BatchDesc& b, int d, cudaStream_t st);
int decode_units(const BatchDesc& b);
int decode_splits(int d, int heads, int units);
cudaError_t launch_append(const AppendArgs& a, const BatchDesc& b, int d, int Hkv,
                          cudaStream_t st);
cudaError_t launch_attention(const AttnArgs& a, const BatchDesc& b, int d, cudaStream_t st);
cudaError_t launch_combine(const float* part_o, const float* part_lse, int n_splits, int T,
                           int Hq, int d, uint16_t* out, float* lse, cudaStream_t st);
int attention_smem_bytes(int d);

}  // namespace kvr
