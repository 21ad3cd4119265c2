// kvr_artifact.cu -- moving one sequence's cache between its pages and an
// artifact (Algorithm 1 stores (K, V) per layer; Algorithm 2 deserializes
// them; Sec. 3.3: the bf16 move is value-preserving), and the per-tensor
// symmetric int8 artifact of Sec. 5 "Quantizing the artifact".
//
// Artifact layout [layers][2][Hkv][L][d]; page layout: page p holds the 128
// positions of every (layer, K|V, head) as one contiguous run of 128 rows.
// Every kernel walks (page, layer, K|V, head) tiles: grid.x = the sequence's
// pages, grid.y = layers * 2 * Hkv; a tile is up to 128 contiguous cache rows
// of d bf16 (32 KB at d = 128) on both sides.  The work is a stream (HBM- or
// host-link-bound): 16-byte accesses, eight loads in flight per thread before
// the stores, no shared-memory staging beyond the block reduction.
//
// int8 readings (shared with the CPU oracle): a tensor is one layer's K or one
// layer's V over every KV head and position; s = max|x| / 127 and code =
// round-half-even(x / s) clamped to [-127, 127] (0 when s = 0), with the
// division an IEEE fp32 operation so that the integer decision is the same
// wherever it is taken; the loaded cache value is bf16(code * s), an fp32
// product rounded once.
#include "kvr_artifact.cuh"
#include "kvr_ptx.cuh"

namespace kvr {
namespace {

constexpr int kThreads = 256;
constexpr int kUnroll = 8;

struct Tile {
  int layer, kv, g, lk, ntok;
  int64_t row;       // first cache row of the tile
  int64_t art_elem;  // first artifact element of the tile
};

__device__ __forceinline__ bool tile_of(const ArtifactArgs& a, Tile& t) {
  const int pi = blockIdx.x;
  const int y = blockIdx.y;
  t.g = y % a.Hkv;
  t.lk = y / a.Hkv;
  t.layer = t.lk >> 1;
  t.kv = t.lk & 1;
  t.ntok = min(kPageTokens, a.L - pi * kPageTokens);
  const int page = a.table[pi];
  if (page < 0 || page >= a.n_pages) {
    if (threadIdx.x == 0) atomicOr(a.err, kDevErrBounds);
    return false;
  }
  t.row = kv_row(page, t.layer, t.kv, t.g, a.layers, a.Hkv);
  t.art_elem = ((static_cast<int64_t>(t.lk) * a.Hkv + t.g) * a.L + static_cast<int64_t>(pi) * kPageTokens) * a.d;
  return true;
}

// ------------------------------------------------------------ bf16 copy ----

template <bool kToPages>
__global__ void __launch_bounds__(kThreads) copy_kernel(const __grid_constant__ ArtifactArgs a) {
  griddep_wait();
  griddep_launch_dependents();
  Tile t;
  if (!tile_of(a, t)) return;
  uint4* page = reinterpret_cast<uint4*>(a.pages + t.row * a.d * 2);
  uint4* art = reinterpret_cast<uint4*>(a.art + t.art_elem * 2);
  const uint4* src = kToPages ? art : page;
  uint4* dst = kToPages ? page : art;
  const int nvec = t.ntok * a.d / 8;
  for (int base = threadIdx.x; base < nvec; base += kThreads * kUnroll) {
    uint4 r[kUnroll];
#pragma unroll
    for (int k = 0; k < kUnroll; ++k) {
      const int i = base + k * kThreads;
      if (i < nvec) r[k] = __ldcs(src + i);
    }
#pragma unroll
    for (int k = 0; k < kUnroll; ++k) {
      const int i = base + k * kThreads;
      if (i < nvec) dst[i] = r[k];
    }
  }
}

// ----------------------------------------------------------------- int8 ----

// Largest bf16 magnitude (bits with the sign cleared order like the values).
__device__ __forceinline__ uint32_t absmax_bits8(uint4 v) {
  uint32_t m = 0;
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) m = max(m, max(w[i] & 0x7fffu, (w[i] >> 16) & 0x7fffu));
  return m;
}

__device__ __forceinline__ uint32_t code_of(uint32_t bf16_bits, float s) {
  const float x = __uint_as_float(bf16_bits << 16);
  const float c = s > 0.0f ? fminf(fmaxf(rintf(__fdiv_rn(x, s)), -127.0f), 127.0f) : 0.0f;
  return static_cast<uint32_t>(static_cast<int>(c)) & 0xffu;
}

__global__ void __launch_bounds__(kThreads) q8_absmax_kernel(const __grid_constant__ ArtifactArgs a) {
  __shared__ uint32_t red[kThreads / 32];
  griddep_wait();
  griddep_launch_dependents();
  Tile t;
  uint32_t m = 0;
  const bool ok = tile_of(a, t);
  if (ok) {
    const uint4* src = reinterpret_cast<const uint4*>(a.pages + t.row * a.d * 2);
    const int nvec = t.ntok * a.d / 8;
    for (int i = threadIdx.x; i < nvec; i += kThreads) m = max(m, absmax_bits8(src[i]));
  }
  m = __reduce_max_sync(0xffffffffu, m);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = m;
  __syncthreads();
  if (threadIdx.x == 0 && ok) {
#pragma unroll
    for (int i = 0; i < kThreads / 32; ++i) m = max(m, red[i]);
    atomicMax(a.amax + t.lk, m);
  }
}

__global__ void __launch_bounds__(kThreads) q8_quant_kernel(const __grid_constant__ ArtifactArgs a) {
  griddep_wait();
  griddep_launch_dependents();
  Tile t;
  if (!tile_of(a, t)) return;
  const float s = __fdiv_rn(__uint_as_float(a.amax[t.lk] << 16), 127.0f);
  if (blockIdx.x == 0 && t.g == 0 && threadIdx.x == 0) a.scales[t.lk] = s;
  const uint4* src = reinterpret_cast<const uint4*>(a.pages + t.row * a.d * 2);
  uint2* dst = reinterpret_cast<uint2*>(a.codes + t.art_elem);
  const int nvec = t.ntok * a.d / 8;
  for (int i = threadIdx.x; i < nvec; i += kThreads) {
    const uint4 v = src[i];
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
    uint32_t c[8];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      c[2 * j] = code_of(w[j] & 0xffffu, s);
      c[2 * j + 1] = code_of(w[j] >> 16, s);
    }
    dst[i] = make_uint2(c[0] | c[1] << 8 | c[2] << 16 | c[3] << 24, c[4] | c[5] << 8 | c[6] << 16 | c[7] << 24);
  }
}

__global__ void __launch_bounds__(kThreads) q8_dequant_kernel(const __grid_constant__ ArtifactArgs a) {
  griddep_wait();
  griddep_launch_dependents();
  Tile t;
  if (!tile_of(a, t)) return;
  const float s = a.scales[t.lk];
  const uint4* src = reinterpret_cast<const uint4*>(a.codes + t.art_elem);
  uint4* dst = reinterpret_cast<uint4*>(a.pages + t.row * a.d * 2);
  const int nvec = t.ntok * a.d / 16;
  for (int base = threadIdx.x; base < nvec; base += kThreads * (kUnroll / 2)) {
    uint4 r[kUnroll / 2];
#pragma unroll
    for (int k = 0; k < kUnroll / 2; ++k) {
      const int i = base + k * kThreads;
      if (i < nvec) r[k] = __ldcs(src + i);
    }
#pragma unroll
    for (int k = 0; k < kUnroll / 2; ++k) {
      const int i = base + k * kThreads;
      if (i >= nvec) continue;
      const uint32_t w[4] = {r[k].x, r[k].y, r[k].z, r[k].w};
      uint32_t o[8];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        o[2 * j] = dequant2(w[j], 0, s);
        o[2 * j + 1] = dequant2(w[j], 2, s);
      }
      dst[2 * i] = make_uint4(o[0], o[1], o[2], o[3]);
      dst[2 * i + 1] = make_uint4(o[4], o[5], o[6], o[7]);
    }
  }
}

// Codes of full tiles into int8 pages (the decode kernel's layout): each
// (layer, K|V, head) block of 128 keys holds the codes + 128 (x ^ 0x80) -- K
// as [128 keys][d] rows, V transposed as [d][128 keys].
__global__ void __launch_bounds__(kThreads) q8_codes_kernel(const __grid_constant__ ArtifactArgs a) {
  __shared__ __align__(16) uint8_t tile[kPageTokens * 128];
  griddep_wait();
  griddep_launch_dependents();
  Tile t;
  if (!tile_of(a, t)) return;
  // int8 row space: page p's rows of d bytes start at byte p * page_bytes,
  // i.e. at row p * 2 * rows_per_page (rows of a bf16 page are 2 d bytes)
  const int64_t rows_per_page = static_cast<int64_t>(a.layers) * 2 * a.Hkv * kPageTokens;
  const int64_t row8 = t.row + static_cast<int64_t>(a.table[blockIdx.x]) * rows_per_page;
  const uint4* src = reinterpret_cast<const uint4*>(a.codes + t.art_elem);
  uint4* dst = reinterpret_cast<uint4*>(a.pages + row8 * a.d);
  const int nvec = kPageTokens * a.d / 16;  // full tiles only
  const uint32_t bias = 0x80808080u;
  if (t.kv == 0) {
    for (int i = threadIdx.x; i < nvec; i += kThreads) {
      const uint4 v = __ldcs(src + i);
      dst[i] = make_uint4(v.x ^ bias, v.y ^ bias, v.z ^ bias, v.w ^ bias);
    }
    return;
  }
  for (int i = threadIdx.x; i < nvec; i += kThreads) reinterpret_cast<uint4*>(tile)[i] = __ldcs(src + i);
  __syncthreads();
  constexpr int kVecPerRow = kPageTokens / 16;  // 16-key vectors of one transposed row
  for (int i = threadIdx.x; i < nvec; i += kThreads) {
    const int dd = i / kVecPerRow, k0 = (i % kVecPerRow) * 16;
    uint32_t w[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const uint8_t* c = tile + (k0 + 4 * j) * a.d + dd;
      w[j] = (uint32_t(c[0]) | uint32_t(c[a.d]) << 8 | uint32_t(c[2 * a.d]) << 16 | uint32_t(c[3 * a.d]) << 24) ^ bias;
    }
    dst[i] = make_uint4(w[0], w[1], w[2], w[3]);
  }
}

dim3 tile_grid(const ArtifactArgs& a) {
  const int tiles = a.n_tiles > 0 ? a.n_tiles : (a.L + kPageTokens - 1) / kPageTokens;
  return dim3(tiles, a.layers * 2 * a.Hkv);
}

}  // namespace

cudaError_t launch_artifact_copy(const ArtifactArgs& a, bool to_pages, cudaStream_t st) {
  if (a.L <= 0) return cudaSuccess;
  return to_pages ? launch_kernel(copy_kernel<true>, tile_grid(a), dim3(kThreads), 0, st, 0, a)
                  : launch_kernel(copy_kernel<false>, tile_grid(a), dim3(kThreads), 0, st, 0, a);
}

cudaError_t launch_q8_export(const ArtifactArgs& a, cudaStream_t st) {
  if (a.L <= 0) return cudaSuccess;
  cudaError_t e = launch_kernel(q8_absmax_kernel, tile_grid(a), dim3(kThreads), 0, st, 0, a);
  if (e != cudaSuccess) return e;
  return launch_kernel(q8_quant_kernel, tile_grid(a), dim3(kThreads), 0, st, 0, a);
}

cudaError_t launch_q8_codes_to_pages(const ArtifactArgs& a, cudaStream_t st) {
  if (a.L <= 0 || a.n_tiles <= 0) return cudaSuccess;
  return launch_kernel(q8_codes_kernel, tile_grid(a), dim3(kThreads), 0, st, 0, a);
}

cudaError_t launch_q8_load(const ArtifactArgs& a, cudaStream_t st) {
  if (a.L <= 0) return cudaSuccess;
  return launch_kernel(q8_dequant_kernel, tile_grid(a), dim3(kThreads), 0, st, 0, a);
}

}  // namespace kvr
