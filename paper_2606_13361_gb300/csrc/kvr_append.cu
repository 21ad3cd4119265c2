// kvr_append.cu -- append step for new tokens of one layer.
//
// Per token t (sequence b, position p = start_b + t - cu_q[b]) and head:
//   q', k' = RoPE(RMSNorm(x) * w, p)   (per-head RMSNorm over head_dim, then
//                                       rotate-half RoPE at position p)
//   v' = v
// q' goes to q_out; k', v' go to the cache row of position p.  Sec. 3.2: the
// continuation tokens take positions L, L+1, ... so their RoPE matches a
// from-scratch pass.  fp32 arithmetic, one rounding to bf16.
//
// Each thread owns 8 consecutive elements (one 16-byte load and store); the
// d/8 threads of one head vector sit in the same warp and reduce the sum of
// squares and exchange RoPE partners with shuffles.  cos/sin come from a
// [max_positions][d/2] fp32 table built on the host in fp64.
#include "kvr_internal.h"
#include "kvr_ptx.cuh"
#include "kvr_rope.cuh"

namespace kvr {
namespace {

__device__ __forceinline__ int seq_of_token(const BatchDesc& bd, int t) {
  int lo = 0, hi = bd.n_seqs - 1;
  while (lo < hi) {
    int mid = (lo + hi + 1) >> 1;
    if (bd.cu_q[mid] <= t) lo = mid; else hi = mid - 1;
  }
  return lo;
}

template <int D>
__global__ void __launch_bounds__(256) append_kernel(const __grid_constant__ AppendArgs a,
                                                     const __grid_constant__ BatchDesc bd) {
  constexpr int TPI = D / 8;       // threads per head vector
  const int Hkv = a.geom.Hkv;
  const int HS = a.Hq + 2 * Hkv;   // q heads, k heads, v heads
  const int64_t item = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) / TPI;
  const int li = threadIdx.x % TPI;
  const int64_t n_items = static_cast<int64_t>(bd.T) * HS;
  const bool active = item < n_items;
  const int t = active ? static_cast<int>(item / HS) : 0;
  const int hs = active ? static_cast<int>(item % HS) : 0;

  const int kind = hs < a.Hq ? 0 : (hs < a.Hq + Hkv ? 1 : 2);  // 0 q, 1 k, 2 v
  const int head = kind == 0 ? hs : (kind == 1 ? hs - a.Hq : hs - a.Hq - Hkv);
  const uint16_t* src = kind == 0 ? a.q_pre + (static_cast<int64_t>(t) * a.Hq + head) * D
                      : kind == 1 ? a.k_pre + (static_cast<int64_t>(t) * Hkv + head) * D
                                  : a.v + (static_cast<int64_t>(t) * Hkv + head) * D;
  griddep_wait();
  griddep_launch_dependents();
  uint4 raw = make_uint4(0, 0, 0, 0);
  if (active) raw = *reinterpret_cast<const uint4*>(src + li * 8);

  const int b = seq_of_token(bd, t);
  const int pos = bd.start[b] + (t - bd.cu_q[b]);

  // Every lane runs the norm/RoPE arithmetic (the shuffles need the whole
  // warp); v vectors keep their raw bits.
  const int pc = min(max(pos, 0), a.max_positions - 1);
  const float2* cs = a.rope + static_cast<int64_t>(pc) * (D / 2) + (li % (TPI / 2)) * 8;
  const uint4 wraw = *reinterpret_cast<const uint4*>((kind == 0 ? a.q_w : a.k_w) + li * 8);
  uint4 outv = norm_rope8<D>(raw, wraw, li, cs, a.eps);
  if (kind == 2) outv = raw;
  if (!active) return;
  if (kind == 0) {
    *reinterpret_cast<uint4*>(a.q_out + (static_cast<int64_t>(t) * a.Hq + head) * D + li * 8) = outv;
    return;
  }
  const int pidx = pos / kPageTokens;
  int page = -1;
  if (pos >= 0 && pos < a.max_positions && pidx < bd.max_pages)
    page = bd.page_table[static_cast<int64_t>(bd.slot[b]) * bd.max_pages + pidx];
  if (page < 0 || page >= a.geom.n_pages) {
    if (li == 0) atomicOr(a.err, kDevErrBounds);
    return;
  }
  const int64_t row = kv_row(page, a.layer, kind - 1, head, a.geom.layers, Hkv) + pos % kPageTokens;
  *reinterpret_cast<uint4*>(a.geom.pages + row * (D * 2) + li * 16) = outv;
}

}  // namespace

cudaError_t launch_append(const AppendArgs& a, const BatchDesc& b, int d, int Hkv, cudaStream_t st) {
  const int64_t items = static_cast<int64_t>(b.T) * (a.Hq + 2 * Hkv);
  if (items == 0) return cudaSuccess;
  const int64_t threads = items * (d / 8);
  const unsigned grid = static_cast<unsigned>((threads + 255) / 256);
  if (d == 64) return launch_kernel(append_kernel<64>, dim3(grid), dim3(256), 0, st, 0, a, b);
  return launch_kernel(append_kernel<128>, dim3(grid), dim3(256), 0, st, 0, a, b);
}

}  // namespace kvr
