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
// Each thread owns 8 consecutive elements of a head vector (16-byte loads and
// stores); the d/8 threads of one head vector sit in the same warp and reduce
// the sum of squares and exchange RoPE partners with shuffles.  cos/sin come from a
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

// A block takes whole tokens: its VPB vector slots cover the HS = Hq + 2 Hkv
// head vectors of one token (slot, slot + VPB, ... : up to NI per thread), or
// of VPB / HS tokens when a token has fewer vectors than the block has slots.
// Every input load is issued before any arithmetic, and a thread reads its
// (cos, sin) pairs and both norm weights once for all of its heads: they are
// the same for every head of a token.  FLAT (small batches, NI = 1): block i
// takes vectors [i VPB, (i + 1) VPB) of the token-major list instead, so that
// a few tokens still spread over the GPU.
template <int D, int NI, bool FLAT>
__global__ void __launch_bounds__(256) append_kernel(const __grid_constant__ AppendArgs a,
                                                     const __grid_constant__ BatchDesc bd) {
  constexpr int TPI = D / 8;       // threads per head vector
  constexpr int VPB = 256 / TPI;   // vector slots per block
  const int Hkv = a.geom.Hkv;
  const int HS = a.Hq + 2 * Hkv;   // q heads, k heads, v heads
  const int li = threadIdx.x % TPI;
  const int slot = threadIdx.x / TPI;
  static_assert(!FLAT || NI == 1, "the flat mapping has one vector per thread");
  const bool packed = FLAT || HS <= VPB;  // one vector per thread
  const int tpb = packed ? VPB / HS : 1;
  const int flat = blockIdx.x * VPB + slot;
  const int t = FLAT ? flat / HS : blockIdx.x * tpb + (packed ? slot / HS : 0);
  const int hs0 = FLAT ? flat - t * HS : (packed ? slot % HS : slot);
  const bool tok_ok = t < bd.T && (FLAT || !packed || slot < tpb * HS);
  griddep_wait();
  griddep_launch_dependents();
  uint4 raw[NI];
#pragma unroll
  for (int k = 0; k < NI; ++k) {
    const int hs = hs0 + k * VPB;
    raw[k] = make_uint4(0, 0, 0, 0);
    if (tok_ok && (k == 0 || !packed) && hs < HS) {
      const uint16_t* src = hs < a.Hq         ? a.q_pre + (static_cast<int64_t>(t) * a.Hq + hs) * D
                            : hs < a.Hq + Hkv ? a.k_pre + (static_cast<int64_t>(t) * Hkv + hs - a.Hq) * D
                                              : a.v + (static_cast<int64_t>(t) * Hkv + hs - a.Hq - Hkv) * D;
      raw[k] = __ldcs(reinterpret_cast<const uint4*>(src + li * 8));
    }
  }
  const int tc = tok_ok ? t : 0;
  const int b = seq_of_token(bd, tc);
  const int pos = bd.start[b] + (tc - bd.cu_q[b]);
  const int pc = min(max(pos, 0), a.max_positions - 1);
  const float2* cs = a.rope + static_cast<int64_t>(pc) * (D / 2) + (li % (TPI / 2)) * 8;
  float2 csv[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) csv[i] = cs[i];
  const uint4 wq = *reinterpret_cast<const uint4*>(a.q_w + li * 8);
  const uint4 wk = *reinterpret_cast<const uint4*>(a.k_w + li * 8);
  const int pidx = pos / kPageTokens;
  int page = -1;
  if (tok_ok && pos >= 0 && pos < a.max_positions && pidx < bd.max_pages)
    page = bd.page_table[static_cast<int64_t>(bd.slot[b]) * bd.max_pages + pidx];
#pragma unroll
  for (int k = 0; k < NI; ++k) {
    const int hs = hs0 + k * VPB;
    if (packed && k > 0) break;
    if (__all_sync(0xffffffffu, hs >= HS)) break;  // no head left in this warp
    const bool active = tok_ok && hs < HS;
    const int kind = hs < a.Hq ? 0 : (hs < a.Hq + Hkv ? 1 : 2);  // 0 q, 1 k, 2 v
    const int head = kind == 0 ? hs : (kind == 1 ? hs - a.Hq : hs - a.Hq - Hkv);
    // Every lane runs the norm/RoPE arithmetic (the shuffles need the whole
    // warp); v vectors keep their raw bits.
    uint4 outv = norm_rope8v<D>(raw[k], kind == 0 ? wq : wk, li, csv, a.eps);
    if (kind == 2) outv = raw[k];
    if (!active) continue;
    if (kind == 0) {
      *reinterpret_cast<uint4*>(a.q_out + (static_cast<int64_t>(t) * a.Hq + head) * D + li * 8) = outv;
      continue;
    }
    if (page < 0 || page >= a.geom.n_pages) {
      if (li == 0) atomicOr(a.err, kDevErrBounds);
      continue;
    }
    const int64_t row = kv_row(page, a.layer, kind - 1, head, a.geom.layers, Hkv) + pos % kPageTokens;
    *reinterpret_cast<uint4*>(a.geom.pages + row * (D * 2) + li * 16) = outv;
  }
}

template <int D, int NI>
cudaError_t launch_append_ni(const AppendArgs& a, const BatchDesc& b, int HS, cudaStream_t st) {
  constexpr int VPB = 256 / (D / 8);
  const int tpb = HS <= VPB ? VPB / HS : 1;
  const unsigned grid = static_cast<unsigned>((b.T + tpb - 1) / tpb);
  return launch_kernel(append_kernel<D, NI, false>, dim3(grid), dim3(256), 0, st, 0, a, b);
}

template <int D>
cudaError_t launch_append_d(const AppendArgs& a, const BatchDesc& b, int HS, cudaStream_t st) {
  constexpr int VPB = 256 / (D / 8);
  const int ni = (HS + VPB - 1) / VPB;  // head vectors per thread
  // fewer tokens than about two per SM: one vector per thread over the flat list
  if (ni > 1 && b.T < 256) {
    const int64_t vectors = static_cast<int64_t>(b.T) * HS;
    const unsigned grid = static_cast<unsigned>((vectors + VPB - 1) / VPB);
    return launch_kernel(append_kernel<D, 1, true>, dim3(grid), dim3(256), 0, st, 0, a, b);
  }
  if (ni <= 1) return launch_append_ni<D, 1>(a, b, HS, st);
  if (ni <= 2) return launch_append_ni<D, 2>(a, b, HS, st);
  if (ni <= 3) return launch_append_ni<D, 3>(a, b, HS, st);
  if (ni <= 4) return launch_append_ni<D, 4>(a, b, HS, st);
  if (ni <= 8) return launch_append_ni<D, 8>(a, b, HS, st);
  return cudaErrorInvalidValue;  // more than 8 * VPB head vectors per token
}

}  // namespace

cudaError_t launch_append(const AppendArgs& a, const BatchDesc& b, int d, int Hkv, cudaStream_t st) {
  if (b.T == 0) return cudaSuccess;
  const int HS = a.Hq + 2 * Hkv;
  return d == 64 ? launch_append_d<64>(a, b, HS, st) : launch_append_d<128>(a, b, HS, st);
}

}  // namespace kvr
