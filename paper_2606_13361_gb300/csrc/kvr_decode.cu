// kvr_decode.cu -- reuse attention for batches with few query rows per KV head
// (decode steps: Algorithm 2's loop with |cur| = 1, for up to 8 rows per head).
//
// A decode row attends over thousands of cached keys at ~4 flop per byte, so
// the call is bound by HBM and by latency, not by tensor throughput.  The keys
// of each KV head are cut into 32-key units (K and V of one unit: 2 x 8 KB at
// head_dim 128), staged by TMA into 128B-swizzled shared memory.  CTA = one KV
// head x one split of its units, 12 warps; warp w takes units w, w+12, ... and
// keeps its own online softmax (exp2 domain) over them.  Within a warp the
// <= 8 query rows are the n = 8 side of m16n8k16 MMAs, keys and head
// dimensions the m = 16 side: S^T = K Q^T and O^T += V^T P^T (q fragments stay
// in registers for the whole call, K through ldmatrix, V through
// ldmatrix.trans, P^T from the S^T accumulators by an 8x8 register
// transpose), so no MMA lane is padding when 8 rows are present.  Each warp
// leaves its state in its own staging slot; the splits of a KV head form one
// thread-block cluster (<= 16 CTAs), every CTA weighs its warps' states and
// pushes each owner CTA its slice of output columns with 16-byte asynchronous
// remote stores that count down the owner's receive barrier, and each owner
// merges its slice over the splits (sums spread over lanes and added in a
// fixed shuffle tree).
// Long contexts spread a head over up to 4 clusters: each cluster's owners
// leave their slices in global memory and the last cluster to arrive merges
// them in cluster order.  A row sees a key iff its tile is shared by the batch
// or owned by its sequence and the key's position is <= the row's (Sec. 3.2:
// the mask spans the cached context plus the new tokens).
//
// The fused variant (a decode step: Algorithm 2's forward for the new token)
// also does the append: every CTA norms and ropes its rows' q and the new
// tokens' k with the same arithmetic as the append kernel, patches the new
// keys and values into its staged tile once the copy lands (so no CTA depends
// on the cache write), and the warp whose unit holds a new key writes it to
// the cache for later steps.
//
// The Q8 variant (a sequence with an int8-resident prefix, Sec. 5) reads
// those pages' codes instead, two units in flight per warp, and builds exact
// f16 MMA fragments from them directly; the per-tensor scales multiply the
// scores and the probabilities.
#include <cuda_bf16.h>
#include <math.h>

#include <algorithm>

#include "kvr_internal.h"
#include "kvr_ptx.cuh"
#include "kvr_rope.cuh"

namespace kvr {
#ifdef KVR_STAGE_TRACE
KVR_STAGE_BUFFER(g_stage_decode);
#endif
namespace {

// Warps per CTA: 12 (one CTA per SM) or 6 (two per SM, so that the next
// launch's CTAs are resident beside this one's; see decode_splits).
constexpr int kWarpsMax = 12;
constexpr int kUnit = 32;  // keys per unit
constexpr int kRows = kDecodeMaxRows;
constexpr float kLn2 = 0.69314718055994530942f;

template <int D, int kWarps>
struct DecLayout {
  static constexpr int kBox = kUnit * 64 * 2;       // 32 keys x 64 columns, 128B-swizzled
  static constexpr int kUnitBytes = kUnit * D * 2;  // K (or V) of one unit
  static constexpr int kStride = D + 4;             // merge row: D values, max, sum, pad
  static constexpr int kK = 0;
  static constexpr int kV = kK + kWarps * kUnitBytes;
  // a warp's state for the CTA merge: the K half of its slot once its units
  // are consumed, fp32 [row][kStride]
  // split partials pushed to this CTA: fp32 [source split][row][cw] for its
  // cw output columns (cw = ceil(D / splits) rounded up to a multiple of 4),
  // then fp32 [source split][row][max, sum]; S cw <= D + 4 S
  static constexpr int kRecv = kV + kWarps * kUnitBytes;
  static constexpr int kRecvFloats = kRows * (D + 6 * 16);
  static constexpr int kQ = kRecv + kRecvFloats * 4;             // bf16 [row][D]: roped q
  static constexpr int kNewK = kQ + kRows * D * 2;               // bf16 [token][D]: new k (fused)
  static constexpr int kNewV = kNewK + kRows * D * 2;            // bf16 [token][D]: new v (fused)
  static constexpr int kQ16 = kNewV + kRows * D * 2;            // f16 q fragments [k-step][lane] (int8 units)
  static constexpr int kBar = kQ16 + kRows * D * 2;             // slot barriers (up to 2 per warp) + receive barrier
  static constexpr int kMisc = kBar + (2 * kWarps + 1) * 8;          // abort flag, page of each first unit
  static constexpr int kScl = kMisc + 16 * 4;                   // fp32 [row seq][K|V]: int8 scales
  static constexpr int kEnd = kScl + kRows * 2 * 4;
  static constexpr int kAlloc = kEnd + 1024;
  static_assert(kRows * kStride * 4 <= kUnitBytes, "a warp state fits the K half of its slot");
  static_assert((kStride * 4) % 16 == 0 && kUnitBytes % 16 == 0 && kRecv % 16 == 0, "16-byte rows");
};

__device__ __forceinline__ void mma_16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                          uint32_t a3, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
      "{%8, %9}, {%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// The same product with f16 operands (int8 codes and the f16 copy of q).
__device__ __forceinline__ void mma_16816_f16(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                              uint32_t a3, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
      "{%8, %9}, {%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t pack_f16x2(float lo, float hi) {
  uint32_t r;
  asm("cvt.rn.f16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
  return r;
}

// Eight bf16 -> eight f16 (exact in the normal f16 range; saturated beyond it).
__device__ __forceinline__ uint4 bf16x8_to_f16x8(uint4 v) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
  uint32_t o[4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
    asm("cvt.rn.satfinite.f16x2.f32 %0, %1, %2;"
        : "=r"(o[i])
        : "f"(__uint_as_float(w[i] & 0xffff0000u)), "f"(__uint_as_float(w[i] << 16)));
  return make_uint4(o[0], o[1], o[2], o[3]);
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                        uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                          uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

// 8x8 b16 matrix transpose across the warp (thread lane holds row lane/4,
// columns 2(lane%4), 2(lane%4)+1, before and after).
__device__ __forceinline__ uint32_t movmatrix_t(uint32_t x) {
  uint32_t y;
  asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(y) : "r"(x));
  return y;
}

// byte offset of (row, 16-byte chunk c) in a 128B-swizzled tile of 64-column boxes
template <int D>
__device__ __forceinline__ uint32_t sw_off(int row, int c) {
  return (c >> 3) * DecLayout<D, kWarpsMax>::kBox + row * 128 + (((c & 7) ^ (row & 7)) << 4);
}

// Two int8 codes stored as code + 128 (bytes of x picked by `sel`) -> two
// exact f16 codes: code + 128 becomes the low mantissa byte of 1024 (prmt),
// then 1152 = 1024 + 128 is subtracted.
__device__ __forceinline__ uint32_t code2_f16(uint32_t x, uint32_t sel) {
  uint32_t r;
  asm("add.rn.f16x2 %0, %1, %2;" : "=r"(r) : "r"(__byte_perm(x, 0x64646464u, sel)), "r"(0xE480E480u));
  return r;
}

// The same with a power-of-two factor: code * 2^-e from one fma with (mul,
// add) = (2^-e, -1152 * 2^-e); exact for -4 <= e <= 14 (every operand and
// result a normal f16).
__device__ __forceinline__ uint32_t codes2_f16(uint32_t x, uint32_t sel, uint32_t mul, uint32_t add) {
  uint32_t r;
  asm("fma.rn.f16x2 %0, %1, %2, %3;" : "=r"(r) : "r"(__byte_perm(x, 0x64646464u, sel)), "r"(mul), "r"(add));
  return r;
}

// The power of two 2^e (-4 <= e <= 14) that brings an int8 tensor's scale s
// into [1, 2) where it can: the codes of that tensor are staged as code * 2^-e
// and the factor s 2^e travels with the probabilities, so that neither leaves
// the normal f16 range.  Returns e; `mul`, `add` are the f16x2 fma operands.
__device__ __forceinline__ int code_exponent(float s, uint32_t* mul, uint32_t* add) {
  const int E = static_cast<int>((__float_as_uint(s) >> 23) & 0xffu);  // s = m 2^(E - 127)
  const int e = min(max(127 - E, -4), 14);
  const uint32_t m16 = static_cast<uint32_t>(15 - e) << 10;                 // 2^-e
  const uint32_t a16 = 0x8000u | (static_cast<uint32_t>(25 - e) << 10) | 0x080u;  // -1152 * 2^-e
  *mul = m16 | m16 << 16;
  *add = a16 | a16 << 16;
  return e;
}

// f16 q of row r, dims d0 .. d0 + 7 (d0 a multiple of 8) -> the fragment
// order of the int8 units' S^T products: the uint2 at [k][4 r + tq] holds
// dims (D / 4) tq + 4 k .. + 3 of row r.
template <int D>
__device__ __forceinline__ void put_q16(uint16_t* q16, int r, int d0, uint4 v) {
  uint2* f = reinterpret_cast<uint2*>(q16);
  const int tq = d0 / (D / 4), k = (d0 % (D / 4)) / 4;
  f[k * 32 + 4 * r + tq] = make_uint2(v.x, v.y);
  f[(k + 1) * 32 + 4 * r + tq] = make_uint2(v.z, v.w);
}

__device__ __forceinline__ int seq_of(const SmallBatch& bd, int t) {
  int lo = 0, hi = bd.n_seqs - 1;
  while (lo < hi) {
    int mid = (lo + hi + 1) >> 1;
    if (bd.cu_q[mid] <= t) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// Unit u of the batch's key list: shared units first (4 per shared page),
// then each sequence's own units up to its last row's position.
struct UnitMap {
  int shared_units;
  int n_seqs;
  int own[kRows];
  __device__ void locate(const SmallBatch& bd, int u, int* key_base, int* owner, int* slot) const {
    if (u < shared_units) {
      *key_base = u * kUnit;
      *owner = -1;
      *slot = bd.slot[0];
      return;
    }
    u -= shared_units;
    int b = 0;
    while (b < n_seqs - 1 && u >= own[b]) {
      u -= own[b];
      ++b;
    }
    *key_base = bd.shared_pages * kPageTokens + u * kUnit;
    *owner = b;
    *slot = bd.slot[b];
  }
};

// Q8: some row of the batch reads int8 copies of its full pages (a separate
// instantiation, so that the bf16-only kernel carries none of that code).
template <int D, bool FUSED, bool Q8, int kWarps>
__global__ void __launch_bounds__(kWarps * 32, kWarpsMax / kWarps)
decode_kernel(const __grid_constant__ DecodeArgs a, const __grid_constant__ SmallBatch bd) {
  using Lay = DecLayout<D, kWarps>;
  constexpr int kThreads = kWarps * 32;
  constexpr int KS = D / 16;  // k-steps over the head dimension
  constexpr int stride = Lay::kStride;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + Lay::kBar);
  int* misc = reinterpret_cast<int*>(smem + Lay::kMisc);
  constexpr int NB = Q8 ? 2 : 1;  // slot barriers per warp
  uint64_t* recv_bar = full + NB * kWarps;
  float* recv = reinterpret_cast<float*>(smem + Lay::kRecv);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int gq = lane >> 2, tq = lane & 3;  // fragment row group / thread-in-group
  // stage slots: 0 entry, 1 grid dependency resolved, 2 prologue done, 3 warp 0's
  // first unit landed, 4 + w warp w's last unit done, 16 merge start, 17 warp
  // states stored, 18 cluster merge start, 19 pushes issued, 20 partials
  // received, 21 end; with 6 warps also 10 + w warp w's first unit done,
  // 22 + w its second unit landed, 28 first copies issued (warp 0), 29 q/k
  // norm + rope done (last warp), 30 q fragments loaded (warp 0), 31 warp 0's first copy landed
  if (threadIdx.x == 0) KVR_STAGE(g_stage_decode, a.layer, 0);
  // block = (KV head g, cluster cl of that head, split = rank in the cluster);
  // the head's units are cut into n_splits x n_clusters parts
  const int g = blockIdx.x / (a.n_splits * a.n_clusters);
  const int part = blockIdx.x % (a.n_splits * a.n_clusters);
  const int cl = part / a.n_splits;
  const int split = part % a.n_splits;
  const int n_parts = a.n_splits * a.n_clusters;

  UnitMap um;
  um.shared_units = bd.shared_pages * (kPageTokens / kUnit);
  um.n_seqs = bd.n_seqs;
  int total = um.shared_units;
  for (int b = 0; b < bd.n_seqs; ++b) {
    const int maxpos = bd.start[b] + (bd.cu_q[b + 1] - bd.cu_q[b]) - 1;
    const int keys = maxpos + 1 - bd.shared_pages * kPageTokens;
    um.own[b] = keys > 0 ? (keys + kUnit - 1) / kUnit : 0;
    total += um.own[b];
  }
  const int u0 = static_cast<int>(static_cast<int64_t>(total) * part / n_parts);
  const int u1 = static_cast<int>(static_cast<int64_t>(total) * (part + 1) / n_parts);
  const int n = u1 - u0;

  const int S = a.n_splits;
  const int R = bd.T * a.G;  // rows: token-major, then the G query heads of KV head g
  // output columns merged by each CTA of the cluster (a multiple of 4)
  const int cw = ((D + S - 1) / S + 3) / 4 * 4;
  if (threadIdx.x == 0) {
    for (int w = 0; w < NB * kWarps; ++w) mbar_init(&full[w], 1);
    mbar_init(recv_bar, 1);
    fence_barrier_init();
    // an owner of my_cw columns receives R (my_cw + 2) floats from each of the S splits
    const int my_cw0 = max(0, min(D, (split + 1) * cw) - split * cw);
    if (S > 1 && my_cw0 > 0) mbar_arrive_expect_tx(recv_bar, static_cast<uint32_t>(S * R * (my_cw0 + 2) * 4));
    misc[0] = 0;  // abort flag
  }
  // Before the previous kernel's results are visible: pull this CTA's first
  // units into L2.  The pages of cached keys are not written by earlier
  // kernels (only the new tokens' rows are, and those are patched from the
  // inputs); a page-table entry read here may be stale, which only wastes a
  // prefetch: addresses are checked against the pool, and the copies below
  // look the pages up again.
  if (threadIdx.x < min(n, 2 * kWarps) && a.pages != nullptr) {
    int key_base, owner, slot;
    um.locate(bd, u0 + threadIdx.x, &key_base, &owner, &slot);
    const int pidx = key_base / kPageTokens;
    const int page = (pidx < bd.max_pages) ? bd.page_table[static_cast<int64_t>(slot) * bd.max_pages + pidx] : -1;
    if (Q8 && pidx < a.q8_n[owner < 0 ? 0 : owner]) {  // the unit's int8 copy
      const int page8 = a.q8_table[static_cast<int64_t>(slot) * bd.max_pages + pidx];
      const int64_t rpp = static_cast<int64_t>(a.layers) * 2 * a.Hkv * kPageTokens;
      const int64_t rk = kv_row(page8, a.layer, 0, g, a.layers, a.Hkv) + page8 * rpp + key_base % kPageTokens;
      const int64_t rvb = kv_row(page8, a.layer, 1, g, a.layers, a.Hkv) + page8 * rpp;
      if (page8 >= 0 && rk >= 0 && rvb + kPageTokens <= 2 * a.n_pool_rows) {
        l2_prefetch(a.pages + rk * D, Lay::kUnitBytes / 2);
        tma_prefetch_2d(&a.tm_q8t, key_base % kPageTokens, static_cast<int>(rvb / kPageTokens * D));
      }
    } else if (page >= 0) {
      const int64_t rk = kv_row(page, a.layer, 0, g, a.layers, a.Hkv) + key_base % kPageTokens;
      const int64_t rv = kv_row(page, a.layer, 1, g, a.layers, a.Hkv) + key_base % kPageTokens;
      if (rk >= 0 && rv + kUnit <= a.n_pool_rows) {
        l2_prefetch(a.pages + rk * (D * 2), Lay::kUnitBytes);
        l2_prefetch(a.pages + rv * (D * 2), Lay::kUnitBytes);
      }
    }
  }
  // The rows read right after the dependency (q, the new tokens' k and v, the
  // norm weights) may be written by the previous kernel; an L2 prefetch is
  // only a hint, and L2 is where those writes land, so it can start now.
  if (warp == kWarps - 1) {
    const int T = bd.T;
    const uint16_t* src = nullptr;
    if (lane < R) {
      const int t = lane / a.G, h = g * a.G + lane % a.G;
      src = (FUSED ? a.q_pre : a.q) + (static_cast<int64_t>(t) * a.Hq + h) * D;
    } else if (FUSED && lane < R + 2 * T) {
      const int t = (lane - R) % T;
      src = (lane < R + T ? a.k_pre : a.v_new) + (static_cast<int64_t>(t) * a.Hkv + g) * D;
    } else if (FUSED && lane < R + 2 * T + 2) {
      src = lane == R + 2 * T ? a.q_w : a.k_w;
    }
    if (src != nullptr) l2_prefetch(src, D * 2);
  }
  // The (cos, sin) pairs this lane needs in the fused norm + RoPE below come
  // from the context's own table, which no kernel writes: read them before
  // the grid dependency, off the critical path.
  constexpr int TPI = D / 8, VPW = 32 / TPI;
  // (with 12 warps one pass covers every vector; with 6 the later passes
  // read their pairs after the dependency, below)
  float2 csv[8];
  if constexpr (FUSED) {
    const int vb = (kWarps - 1 - warp) * VPW + lane / TPI;
    const int T = bd.T;
    const int t = vb < R ? vb / a.G : min(vb - R, T - 1);
    const int b = seq_of(bd, min(t, T - 1));
    const int pc = min(max(bd.start[b] + (t - bd.cu_q[b]), 0), a.max_positions - 1);
    const float2* cs = a.rope + static_cast<int64_t>(pc) * (D / 2) + ((lane % TPI) % (TPI / 2)) * 8;
#pragma unroll
    for (int i = 0; i < 8; ++i) csv[i] = vb < R + T ? cs[i] : make_float2(0.f, 0.f);
  }
  __syncthreads();
  // Receive barriers of the cluster are initialised before any CTA pushes into
  // another: this arrive pairs with the wait just before the split merge.
  if (S > 1) cluster_arrive();
  volatile int* abort_flag = misc;
  griddep_wait();  // global memory from here on
  griddep_launch_dependents();
  if (threadIdx.x == 0) KVR_STAGE(g_stage_decode, a.layer, 1);

  // Copy unit i into the warp's slot (bf16: the whole slot, barrier NB w) or,
  // for a unit of an int8 page, into half h of it (barrier NB w + h): K codes
  // [32 keys][D] at the half's start, V^T codes [D][32 keys] after them.
  // Returns the unit's bf16 page (for the fused patch), or -1.
  auto issue = [&](int i, int h) -> int {
    int key_base, owner, slot;
    um.locate(bd, u0 + i, &key_base, &owner, &slot);
    const int pidx = key_base / kPageTokens;
    const int w = i % kWarps;
    if (Q8 && pidx < a.q8_n[owner < 0 ? 0 : owner]) {
      // new keys never sit in an int8 page (its positions are all below the length)
      const int page8 = a.q8_table[static_cast<int64_t>(slot) * bd.max_pages + pidx];
      const int64_t rpp = static_cast<int64_t>(a.layers) * 2 * a.Hkv * kPageTokens;
      int64_t rk = kv_row(page8, a.layer, 0, g, a.layers, a.Hkv) + page8 * rpp + key_base % kPageTokens;
      int64_t rvb = kv_row(page8, a.layer, 1, g, a.layers, a.Hkv) + page8 * rpp;  // the V block's first row
      if (page8 < 0 || rk < 0 || rvb + kPageTokens > 2 * a.n_pool_rows) {
        atomicOr(a.err, kDevErrBounds);
        rk = rvb = 0;
      }
      uint64_t* bar = &full[NB * w + h];
      uint8_t* dst = smem + (h ? Lay::kV : Lay::kK) + w * Lay::kUnitBytes;
      mbar_arrive_expect_tx(bar, Lay::kUnitBytes);
      tma_load_2d(dst, &a.tm_q8, bar, 0, static_cast<int>(rk));
      tma_load_2d(dst + Lay::kUnitBytes / 2, &a.tm_q8t, bar, key_base % kPageTokens,
                  static_cast<int>(rvb / kPageTokens * D));
      return -1;
    }
    const int page = (pidx < bd.max_pages) ? bd.page_table[static_cast<int64_t>(slot) * bd.max_pages + pidx] : -1;
    int64_t rk = kv_row(page, a.layer, 0, g, a.layers, a.Hkv) + key_base % kPageTokens;
    int64_t rv = kv_row(page, a.layer, 1, g, a.layers, a.Hkv) + key_base % kPageTokens;
    if (page < 0 || rv + kUnit > a.n_pool_rows) {
      atomicOr(a.err, kDevErrBounds);
      rk = rv = 0;
    }
    uint64_t* bar = &full[NB * w];
    mbar_arrive_expect_tx(bar, 2 * Lay::kUnitBytes);
#pragma unroll
    for (int c = 0; c < D / 64; ++c) {
      tma_load_2d(smem + Lay::kK + w * Lay::kUnitBytes + c * Lay::kBox, &a.tm_kv32, bar, c * 64,
                  static_cast<int>(rk));
      tma_load_2d(smem + Lay::kV + w * Lay::kUnitBytes + c * Lay::kBox, &a.tm_kv32, bar, c * 64,
                  static_cast<int>(rv));
    }
    return (page < 0 || rv + kUnit > a.n_pool_rows) ? -1 : page;
  };
  // The first units' copies start at once, issued by lanes 0 and 1 of warps
  // 0-5 (slots w and w + 6), so all page lookups are one round trip; the q/k
  // norm + rope runs on the last warps and the new v copy on warp 8
  // meanwhile, so their global loads overlap instead of queueing behind one
  // another.
  if (warp < kWarps / 2 && lane < 2) {
    const int sl = warp + (kWarps / 2) * lane;
    if (sl < min(n, kWarps)) misc[1 + sl] = issue(sl, 0);
    if (threadIdx.x == 0) KVR_STAGE(g_stage_decode, a.layer, 28);
  }
#ifdef KVR_STAGE_TRACE
  // traced builds only: lane 2 of warp 1 (idle in the prologue) watches warp
  // 0's first copy land, so its true latency is seen (a bounded poll)
  if (kWarps == 6 && warp == 1 && lane == 2 && n > 0) {
    const uint64_t tw = global_timer_ns();
    while (!mbar_try_wait(&full[0], 0) && global_timer_ns() - tw < 100000) {
    }
    KVR_STAGE(g_stage_decode, a.layer, 31);
  }
#endif
  // the int8 scales of each batch sequence, once per CTA (visible to the
  // units after the barrier below)
  float* scl = reinterpret_cast<float*>(smem + Lay::kScl);
  if constexpr (Q8) {
    if (threadIdx.x < 2 * bd.n_seqs) {
      const int b = threadIdx.x >> 1;
      const int64_t at = (static_cast<int64_t>(bd.slot[b]) * a.layers + a.layer) * 2 + (threadIdx.x & 1);
      scl[threadIdx.x] = a.q8_n[b] > 0 ? a.q8_scales[at] : 1.f;
    }
  }

  // q rows: row gq is this lane's column of the Q^T fragments; rows 2tq and
  // 2tq + 1 are its columns of the S^T and O^T accumulators
  const bool row_ok = gq < R;
  int pos_r[2] = {-1, -1}, own_r[2] = {-2, -2};
#pragma unroll
  for (int j = 0; j < 2; ++j) {
    const int r = 2 * tq + j;
    if (r < R) {
      const int t = r / a.G;
      own_r[j] = seq_of(bd, t);
      pos_r[j] = bd.start[own_r[j]] + (t - bd.cu_q[own_r[j]]);
    }
  }
  // ---- roped q rows (and, fused, the new tokens' k and v) into shared memory ----
  uint16_t* qs = reinterpret_cast<uint16_t*>(smem + Lay::kQ);
  uint16_t* nk = reinterpret_cast<uint16_t*>(smem + Lay::kNewK);
  uint16_t* nv = reinterpret_cast<uint16_t*>(smem + Lay::kNewV);
  uint16_t* q16 = reinterpret_cast<uint16_t*>(smem + Lay::kQ16);
  const int T = bd.T;
  if constexpr (FUSED) {
    // one D/8-lane group per vector: rows 0..R-1 are q rows, R..R+T-1 the new
    // keys; vectors 0, 1, ... go to the last warp first (one pass: see above)
    const int li = lane % TPI;
    for (int vb0 = (kWarps - 1 - warp) * VPW; vb0 < R + T; vb0 += kWarps * VPW) {
      const int vb = vb0 + lane / TPI;
      if (vb0 != (kWarps - 1 - warp) * VPW) {  // past the first pass: this vector's (cos, sin)
        const int tt = vb < R ? vb / a.G : min(vb - R, T - 1);
        const int bb = seq_of(bd, min(tt, T - 1));
        const int pc = min(max(bd.start[bb] + (tt - bd.cu_q[bb]), 0), a.max_positions - 1);
        const float2* cs = a.rope + static_cast<int64_t>(pc) * (D / 2) + ((lane % TPI) % (TPI / 2)) * 8;
#pragma unroll
        for (int i = 0; i < 8; ++i) csv[i] = vb < R + T ? cs[i] : make_float2(0.f, 0.f);
      }
      const bool is_q = vb < R, live = vb < R + T;
      const int t = is_q ? vb / a.G : min(vb - R, T - 1);
      const int b = seq_of(bd, min(t, T - 1));
      const int p = bd.start[b] + (t - bd.cu_q[b]);
      const int h = is_q ? g * a.G + vb % a.G : g;
      const uint16_t* src = is_q ? a.q_pre + (static_cast<int64_t>(t) * a.Hq + h) * D
                                 : a.k_pre + (static_cast<int64_t>(t) * a.Hkv + g) * D;
      const uint4 raw = live ? *reinterpret_cast<const uint4*>(src + li * 8) : make_uint4(0, 0, 0, 0);
      const uint4 wraw = *reinterpret_cast<const uint4*>((is_q ? a.q_w : a.k_w) + li * 8);
      (void)p;
      const uint4 y = norm_rope8v<D>(raw, wraw, li, csv, a.eps);
      if (live) {
        if (is_q) {
          *reinterpret_cast<uint4*>(qs + vb * D + li * 8) = y;
          if constexpr (Q8) put_q16<D>(q16, vb, li * 8, bf16x8_to_f16x8(y));
          if (part == 0 && a.q_out != nullptr)
            *reinterpret_cast<uint4*>(a.q_out + (static_cast<int64_t>(t) * a.Hq + h) * D + li * 8) = y;
        } else {
          *reinterpret_cast<uint4*>(nk + t * D + li * 8) = y;
        }
      }
    }
    if (warp == kWarps - 1 && lane == 0) KVR_STAGE(g_stage_decode, a.layer, 29);
    if (warp == (kWarps == 12 ? 8 : 0))
      for (int i = lane; i < T * (D / 8); i += 32) {
        const int t = i / (D / 8), c8 = i % (D / 8);
        *reinterpret_cast<uint4*>(nv + t * D + c8 * 8) =
            *reinterpret_cast<const uint4*>(a.v_new + (static_cast<int64_t>(t) * a.Hkv + g) * D + c8 * 8);
      }
  } else {
    for (int i = kThreads - 1 - threadIdx.x; i < R * (D / 8); i += kThreads) {
      const int r = i / (D / 8), c8 = i % (D / 8);
      const int t = r / a.G, h = g * a.G + r % a.G;
      const uint4 y = *reinterpret_cast<const uint4*>(a.q + (static_cast<int64_t>(t) * a.Hq + h) * D + c8 * 8);
      *reinterpret_cast<uint4*>(qs + r * D + c8 * 8) = y;
      if constexpr (Q8) put_q16<D>(q16, r, c8 * 8, bf16x8_to_f16x8(y));
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) KVR_STAGE(g_stage_decode, a.layer, 2);
  int unit_page = misc[1 + warp];  // page of the unit in this warp's slot (when warp < n)
  // Q^T B-fragments (column = row gq; bf16 pairs at dims 16k + 2tq and 16k + 8 + 2tq)
  uint32_t qa0[KS], qa2[KS];
  {
    const uint32_t* qrow = reinterpret_cast<const uint32_t*>(qs + (row_ok ? gq : 0) * D);
#pragma unroll
    for (int k = 0; k < KS; ++k) {
      qa0[k] = row_ok ? qrow[8 * k + tq] : 0u;
      qa2[k] = row_ok ? qrow[8 * k + 4 + tq] : 0u;
    }
  }
#ifdef KVR_STAGE_TRACE
  if (threadIdx.x == 0) {  // (after the q fragments arrived)
    uint32_t qsum = 0;
    for (int k = 0; k < KS; ++k) qsum ^= qa0[k] ^ qa2[k];
    if (qsum != 0x9e3779b9u) KVR_STAGE(g_stage_decode, a.layer, 30);
  }
#endif
  const float c = a.scale_log2;
  // per row 2tq + j: reference maximum, this lane's share of the row sum
  float m[2] = {-INFINITY, -INFINITY}, l[2] = {0.f, 0.f};
  // O^T accumulators: dims 16 md + gq (regs 0, 1) and + 8 (regs 2, 3), rows 2tq, 2tq + 1
  constexpr int MD = D / 16;
  float o[MD][4];
#pragma unroll
  for (int i = 0; i < MD; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  const uint32_t kt = smem_u32(smem + Lay::kK + warp * Lay::kUnitBytes);
  const uint32_t vt = smem_u32(smem + Lay::kV + warp * Lay::kUnitBytes);
  // V^T A-fragments of a bf16 unit, (k-step kk, m-tile md) pairs in kk-major
  // order, kVG per group, two groups in registers at a time
  constexpr int kVG = 4, kVGroups = 2 * MD / kVG;
  uint32_t va[2][kVG][4];
  auto load_v = [&](int grp, uint32_t(&dst)[kVG][4]) {
#pragma unroll
    for (int i = 0; i < kVG; ++i) {
      const int it = grp * kVG + i, kk = it / MD, md = it % MD;
      ldsm_x4_t(vt + sw_off<D>(16 * kk + (lane & 7) + ((lane >> 4) & 1) * 8, 2 * md + ((lane >> 3) & 1)), dst[i][0],
                dst[i][1], dst[i][2], dst[i][3]);
    }
  };

  // one unit: its tiles staged in the warp's slot (bf16) or at `half` (int8)
  auto run_unit = [&](int i, int unit_page_in, const uint8_t* half) {
      int key_base, owner, slot;
      um.locate(bd, u0 + i, &key_base, &owner, &slot);
      // An int8 unit (its codes + 128 at `half`: K [32 keys][D], V^T [D][32
      // keys]): K = code_k s_k and V = code_v s_v, the codes exact in f16
      // fragments (V's as code_v 2^-e); s_k scales the scores, s_v 2^e the
      // probabilities fed to P V.
      const bool q8u = Q8 && key_base / kPageTokens < a.q8_n[owner < 0 ? 0 : owner];
      float cu = c, s_v = 1.f;
      uint32_t vmul = 0, vadd = 0;
      if (q8u) {
        const float* sc = scl + 2 * (owner < 0 ? 0 : owner);
        cu = c * sc[0];
        const int e = code_exponent(sc[1], &vmul, &vadd);
        s_v = sc[1] * __uint_as_float(static_cast<uint32_t>(127 + e) << 23);  // exact: a power of two
      }
      if constexpr (FUSED) {
        // new keys of the owner sequence inside this unit: use the values computed
        // above (the cache copy may predate this launch's write)
        if (owner >= 0) {
          const int tb = bd.cu_q[owner], te = bd.cu_q[owner + 1];
          bool any = false;
          for (int t = tb; t < te; ++t) {
            const int kr = bd.start[owner] + (t - tb) - key_base;
            if (kr >= 0 && kr < kUnit) {
              any = true;
              // this warp owns the unit holding the new key: patch the staged tile
              // and write the cache row (the unit's page is known from the copy)
              const int page = __shfl_sync(0xffffffffu, unit_page_in, 0);
              for (int c8 = lane; c8 < 2 * (D / 8); c8 += 32) {
                const int kv = c8 / (D / 8), cc = c8 % (D / 8);
                uint8_t* tile = smem + (kv ? Lay::kV : Lay::kK) + warp * Lay::kUnitBytes;
                const uint4 val = *reinterpret_cast<const uint4*>((kv ? nv : nk) + t * D + cc * 8);
                *reinterpret_cast<uint4*>(tile + sw_off<D>(kr, cc)) = val;
                if (page >= 0) {
                  const int64_t row = kv_row(page, a.layer, kv, g, a.layers, a.Hkv) + (key_base + kr) % kPageTokens;
                  *reinterpret_cast<uint4*>(a.pages + row * (D * 2) + cc * 16) = val;
                }
              }
            }
          }
          if (any) __syncwarp();
        }
      }
      // ---- S^T = K Q^T: 2 m-tiles of 16 keys; two accumulators per tile (even
      // and odd k-steps) keep the dependent chains short ----
      float st[2][2][4];
  #pragma unroll
      for (int mt = 0; mt < 2; ++mt)
  #pragma unroll
        for (int h = 0; h < 2; ++h) st[mt][h][0] = st[mt][h][1] = st[mt][h][2] = st[mt][h][3] = 0.f;
      if (Q8 && q8u) {
        // fragments straight from the codes: native row gq + 8 hh of m-tile mt
        // is key kappa = 8 (gq >> 1) + 4 mt + 2 hh + (gq & 1) (the key order
        // the V^T fragments below use); this lane's k-step k takes dims
        // (D / 4) tq + 4 k .. + 3, and the f16 q fragments follow the same order
        const int g1 = gq & 1;
        const uint8_t* kc = half + (gq >> 1) * 8 * D + g1 * D;
        const uint2* qf2 = reinterpret_cast<const uint2*>(q16);
  #pragma unroll
        for (int h = 0; h < D / 64; ++h) {
          uint4 kw[2][2];
  #pragma unroll
          for (int mt = 0; mt < 2; ++mt)
  #pragma unroll
            for (int hh = 0; hh < 2; ++hh) {
              const int lo = 4 * mt + 2 * hh + g1;  // kappa & 7
              const int off = (4 * mt + 2 * hh) * D + (D == 128 ? (((2 * tq + h) ^ lo) << 4) : 16 * tq);
              kw[mt][hh] = *reinterpret_cast<const uint4*>(kc + off);
            }
  #pragma unroll
          for (int kq = 0; kq < 4; ++kq) {
            const int k = 4 * h + kq;
            const uint2 qb = row_ok ? qf2[k * 32 + lane] : make_uint2(0u, 0u);
  #pragma unroll
            for (int mt = 0; mt < 2; ++mt) {
              const uint32_t wl = kq == 0 ? kw[mt][0].x : kq == 1 ? kw[mt][0].y : kq == 2 ? kw[mt][0].z : kw[mt][0].w;
              const uint32_t wh = kq == 0 ? kw[mt][1].x : kq == 1 ? kw[mt][1].y : kq == 2 ? kw[mt][1].z : kw[mt][1].w;
              mma_16816_f16(st[mt][k & 1], code2_f16(wl, 0x4140u), code2_f16(wh, 0x4140u), code2_f16(wl, 0x4342u),
                            code2_f16(wh, 0x4342u), qb.x, qb.y);
            }
          }
        }
      } else {
        // K fragments are loaded one group of two k-steps ahead of the MMAs
        // that use them (the asm statements keep their order), so a warp
        // waits for ldmatrix once per group instead of once per MMA
        uint32_t ka[2][2][2][4];  // [buffer][k-step in group][mt][reg]
        auto load_k = [&](int grp, uint32_t(&dst)[2][2][4]) {
  #pragma unroll
          for (int kq = 0; kq < 2; ++kq)
  #pragma unroll
            for (int mt = 0; mt < 2; ++mt)
              ldsm_x4(kt + sw_off<D>(16 * mt + (lane & 7) + ((lane >> 3) & 1) * 8, 2 * (2 * grp + kq) + (lane >> 4)),
                      dst[kq][mt][0], dst[kq][mt][1], dst[kq][mt][2], dst[kq][mt][3]);
        };
        load_k(0, ka[0]);
  #pragma unroll
        for (int grp = 0; grp < KS / 2; ++grp) {
          if (grp + 1 < KS / 2) load_k(grp + 1, ka[(grp + 1) & 1]);
  #pragma unroll
          for (int kq = 0; kq < 2; ++kq)
  #pragma unroll
            for (int mt = 0; mt < 2; ++mt) {
              const int k = 2 * grp + kq;
              const uint32_t(&f)[4] = ka[grp & 1][kq][mt];
              mma_16816(st[mt][k & 1], f[0], f[1], f[2], f[3], qa0[k], qa2[k]);
            }
        }
        // the first V^T fragments do not depend on the softmax: start them now
        load_v(0, va[0]);
      }
      // ---- online softmax per row 2tq + j (value (mt, hh, j): key 16 mt + gq + 8 hh) ----
      float sv[2][2][2];  // [mt][hh][j]
  #pragma unroll
      for (int mt = 0; mt < 2; ++mt)
  #pragma unroll
        for (int hh = 0; hh < 2; ++hh)
  #pragma unroll
          for (int j = 0; j < 2; ++j) sv[mt][hh][j] = st[mt][0][2 * hh + j] + st[mt][1][2 * hh + j];
      float alpha[2], mu[2];
  #pragma unroll
      for (int j = 0; j < 2; ++j) {
        const bool own_ok = (2 * tq + j < R) && (owner == -1 || owner == own_r[j]);
        float tmax = -INFINITY;
  #pragma unroll
        for (int mt = 0; mt < 2; ++mt)
  #pragma unroll
          for (int hh = 0; hh < 2; ++hh) {
            const int kp = key_base + (q8u ? 8 * (gq >> 1) + 4 * mt + 2 * hh + (gq & 1) : 16 * mt + 8 * hh + gq);
            sv[mt][hh][j] = (own_ok && kp <= pos_r[j]) ? sv[mt][hh][j] * cu : -INFINITY;
            tmax = fmaxf(tmax, sv[mt][hh][j]);
          }
        tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, 4));
        tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, 8));
        tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, 16));
        const float m_new = fmaxf(m[j], tmax);
        mu[j] = (m_new == -INFINITY) ? 0.f : m_new;
        alpha[j] = (m_new == m[j]) ? 1.f : fast_exp2(m[j] - mu[j]);
        m[j] = m_new;
      }
      // P^T B-fragments: keys 16 kk + 2tq.. (b0) and 16 kk + 8 + 2tq.. (b1), row gq
      uint32_t pb[2][2];
  #pragma unroll
      for (int mt = 0; mt < 2; ++mt)
  #pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
          const float p0 = fast_exp2(sv[mt][hh][0] - mu[0]), p1 = fast_exp2(sv[mt][hh][1] - mu[1]);
          l[0] = (mt == 0 && hh == 0 ? l[0] * alpha[0] : l[0]) + p0;
          l[1] = (mt == 0 && hh == 0 ? l[1] * alpha[1] : l[1]) + p1;
          pb[mt][hh] = movmatrix_t(q8u ? pack_f16x2(p0 * s_v, p1 * s_v) : pack_bf16x2(p0, p1));
        }
  #pragma unroll
      for (int md = 0; md < MD; ++md) {
        o[md][0] *= alpha[0];
        o[md][1] *= alpha[1];
        o[md][2] *= alpha[0];
        o[md][3] *= alpha[1];
      }
      // ---- O^T += V^T P^T: MD m-tiles of 16 dims, 2 k-steps of 16 keys ----
      if (Q8 && q8u) {
        // native column 2tq + i (+ 8) of k-step kk is key 8 tq + 4 kk + i (+ 2):
        // the row's 8 bytes at key 8 tq serve both k-steps
        const uint8_t* vc = half + Lay::kUnitBytes / 2 + gq * kUnit + 8 * tq;
  #pragma unroll
        for (int md = 0; md < MD; ++md) {
          const uint2 w0 = *reinterpret_cast<const uint2*>(vc + 16 * md * kUnit);
          const uint2 w1 = *reinterpret_cast<const uint2*>(vc + (16 * md + 8) * kUnit);
  #pragma unroll
          for (int kk = 0; kk < 2; ++kk) {
            const uint32_t wl = kk ? w0.y : w0.x, wh = kk ? w1.y : w1.x;
            mma_16816_f16(o[md], codes2_f16(wl, 0x4140u, vmul, vadd), codes2_f16(wh, 0x4140u, vmul, vadd),
                          codes2_f16(wl, 0x4342u, vmul, vadd), codes2_f16(wh, 0x4342u, vmul, vadd), pb[kk][0],
                          pb[kk][1]);
          }
        }
      } else {
        // group 0 was loaded before the softmax; each later group is loaded
        // while the MMAs of the one before it issue
  #pragma unroll
        for (int grp = 0; grp < kVGroups; ++grp) {
          if (grp + 1 < kVGroups) load_v(grp + 1, va[(grp + 1) & 1]);
  #pragma unroll
          for (int i = 0; i < kVG; ++i) {
            const int it = grp * kVG + i, kk = it / MD, md = it % MD;
            const uint32_t(&f)[4] = va[grp & 1][i];
            mma_16816(o[md], f[0], f[1], f[2], f[3], pb[kk][0], pb[kk][1]);
          }
        }
      }
  };

  if constexpr (!Q8) {
    for (int i = warp, use = 0; i < n; i += kWarps, ++use) {
      const bool ok = __all_sync(0xffffffffu, mbar_wait(&full[warp], use & 1, abort_flag, a.err));
      if (!ok) {
        volatile int no_abort = 0;  // unwinding: let this slot's copy land first
        if (lane == 0) mbar_wait(&full[warp], use & 1, &no_abort, a.err);
        __syncwarp();
        break;
      }
      if (lane == 0 && use == 0 && warp == 0) KVR_STAGE(g_stage_decode, a.layer, 3);
      if (kWarps == 6 && lane == 0 && use == 1) KVR_STAGE(g_stage_decode, a.layer, 22 + warp);
      run_unit(i, unit_page, nullptr);
      __syncwarp();
      if (lane == 0) KVR_STAGE(g_stage_decode, a.layer, 4 + warp);
      if (kWarps == 6 && lane == 0 && use == 0) KVR_STAGE(g_stage_decode, a.layer, 10 + warp);
      if (lane == 0 && i + kWarps < n) unit_page = issue(i + kWarps, 0);  // refill this warp's slot
    }
  } else {
    // Up to two units in flight per warp: an int8 unit takes one half of the
    // slot (its K region or its V region, barrier 2 warp + half), a bf16 unit
    // the whole slot (barrier 2 warp).  The schedule is the same in every
    // lane; lane 0 issues the copies.
    auto is8 = [&](int i) {
      int kb, ow, sl;
      um.locate(bd, u0 + i, &kb, &ow, &sl);
      return kb / kPageTokens < a.q8_n[ow < 0 ? 0 : ow];
    };
    auto half_ptr = [&](int h) -> const uint8_t* {
      return smem + (h ? Lay::kV : Lay::kK) + warp * Lay::kUnitBytes;
    };
    int f_u = warp < n ? warp : -1, f_h = 0, f_pg = unit_page;  // front unit
    bool f_8 = f_u >= 0 && is8(f_u);
    int s_u = -1, s_h = 1, s_pg = -1;  // second unit (int8 only, behind an int8 front)
    int nxt = warp + kWarps;
    uint32_t par = 0;  // phase parity of the two half barriers
    auto fill = [&]() {
      if (f_u < 0 && nxt < n) {
        f_u = nxt;
        f_h = 0;
        f_8 = is8(nxt);
        nxt += kWarps;
        if (lane == 0) f_pg = issue(f_u, 0);
      }
      if (f_u >= 0 && f_8 && s_u < 0 && nxt < n && is8(nxt)) {
        s_u = nxt;
        s_h = 1 - f_h;
        nxt += kWarps;
        if (lane == 0) s_pg = issue(s_u, s_h);
      }
    };
    fill();
    while (f_u >= 0) {
      const int bi = 2 * warp + f_h;
      const bool ok = __all_sync(0xffffffffu, mbar_wait(&full[bi], (par >> f_h) & 1, abort_flag, a.err));
      if (!ok) {
        volatile int no_abort = 0;  // unwinding: let the copies in flight land first
        if (lane == 0) {
          mbar_wait(&full[bi], (par >> f_h) & 1, &no_abort, a.err);
          if (s_u >= 0) mbar_wait(&full[2 * warp + s_h], (par >> s_h) & 1, &no_abort, a.err);
        }
        __syncwarp();
        break;
      }
      par ^= 1u << f_h;
      run_unit(f_u, f_pg, half_ptr(f_h));
      __syncwarp();
      f_u = s_u;
      f_h = s_h;
      f_pg = s_pg;
      f_8 = s_u >= 0;
      s_u = -1;
      fill();
    }
  }

  // ---- merge the warp states (rows < R) ----
  // row sums: the lanes of one tq hold disjoint key shares of rows 2tq, 2tq + 1
#pragma unroll
  for (int j = 0; j < 2; ++j) {
    l[j] += __shfl_xor_sync(0xffffffffu, l[j], 4);
    l[j] += __shfl_xor_sync(0xffffffffu, l[j], 8);
    l[j] += __shfl_xor_sync(0xffffffffu, l[j], 16);
  }
  if (threadIdx.x == 0) KVR_STAGE(g_stage_decode, a.layer, 16);
  // Each warp leaves its state in the K half of its own slot (its units are
  // consumed): fp32 [row][kStride] = O^T columns (relative to the warp's
  // maximum), then the maximum and the row sum.
  auto wstate = [&](int w) -> float* { return reinterpret_cast<float*>(smem + Lay::kK + w * Lay::kUnitBytes); };
#pragma unroll
  for (int j = 0; j < 2; ++j) {
    const int r = 2 * tq + j;
    if (r < R) {
      float* row = wstate(warp) + r * stride;
#pragma unroll
      for (int md = 0; md < MD; ++md) {
        row[16 * md + gq] = o[md][j];
        row[16 * md + 8 + gq] = o[md][2 + j];
      }
      if (gq == 0) {
        row[D] = m[j];
        row[D + 1] = l[j];
      }
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) KVR_STAGE(g_stage_decode, a.layer, 17);
  // Row r of this CTA's partial: the warps' weights exp2(m_w - M) relative to
  // the CTA maximum M (exp2 domain); *L_out = sum_w weight_w l_w.
  auto cta_weights = [&](int r, float (&wts)[kWarps], float* M_out, float* L_out) {
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) {
      wts[w] = wstate(w)[r * stride + D];
      M = fmaxf(M, wts[w]);
    }
    float L = 0.f;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) {
      wts[w] = M == -INFINITY ? 0.f : fast_exp2(wts[w] - M);
      L = fmaf(wts[w], wstate(w)[r * stride + D + 1], L);
    }
    *M_out = M;
    *L_out = L;
  };
  // columns c0 .. c0 + 3 of row r: sum_w weight_w O_w
  auto cta_part4 = [&](int r, int c0, const float (&wts)[kWarps]) -> float4 {
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int w = 0; w < kWarps; ++w) {
      const float4 v = *reinterpret_cast<const float4*>(wstate(w) + r * stride + c0);
      acc.x = fmaf(wts[w], v.x, acc.x);
      acc.y = fmaf(wts[w], v.y, acc.y);
      acc.z = fmaf(wts[w], v.z, acc.z);
      acc.w = fmaf(wts[w], v.w, acc.w);
    }
    return acc;
  };
  // output row r, columns c0 .. c0 + 3 (and its log-sum-exp with column 0)
  auto store4 = [&](int r, int c0, float4 acc, float lsum, float M) {
    const int t = r / a.G, h = g * a.G + r % a.G;
    const int64_t orow = static_cast<int64_t>(t) * a.Hq + h;
    const bool ok = lsum > 0.f;
    uint2 pk;
    pk.x = pack_bf16x2(ok ? acc.x / lsum : 0.f, ok ? acc.y / lsum : 0.f);
    pk.y = pack_bf16x2(ok ? acc.z / lsum : 0.f, ok ? acc.w / lsum : 0.f);
    *reinterpret_cast<uint2*>(a.out + orow * D + c0) = pk;
    if (c0 == 0 && a.lse != nullptr) a.lse[orow] = ok ? (M + log2f(lsum)) * kLn2 : -INFINITY;
  };
  if (S == 1) {
    for (int i = threadIdx.x; i < R * (D / 4); i += kThreads) {
      const int r = i / (D / 4), c0 = 4 * (i % (D / 4));
      float wts[kWarps], M, L;
      cta_weights(r, wts, &M, &L);
      store4(r, c0, cta_part4(r, c0, wts), L, M);
    }
    if (threadIdx.x == 0) KVR_STAGE(g_stage_decode, a.layer, 21);
    return;  // uniform over the launch (one split means no cluster)
  }

  // ---- the splits of this KV head are the CTAs of one cluster ----
  // CTA k owns output columns [k cw, k cw + cw) (cw a multiple of 4; the last
  // owners' slices may be short or empty).  Every CTA pushes each owner its
  // weighed partial of that slice (16-byte asynchronous stores) and its rows'
  // (M, L), which count down the owner's receive barrier; each owner merges its
  // slice over the splits.  Both steps spread each sum over lanes and add the
  // lanes' shares in a fixed shuffle tree, so the result does not depend on
  // timing.
  cluster_wait();  // every receive barrier of the cluster is initialised
  if (threadIdx.x == 0) KVR_STAGE(g_stage_decode, a.layer, 18);
  {
    // LPI lanes per (row, 4 columns) item (one with 6 warps: a round of the
    // CTA's warps covers every item; two with 12, lane half h taking warps
    // h kWarps/2 .. h kWarps/2 + kWarps/2 - 1); warp-uniform rounds
    constexpr int LPI = kWarps <= 6 ? 1 : 2;
    constexpr int HW = kWarps / LPI;
    constexpr int IPW = 32 / LPI;  // items per warp and round
    const int h = LPI == 2 ? (lane & 1) : 0;
    const int nv = R * (D / 4);
    for (int i0 = warp * IPW; i0 < nv; i0 += kWarps * IPW) {
      const int i = i0 + lane / LPI;
      const bool live = i < nv;
      const int r = live ? i / (D / 4) : 0, c0 = live ? 4 * (i % (D / 4)) : 0;
      float mw[HW];
      float M = -INFINITY;
#pragma unroll
      for (int k = 0; k < HW; ++k) {
        mw[k] = wstate(h * HW + k)[r * stride + D];
        M = fmaxf(M, mw[k]);
      }
      if (LPI == 2) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, 1));
      float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
      float L = 0.f;
#pragma unroll
      for (int k = 0; k < HW; ++k) {
        const float* sw = wstate(h * HW + k) + r * stride;
        const float x = M == -INFINITY ? 0.f : fast_exp2(mw[k] - M);
        const float4 v = *reinterpret_cast<const float4*>(sw + c0);
        acc.x = fmaf(x, v.x, acc.x);
        acc.y = fmaf(x, v.y, acc.y);
        acc.z = fmaf(x, v.z, acc.z);
        acc.w = fmaf(x, v.w, acc.w);
        L = fmaf(x, sw[D + 1], L);
      }
      if (LPI == 2) {
        acc.x += __shfl_xor_sync(0xffffffffu, acc.x, 1);
        acc.y += __shfl_xor_sync(0xffffffffu, acc.y, 1);
        acc.z += __shfl_xor_sync(0xffffffffu, acc.z, 1);
        acc.w += __shfl_xor_sync(0xffffffffu, acc.w, 1);
        L += __shfl_xor_sync(0xffffffffu, L, 1);
      }
      if (live && h == 0) {
        const int dest = c0 / cw, cc = c0 - dest * cw;
        const uint32_t rb = map_cluster_smem(smem_u32(recv), static_cast<uint32_t>(dest));
        const uint32_t bar = map_cluster_smem(smem_u32(recv_bar), static_cast<uint32_t>(dest));
        st_async_v4_f32(rb + ((split * R + r) * cw + cc) * 4, acc, bar);
        if (cc == 0) st_async_v2_f32(rb + (S * R * cw + (split * R + r) * 2) * 4, M, L, bar);
      }
    }
  }
  if (threadIdx.x == 0) KVR_STAGE(g_stage_decode, a.layer, 19);
  const int C = a.n_clusters;
  const int my_cw = max(0, min(D, (split + 1) * cw) - split * cw);  // this CTA's slice
  if (my_cw == 0) return;  // owns no columns (and, with several clusters, counts nothing)
  bool recv_ok = mbar_wait_cluster(recv_bar, 0, a.err);
  // A split is late (the error word is set).  Every CTA of the cluster pushes
  // all of its bytes once its own waits have ended: at most one of them runs
  // to the limit (a timeout sets the abort flag, and the CTA's later waits
  // then return at once), and the cluster barrier before the pushes only
  // waits for arrivals made before the grid dependency.  So the pushes into
  // this CTA land within a few limits; its shared memory is kept alive that
  // long (no CTA exits while a peer may still write to it), and only then is
  // the merge given up.  With several clusters the arrival is still counted
  // below.
  for (int extra = 0; !recv_ok && extra < 4; ++extra) recv_ok = mbar_wait_cluster(recv_bar, 0, a.err);
  recv_ok = __all_sync(0xffffffffu, recv_ok);  // warp-uniform: the merge below shuffles
  if (threadIdx.x == 0) KVR_STAGE(g_stage_decode, a.layer, 20);
  if (!recv_ok && C == 1) return;
  const float* rml = recv + S * R * cw;  // [split][row][M, L]
  constexpr int PF = decode_part_floats(D);
  float* const mypart = C > 1 ? a.part + (static_cast<int64_t>(g) * kDecodeMaxClusters + cl) * PF : nullptr;
  {
    // one 4-lane group per (row, 4 columns) item of this CTA's slice, lane j
    // of the group holding splits j, j + 4, j + 8, j + 12 (summed in that
    // order, then across the group in a fixed shuffle tree); warp-uniform rounds
    static_assert(kDecodeMaxSplits == 16, "four splits per lane of a 4-lane group");
    const int j = lane & 3;
    const int nit = recv_ok ? R * (my_cw / 4) : 0;
    for (int i0 = warp * 8; i0 < nit; i0 += kWarps * 8) {
      const int it = i0 + (lane >> 2);
      const bool live = it < nit;
      const int r = live ? it / (my_cw / 4) : 0, cc = live ? 4 * (it % (my_cw / 4)) : 0;
      float mj[4];
      float M = -INFINITY;
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int jj = j + 4 * k;
        mj[k] = (live && jj < S) ? rml[(jj * R + r) * 2] : -INFINITY;
        M = fmaxf(M, mj[k]);
      }
      M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, 1));
      M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, 2));
      float s[5] = {0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int jj = j + 4 * k;
        const bool have = live && jj < S;
        const float x = (have && M != -INFINITY) ? fast_exp2(mj[k] - M) : 0.f;
        const float4 v = have ? *reinterpret_cast<const float4*>(recv + (jj * R + r) * cw + cc)
                              : make_float4(0.f, 0.f, 0.f, 0.f);
        s[0] = fmaf(x, v.x, s[0]);
        s[1] = fmaf(x, v.y, s[1]);
        s[2] = fmaf(x, v.z, s[2]);
        s[3] = fmaf(x, v.w, s[3]);
        s[4] = have ? fmaf(x, rml[(jj * R + r) * 2 + 1], s[4]) : s[4];
      }
#pragma unroll
      for (int off = 1; off <= 2; off <<= 1)
#pragma unroll
        for (int q = 0; q < 5; ++q) s[q] += __shfl_xor_sync(0xffffffffu, s[q], off);
      // lane q of the group finalises column cc + q
      if (live) {
        const float av = j == 0 ? s[0] : j == 1 ? s[1] : j == 2 ? s[2] : s[3];
        const float lsum = s[4];
        const int col = split * cw + cc + j;
        if (C == 1) {
          const int t = r / a.G, hq = g * a.G + r % a.G;
          const int64_t orow = static_cast<int64_t>(t) * a.Hq + hq;
          a.out[orow * D + col] = __bfloat16_as_ushort(__float2bfloat16_rn(lsum > 0.f ? av / lsum : 0.f));
          if (col == 0 && a.lse != nullptr) a.lse[orow] = lsum > 0.f ? (M + log2f(lsum)) * kLn2 : -INFINITY;
        } else {
          mypart[r * D + col] = av;
          if (cc == 0 && j == 0) {
            float* ml = mypart + kDecodeMaxRows * D + (split * kDecodeMaxRows + r) * 2;
            ml[0] = M;
            ml[1] = lsum;
          }
        }
      }
    }
  }
  if (C == 1) {
    if (threadIdx.x == 0) KVR_STAGE(g_stage_decode, a.layer, 21);
    return;
  }

  // ---- several clusters per KV head: the last to arrive merges ----
  // Owner CTA k of every cluster left its slice above and counts itself; the
  // one that completes the count merges the clusters' slices in cluster order
  // (the same result whichever arrives last) and resets the count.
  __threadfence();  // every writer's slice is visible before the count moves
  __syncthreads();
  if (threadIdx.x == 0) {
    int* cnt = a.cnt + g * kDecodeMaxSplits + split;
    const int old = atomicAdd(cnt, 1);
    misc[13] = old == C - 1;
    if (old == C - 1) atomicExch(cnt, 0);
  }
  __syncthreads();
  if (!misc[13]) return;
  __threadfence();
  const float* part0 = a.part + static_cast<int64_t>(g) * kDecodeMaxClusters * PF;
  for (int e = threadIdx.x; e < R * (my_cw / 4); e += kThreads) {
    const int r = e / (my_cw / 4), cc = 4 * (e % (my_cw / 4));
    const int col = split * cw + cc;
    float mx[kDecodeMaxClusters], sm[kDecodeMaxClusters];
    float M = -INFINITY;
#pragma unroll
    for (int j = 0; j < kDecodeMaxClusters; ++j) {
      const float* ml = part0 + min(j, C - 1) * PF + kDecodeMaxRows * D + (split * kDecodeMaxRows + r) * 2;
      mx[j] = j < C ? __ldcg(ml) : -INFINITY;
      sm[j] = j < C ? __ldcg(ml + 1) : 0.f;
      M = fmaxf(M, mx[j]);
    }
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    float lsum = 0.f;
#pragma unroll
    for (int j = 0; j < kDecodeMaxClusters; ++j) {  // cluster order
      const float x = (M == -INFINITY || j >= C) ? 0.f : fast_exp2(mx[j] - M);  // 0 for an empty cluster too
      const float4 v = __ldcg(reinterpret_cast<const float4*>(part0 + min(j, C - 1) * PF + r * D + col));
      acc.x = fmaf(x, v.x, acc.x);
      acc.y = fmaf(x, v.y, acc.y);
      acc.z = fmaf(x, v.z, acc.z);
      acc.w = fmaf(x, v.w, acc.w);
      lsum = fmaf(x, sm[j], lsum);
    }
    store4(r, col, acc, lsum, M);
  }
}

template <int D, bool FUSED, bool Q8, int W>
cudaError_t launch_decode_d(const DecodeArgs& a, const SmallBatch& b, cudaStream_t st) {
  static PerDeviceOnce setup;
  const cudaError_t e = setup.run([] {
    cudaError_t r = cudaFuncSetAttribute(decode_kernel<D, FUSED, Q8, W>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         DecLayout<D, W>::kAlloc);
    if (r == cudaSuccess)
      r = cudaFuncSetAttribute(decode_kernel<D, FUSED, Q8, W>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    return r;
  });
  if (e != cudaSuccess) return e;
  return launch_kernel(decode_kernel<D, FUSED, Q8, W>, dim3(a.Hkv * a.n_splits * a.n_clusters), dim3(W * 32),
                       DecLayout<D, W>::kAlloc, st, static_cast<unsigned>(a.n_splits), a, b);
}

// Clusters of c CTAs (c = 1..16) of the W-warp kernel that can be resident at
// once on the current device (a table per device, filled on its first use).
template <int D, int W>
const int* active_clusters_d() {
  static int table[kMaxDevices][17];
  static PerDeviceOnce filled;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
    cudaGetLastError();
    static const int none[17] = {0, 1};
    return none;
  }
  int* t = table[dev];
  filled.run([t] {
    for (int c = 0; c <= 16; ++c) t[c] = 0;
    t[1] = 1;
    if (cudaFuncSetAttribute(decode_kernel<D, false, false, W>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             DecLayout<D, W>::kAlloc) != cudaSuccess ||
        cudaFuncSetAttribute(decode_kernel<D, false, false, W>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) !=
            cudaSuccess) {
      cudaGetLastError();
      return cudaSuccess;  // one CTA per KV head: no cluster is ever requested
    }
    for (int c = 1; c <= 16; ++c) {
      cudaLaunchConfig_t cfg = {};
      cfg.gridDim = dim3(c);
      cfg.blockDim = dim3(W * 32);
      cfg.dynamicSmemBytes = DecLayout<D, W>::kAlloc;
      cudaLaunchAttribute attr[1];
      attr[0].id = cudaLaunchAttributeClusterDimension;
      attr[0].val.clusterDim.x = c;
      attr[0].val.clusterDim.y = 1;
      attr[0].val.clusterDim.z = 1;
      cfg.attrs = attr;
      cfg.numAttrs = 1;
      int n = 0;
      if (cudaOccupancyMaxActiveClusters(&n, decode_kernel<D, false, false, W>, &cfg) == cudaSuccess) t[c] = n;
      cudaGetLastError();
    }
    return cudaSuccess;
  });
  return t;
}

}  // namespace

int decode_units(const SmallBatch& bd) {
  int total = bd.shared_pages * (kPageTokens / kUnit);
  for (int b = 0; b < bd.n_seqs; ++b) {
    const int maxpos = bd.start[b] + (bd.cu_q[b + 1] - bd.cu_q[b]) - 1;
    const int keys = maxpos + 1 - bd.shared_pages * kPageTokens;
    if (keys > 0) total += (keys + kUnit - 1) / kUnit;
  }
  return total;
}

// Splits per KV head and warps per CTA.  Up to 144 units per head (two passes
// of 72 warps), 12 CTAs of 6 warps per head: two such CTAs fit on an SM, so
// the next decode launch is resident beside this one and starts at once.
// Measured on GB300 (Qwen3-4B shapes, 8 KV heads, 36-layer graphs of decode
// steps), 6-warp CTAs x 12 per head against the 12-warp rule below: 33 units
// 5.18 us (5.55), 65 units 5.57 (6.16), 94 units 6.76 (6.72), 120 units 7.17
// (7.25), 121 units 7.28 (7.95); from 157 units on the 12-warp CTAs win (157:
// 8.61 against 8.95 at 16 x 6 warps; 1025: 27.2 against 28.2).  The int8
// variant keeps 12 warps.
// Otherwise 12 warps: as many CTAs as there are 32-key units, capped at the
// largest cluster size of which `heads` clusters are resident together; a
// single CTA when one pass of its warps covers every unit.  Short contexts
// (each CTA's units fit in two passes of its warps at the smaller cap) use the
// largest cluster size of which 2 x `heads` clusters fit: then the next decode
// launch becomes resident beside this one and its L2 prefetch overlaps this
// launch's merge.
int decode_splits(int d, int heads, int units, bool q8, int* clusters, int* warps) {
  *clusters = 1;
  *warps = 12;
  // 6-warp CTAs (two per SM, so the next launch is resident beside this one):
  // up to 12 per KV head, two passes of their warps at most (for int8 pages,
  // one pass of two units in flight per warp).  Measured (36-layer graphs,
  // 120-121 units per head): 7.5-7.7 us per step at 12 CTAs per head, 9.0-9.4
  // at 14 or 16, whose clusters do not fit beside the next launch's (its CTAs
  // then start over about 2 us again).  bf16 units that one pass covers take
  // as few CTAs as that needs but at least 8 (a smaller merge): 33 units 4.79
  // -> 4.56 us, 49 units 4.99 -> 4.70.
  if (units > 12 && units <= 12 * 6 * 2) {
    const int* t6 = d == 64 ? active_clusters_d<64, 6>() : active_clusters_d<128, 6>();
    if (t6[12] >= heads) {
      *warps = 6;
      if (!q8 && units <= 12 * 6) return std::max(8, (units + 5) / 6);  // one pass of the 6 warps
      return 12;
    }
  }
  const int* t = d == 64 ? active_clusters_d<64, 12>() : active_clusters_d<128, 12>();
  constexpr int kWarps = 12;
  int cap = 1, cap2 = 1;
  for (int c = 16; c >= 1; --c)
    if (t[c] >= heads) {
      cap = c;
      break;
    }
  for (int c = 16; c >= 1; --c)
    if (t[c] >= 2 * heads) {
      cap2 = c;
      break;
    }
  if (units <= kWarps) return 1;  // one CTA covers every unit in one pass
  // Between the two-launch cap and 200 units, 10 or 12 CTAs per head when they
  // need fewer passes of the warps than the cap (fewest passes first, then 10).
  // Measured on GB300 (Qwen3-4B shapes, 8 KV heads, cap2 = 6, 36-layer graphs
  // of decode steps): 94 units 6.72 us at 10 CTAs (7.07 at 8, 7.51 at 6); 120
  // units 7.21 at 10 (7.99 at 12, 8.11 at 6); 121 units 7.91 at 12 (8.11 at
  // 11, 8.25 at 10 or 6); 157 units 8.57 at 10 (9.06 at 8, 9.63 at 12, 10.04
  // at 6, 9.56-9.58 over 3-4 clusters per head).
  if (cap2 < 10 && units > cap2 * kWarps && units <= 200) {
    auto passes = [&](int s2) { return ((units + s2 - 1) / s2 + kWarps - 1) / kWarps; };
    int best = cap2;
    for (int s2 : {10, 12})
      if (s2 <= kDecodeMaxSplits && t[s2] >= heads && passes(s2) < passes(best)) best = s2;
    if (best != cap2) return best;
  }
  if (units <= cap2 * 2 * kWarps) return std::max(1, std::min(units, cap2));
  if (units > cap * 2 * kWarps) {
    // Long contexts: a head's splits over several clusters (their partials
    // merged through the pool header), as many CTAs as are resident at once;
    // among equal totals the larger cluster.
    int best_s = cap, best_c = 1;
    for (int s = std::min(cap, kDecodeMaxSplits); s >= 2; --s)
      for (int c = kDecodeMaxClusters; c >= 2; --c)
        if (t[s] >= heads * c && s * c > best_s * best_c) {
          best_s = s;
          best_c = c;
        }
    *clusters = best_c;
    return std::max(1, std::min(units, best_s));
  }
  return std::max(1, std::min(units, cap));
}

cudaError_t launch_decode(const DecodeArgs& a, const SmallBatch& b, int d, bool fused, cudaStream_t st) {
  if (a.Hkv * a.n_splits == 0 || b.T == 0) return cudaSuccess;
  if (a.n_clusters < 1 || a.n_clusters > kDecodeMaxClusters || a.n_splits > kDecodeMaxSplits ||
      (a.n_clusters > 1 && (a.n_splits < 2 || a.part == nullptr || a.cnt == nullptr)))
    return cudaErrorInvalidValue;
  bool q8 = false;
  for (int k = 0; k < b.n_seqs && k < kDecodeMaxRows; ++k) q8 = q8 || a.q8_n[k] > 0;
  if (q8 && a.q8_table == nullptr) return cudaErrorInvalidValue;
  if (q8 && a.n_warps == 6) {  // (two int8 units in flight per warp)
    if (fused)
      return d == 64 ? launch_decode_d<64, true, true, 6>(a, b, st) : launch_decode_d<128, true, true, 6>(a, b, st);
    return d == 64 ? launch_decode_d<64, false, true, 6>(a, b, st) : launch_decode_d<128, false, true, 6>(a, b, st);
  }
  if (q8) {
    if (fused)
      return d == 64 ? launch_decode_d<64, true, true, 12>(a, b, st) : launch_decode_d<128, true, true, 12>(a, b, st);
    return d == 64 ? launch_decode_d<64, false, true, 12>(a, b, st) : launch_decode_d<128, false, true, 12>(a, b, st);
  }
  if (a.n_warps == 6) {
    if (fused)
      return d == 64 ? launch_decode_d<64, true, false, 6>(a, b, st) : launch_decode_d<128, true, false, 6>(a, b, st);
    return d == 64 ? launch_decode_d<64, false, false, 6>(a, b, st) : launch_decode_d<128, false, false, 6>(a, b, st);
  }
  if (fused)
    return d == 64 ? launch_decode_d<64, true, false, 12>(a, b, st) : launch_decode_d<128, true, false, 12>(a, b, st);
  return d == 64 ? launch_decode_d<64, false, false, 12>(a, b, st) : launch_decode_d<128, false, false, 12>(a, b, st);
}

}  // namespace kvr

#ifdef KVR_STAGE_TRACE
extern "C" __attribute__((visibility("default"))) int kvr_stage_read_decode(void* host, int bytes) {
  return static_cast<int>(cudaMemcpyFromSymbol(host, kvr::g_stage_decode, static_cast<size_t>(bytes)));
}
#endif
