// kvr_attn.cu -- causal GQA attention over the paged KV cache on tcgen05/TMEM.
//
// One kernel serves both paths of the paper: the reuse attention of
// continuation/decode tokens over a loaded prefix (Sec. 3.2, Algorithm 2) and
// the full causal prefill attention it replaces (Sec. 1, Sec. 5 Table 1 cost
// (a)).  Both run the same instructions over the same key tiles, which start at
// key 0 and are 128 keys wide, so a row's result depends only on its own query,
// its visible keys and the tile order: with one split per query block, reuse
// rows are bitwise equal to prefill rows (Sec. 3.3, Claim 1).
//
// CTA = one query block (128 packed rows = 128/G tokens x the G query heads of
// one KV head) x one KV head x one key split.  Warp roles:
//   warp 0      TMA producer: Q block once, then K and V tiles into a 2-stage ring
//   warp 1      TMEM owner and MMA issuer: S = Q K^T (128x128, fp32 in TMEM,
//               double buffered), O += P V (128 x d, fp32 in TMEM)
//   warps 2..5  softmax: thread = row = TMEM lane; causal/ownership mask,
//               online softmax in the exp2 domain, P as bf16 into shared memory,
//               O rescale in TMEM, final normalisation and store
// Key tiles: first the pages shared by every sequence of the batch (a loaded
// prefix forked by many consumers: each such tile is staged once per CTA and
// serves every consumer row in it), then each sequence's own pages; a row sees
// key c iff the tile is shared or its own, and c <= its position.
#include <math.h>

#include "kvr_internal.h"
#include "kvr_ptx.cuh"

namespace kvr {
namespace {

constexpr int kStages = 2;
constexpr int kThreads = 192;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kTmemS0 = 0, kTmemS1 = 128, kTmemO = 256;
constexpr float kLn2 = 0.69314718055994530942f;

template <int D>
struct Layout {
  static constexpr int kSub = kBlockRows * 64 * 2;      // one 64-column swizzled sub-tile
  static constexpr int kTile = kBlockRows * D * 2;      // 128 rows x D bf16
  static constexpr int kQ = 0;
  static constexpr int kK = kQ + kTile;
  static constexpr int kV = kK + kStages * kTile;
  static constexpr int kP = kV + kStages * kTile;
  static constexpr int kPBytes = kBlockRows * kPageTokens * 2;
  static constexpr int kBar = kP + kPBytes;
  static constexpr int kMisc = kBar + 256;
  static constexpr int kMiscInts = 16 + kBlockRows;
  static constexpr int kEnd = kMisc + kMiscInts * 4;
  // 1 KB of slack to align the dynamic buffer to the 1024-byte swizzle atom;
  // d = 64 pads to keep one CTA per SM (each CTA allocates all 512 TMEM columns).
  static constexpr int kAlloc = (kEnd + 1024) > 120 * 1024 ? (kEnd + 1024) : 120 * 1024;
};

enum { kBarQ = 0, kBarKFull = 1, kBarVFull = 3, kBarKEmpty = 5, kBarVEmpty = 7, kBarSFull = 9,
       kBarSEmpty = 11, kBarPFull = 13, kBarODone = 14, kBarDrain = 15, kNumBars = 16 };
enum { kMiscTmem = 0, kMiscAbort = 1, kMiscBLo = 2, kMiscBHi = 3, kMiscTotal = 4,
       kMiscBegin = 5, kMiscEnd = 6, kMiscNTile = 16 };

// Sequence holding packed token t: the last b with cu_q[b] <= t (no empty
// sequences in a batch, so cu_q is strictly increasing).
__device__ __forceinline__ int seq_of(const BatchDesc& bd, int t) {
  int lo = 0, hi = bd.n_seqs - 1;
  while (lo < hi) {
    int mid = (lo + hi + 1) >> 1;
    if (bd.cu_q[mid] <= t) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// Walks the key-tile list of one query block: shared tiles 0..shared-1, then
// sequence b_lo's own tiles, b_lo+1's, ...
struct TileCursor {
  int idx, b, jb;
  int b_lo, b_hi, shared;
  const int* ntile;  // own-tile counts of b_lo..b_hi (shared memory)

  __device__ void normalize() {
    while (b <= b_hi && jb >= ntile[b - b_lo]) {
      jb -= ntile[b - b_lo];
      ++b;
    }
  }
  __device__ void init(int start, int blo, int bhi, int sh, const int* nt) {
    b_lo = blo; b_hi = bhi; shared = sh; ntile = nt;
    idx = start; b = b_lo; jb = start > shared ? start - shared : 0;
    normalize();
  }
  __device__ void next() {
    ++idx;
    if (idx > shared) ++jb;
    normalize();
  }
  __device__ int key_base() const { return (idx < shared ? idx : shared + jb) * kPageTokens; }
  __device__ int owner() const { return idx < shared ? -1 : b; }
  __device__ int page_slot_index(const BatchDesc& bd, int* slot) const {
    if (idx < shared) { *slot = bd.slot[b_lo]; return idx; }
    *slot = bd.slot[b < bd.n_seqs ? b : bd.n_seqs - 1];
    return shared + jb;
  }
};

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
attn_kernel(const __grid_constant__ AttnArgs a, const __grid_constant__ BatchDesc bd) {
  using Lay = Layout<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + Lay::kBar);
  int* misc = reinterpret_cast<int*>(smem + Lay::kMisc);
  volatile int* abort_flag = misc + kMiscAbort;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int G = a.G, TB = kBlockRows / G;
  int bid = blockIdx.x;
  const int split = bid % a.n_splits;
  bid /= a.n_splits;
  const int g = bid % a.Hkv;
  bid /= a.Hkv;
  const int rb = a.n_rb - 1 - bid;  // late (longest) query blocks first
  const int tok0 = rb * TB;
  const int tok1 = min(bd.T, tok0 + TB);

  if (threadIdx.x == 0) {
    mbar_init(&bars[kBarQ], 1);
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&bars[kBarKFull + s], 1);
      mbar_init(&bars[kBarVFull + s], 1);
      mbar_init(&bars[kBarKEmpty + s], 1);
      mbar_init(&bars[kBarVEmpty + s], 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(&bars[kBarSFull + s], 1);
      mbar_init(&bars[kBarSEmpty + s], 128);
    }
    mbar_init(&bars[kBarPFull], 128);
    mbar_init(&bars[kBarODone], 1);
    mbar_init(&bars[kBarDrain], 1);
    fence_barrier_init();
    misc[kMiscAbort] = 0;
    // Key-tile plan of this query block and this split's share of it.
    const int b_lo = seq_of(bd, tok0), b_hi = seq_of(bd, tok1 - 1);
    int total = bd.shared_pages;
    for (int b = b_lo; b <= b_hi; ++b) {
      const int tf = max(tok0, bd.cu_q[b]);
      const int tl = min(tok1, bd.cu_q[b + 1]) - 1;
      int nt = 0;
      if (tl >= tf) {
        const int maxpos = bd.start[b] + (tl - bd.cu_q[b]);
        nt = max(0, maxpos / kPageTokens + 1 - bd.shared_pages);
      }
      misc[kMiscNTile + (b - b_lo)] = nt;
      total += nt;
    }
    misc[kMiscBLo] = b_lo;
    misc[kMiscBHi] = b_hi;
    misc[kMiscTotal] = total;
    misc[kMiscBegin] = static_cast<int>(static_cast<int64_t>(total) * split / a.n_splits);
    misc[kMiscEnd] = static_cast<int>(static_cast<int64_t>(total) * (split + 1) / a.n_splits);
  }
  if (warp == 1) {
    tmem_alloc(reinterpret_cast<uint32_t*>(misc + kMiscTmem), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  griddep_wait();  // global memory from here on
  griddep_launch_dependents();

  const uint32_t tmem = static_cast<uint32_t>(misc[kMiscTmem]);
  const int b_lo = misc[kMiscBLo], b_hi = misc[kMiscBHi];
  const int t_begin = misc[kMiscBegin];
  const int n = misc[kMiscEnd] - t_begin;
  const int* ntile = misc + kMiscNTile;

  if (warp == 0) {
    // ------------------------------------------------------------ producer --
    // Lane j looks up the page of tile j (j < 32) so the first tiles' lookups
    // overlap instead of each waiting on the previous one.
    int lane_page = -1;
    if (lane < n) {
      TileCursor lc;
      lc.init(t_begin + lane, b_lo, b_hi, bd.shared_pages, ntile);
      int slot;
      const int pidx = lc.page_slot_index(bd, &slot);
      if (pidx >= 0 && pidx < bd.max_pages) lane_page = bd.page_table[slot * bd.max_pages + pidx];
    }
    int first_pages[32];
#pragma unroll
    for (int j = 0; j < 32; ++j) first_pages[j] = __shfl_sync(0xffffffffu, lane_page, j);
    if (lane == 0 && n > 0) {
      tma_prefetch_desc(&a.tm_q);
      tma_prefetch_desc(&a.tm_kv);
      mbar_arrive_expect_tx(&bars[kBarQ], Lay::kTile);
#pragma unroll
      for (int c = 0; c < D / 64; ++c)
        tma_load_3d(smem + Lay::kQ + c * Lay::kSub, &a.tm_q, &bars[kBarQ], c * 64, g * G, tok0);
      TileCursor cur;
      cur.init(t_begin, b_lo, b_hi, bd.shared_pages, ntile);
      int issued = 0;
      bool ok = true;
      for (int j = 0; j < n && ok; ++j, cur.next()) {
        const int st = j & 1, use = j >> 1;
        int page;
        if (j < 32) {
          page = first_pages[j];
        } else {
          int slot;
          const int pidx = cur.page_slot_index(bd, &slot);
          page = (pidx >= 0 && pidx < bd.max_pages) ? bd.page_table[slot * bd.max_pages + pidx] : -1;
        }
        int64_t rk = kv_row(page, a.layer, 0, g, a.layers, a.Hkv);
        int64_t rv = kv_row(page, a.layer, 1, g, a.layers, a.Hkv);
        if (page < 0 || rv + kPageTokens > a.n_pool_rows) {
          atomicOr(a.err, kDevErrBounds);
          rk = 0;
          rv = 0;
        }
        if (j >= kStages) ok = mbar_wait(&bars[kBarKEmpty + st], (use - 1) & 1, abort_flag, a.err);
        if (!ok) break;
        mbar_arrive_expect_tx(&bars[kBarKFull + st], Lay::kTile);
#pragma unroll
        for (int c = 0; c < D / 64; ++c)
          tma_load_2d(smem + Lay::kK + st * Lay::kTile + c * Lay::kSub, &a.tm_kv,
                      &bars[kBarKFull + st], c * 64, static_cast<int>(rk));
        if (j >= kStages) ok = mbar_wait(&bars[kBarVEmpty + st], (use - 1) & 1, abort_flag, a.err);
        if (!ok) { issued = 2 * j + 1; break; }
        mbar_arrive_expect_tx(&bars[kBarVFull + st], Lay::kTile);
#pragma unroll
        for (int c = 0; c < D / 64; ++c)
          tma_load_2d(smem + Lay::kV + st * Lay::kTile + c * Lay::kSub, &a.tm_kv,
                      &bars[kBarVFull + st], c * 64, static_cast<int>(rv));
        issued = 2 * j + 2;
      }
      if (!ok) {
        // Unwinding: let the copies already in flight land before the CTA exits.
        volatile int no_abort = 0;
        const int last_j = (issued + 1) / 2 - 1;
        for (int j = max(0, last_j - 1); j <= last_j; ++j) {
          mbar_wait(&bars[kBarKFull + (j & 1)], (j >> 1) & 1, &no_abort, a.err);
          if (2 * j + 2 <= issued)
            mbar_wait(&bars[kBarVFull + (j & 1)], (j >> 1) & 1, &no_abort, a.err);
        }
      }
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA --
    if (lane == 0 && n > 0) {
      constexpr uint32_t kIdS = make_idesc_bf16(128, kPageTokens, 0);
      constexpr uint32_t kIdO = make_idesc_bf16(128, D, 1);
      const uint32_t sQ = smem_u32(smem + Lay::kQ);
      const uint32_t sK = smem_u32(smem + Lay::kK);
      const uint32_t sV = smem_u32(smem + Lay::kV);
      const uint32_t sP = smem_u32(smem + Lay::kP);
      bool issued_any = false;
      auto issue_pv = [&](int i) -> bool {
        const int st = i & 1;
        if (!mbar_wait(&bars[kBarPFull], i & 1, abort_flag, a.err)) return false;
        if (!mbar_wait(&bars[kBarVFull + st], (i >> 1) & 1, abort_flag, a.err)) return false;
        tc_fence_after();
#pragma unroll
        for (int kk = 0; kk < kPageTokens / 16; ++kk) {
          const uint64_t ad = make_sdesc_sw128(sP + (kk >> 2) * Lay::kSub + (kk & 3) * 32, 16, 1024);
          const uint64_t bd2 = make_sdesc_sw128(sV + st * Lay::kTile + kk * 2048, Lay::kSub, 1024);
          umma_bf16_ss(tmem + kTmemO, ad, bd2, kIdO, (i > 0 || kk > 0) ? 1u : 0u);
        }
        umma_commit(&bars[kBarODone]);
        umma_commit(&bars[kBarVEmpty + st]);
        return true;
      };
      bool ok = mbar_wait(&bars[kBarQ], 0, abort_flag, a.err);
      for (int j = 0; j < n && ok; ++j) {
        const int st = j & 1, sb = j & 1;
        ok = mbar_wait(&bars[kBarKFull + st], (j >> 1) & 1, abort_flag, a.err);
        if (ok && j >= 2) ok = mbar_wait(&bars[kBarSEmpty + sb], ((j >> 1) - 1) & 1, abort_flag, a.err);
        if (!ok) break;
        tc_fence_after();
        const uint32_t dS = tmem + (sb ? kTmemS1 : kTmemS0);
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint32_t off = (kk >> 2) * Lay::kSub + (kk & 3) * 32;
          const uint64_t ad = make_sdesc_sw128(sQ + off, 16, 1024);
          const uint64_t bd2 = make_sdesc_sw128(sK + st * Lay::kTile + off, 16, 1024);
          umma_bf16_ss(dS, ad, bd2, kIdS, kk > 0 ? 1u : 0u);
        }
        issued_any = true;
        umma_commit(&bars[kBarSFull + sb]);
        umma_commit(&bars[kBarKEmpty + st]);
        if (j >= 1) ok = issue_pv(j - 1);
      }
      if (ok) ok = issue_pv(n - 1);
      if (!ok && issued_any) {
        // Unwinding: wait for the MMAs in flight before TMEM is released.
        volatile int no_abort = 0;
        umma_commit(&bars[kBarDrain]);
        mbar_wait(&bars[kBarDrain], 0, &no_abort, a.err);
      }
    }
  } else {
    // ------------------------------------------------------------ softmax --
    const int quarter = warp & 3;
    const int r = quarter * 32 + lane;
    const uint32_t lane_addr = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
    const int t = tok0 + r / G;
    const int h = g * G + r % G;
    const bool valid = t < tok1;
    int my_b = -2, pos = -1;
    if (valid) {
      my_b = seq_of(bd, t);
      pos = bd.start[my_b] + (t - bd.cu_q[my_b]);
    }
    const float c = a.scale_log2;
    // m: reference maximum (raw score units) of this row's exponents.  It moves
    // only when a tile's maximum exceeds it by more than 2^kLazy in the exp2
    // domain (then O and l are rescaled); otherwise exponents use the stale
    // reference (p <= 2^kLazy).  The final O / l and lse are exact either way.
    constexpr float kLazy = 8.0f;
    float m = -INFINITY, l = 0.f;
    TileCursor cur;
    cur.init(t_begin, b_lo, b_hi, bd.shared_pages, ntile);
    bool ok = true;
    for (int j = 0; j < n; ++j, cur.next()) {
      const int sb = j & 1;
      ok = __all_sync(0xffffffffu, mbar_wait(&bars[kBarSFull + sb], (j >> 1) & 1, abort_flag, a.err));
      if (!ok) break;
      tc_fence_after();
      float s[kPageTokens];
      tmem_ld128(lane_addr + (sb ? kTmemS1 : kTmemS0), s);
      tc_fence_before();
      mbar_arrive(&bars[kBarSEmpty + sb]);

      const int owner = cur.owner();
      int nvis = 0;
      if (owner == -1 || owner == my_b) nvis = min(max(pos - cur.key_base() + 1, 0), kPageTokens);
      if (__any_sync(0xffffffffu, nvis < kPageTokens)) {
#pragma unroll
        for (int k = 0; k < kPageTokens; ++k) s[k] = (k < nvis) ? s[k] : -INFINITY;
      }
      // row maximum over 8 independent partial maxima
      float mx[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) mx[i] = s[i];
#pragma unroll
      for (int k = 8; k < kPageTokens; k += 8)
#pragma unroll
        for (int i = 0; i < 8; ++i) mx[i] = fmaxf(mx[i], s[k + i]);
      const float tmax = fmaxf(fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])),
                               fmaxf(fmaxf(mx[4], mx[5]), fmaxf(mx[6], mx[7])));
      float alpha = 1.f;
      if (tmax != -INFINITY && (m == -INFINITY || (tmax - m) * c > kLazy)) {
        alpha = fast_exp2((m - tmax) * c);  // 0 when nothing was accumulated yet
        m = tmax;
      }
      const float mc = (m == -INFINITY) ? 0.f : m * c;
      // exponentials (packed argument), row sum over 4 packed partial sums
      float2 acc[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f),
                       make_float2(0.f, 0.f)};
#pragma unroll
      for (int k = 0; k < kPageTokens; k += 2) {
        const float2 x = ffma2(make_float2(s[k], s[k + 1]), make_float2(c, c), make_float2(-mc, -mc));
        s[k] = fast_exp2(x.x);
        s[k + 1] = fast_exp2(x.y);
        acc[(k >> 1) & 3] = fadd2(acc[(k >> 1) & 3], make_float2(s[k], s[k + 1]));
      }
      const float2 a01 = fadd2(acc[0], acc[1]), a23 = fadd2(acc[2], acc[3]);
      const float2 a03 = fadd2(a01, a23);
      l = l * alpha + (a03.x + a03.y);

      if (j > 0) {
        ok = __all_sync(0xffffffffu, mbar_wait(&bars[kBarODone], (j - 1) & 1, abort_flag, a.err));
        if (!ok) break;
        tc_fence_after();
        if (__any_sync(0xffffffffu, alpha != 1.f)) {
#pragma unroll 1
          for (int q = 0; q < D / 32; ++q) {
            float o[32];
            tmem_ld32(lane_addr + kTmemO + q * 32, o);
#pragma unroll
            for (int i = 0; i < 32; ++i) o[i] *= alpha;
            tmem_st32(lane_addr + kTmemO + q * 32, o);
          }
        }
      }
      // P row -> shared memory, bf16, 128B-swizzled K-major (two 64-key sub-tiles).
#pragma unroll
      for (int ch = 0; ch < kPageTokens / 8; ++ch) {
        uint4 v;
        v.x = pack_bf16x2(s[8 * ch + 0], s[8 * ch + 1]);
        v.y = pack_bf16x2(s[8 * ch + 2], s[8 * ch + 3]);
        v.z = pack_bf16x2(s[8 * ch + 4], s[8 * ch + 5]);
        v.w = pack_bf16x2(s[8 * ch + 6], s[8 * ch + 7]);
        uint8_t* dst = smem + Lay::kP + (ch >> 3) * Lay::kSub + r * 128 + (((ch & 7) ^ (r & 7)) << 4);
        *reinterpret_cast<uint4*>(dst) = v;
      }
      fence_proxy_async_smem();
      tc_fence_before();
      mbar_arrive(&bars[kBarPFull]);
    }
    if (ok && n > 0)
      ok = __all_sync(0xffffffffu, mbar_wait(&bars[kBarODone], (n - 1) & 1, abort_flag, a.err));
    if (ok) {
      tc_fence_after();
      const float inv_l = (l > 0.f) ? 1.f / l : 0.f;
      const float lse2 = (l > 0.f) ? (m * c + log2f(l)) : -INFINITY;
      const int64_t row = static_cast<int64_t>(t) * a.Hq + h;
      if (a.n_splits == 1) {
#pragma unroll 1
        for (int q = 0; q < D / 32; ++q) {
          float o[32];
          if (n > 0) tmem_ld32(lane_addr + kTmemO + q * 32, o);
#pragma unroll
          for (int i = 0; i < 32; ++i) o[i] = (n > 0) ? o[i] * inv_l : 0.f;
          if (valid) {
            uint4* dst = reinterpret_cast<uint4*>(a.out + row * D + q * 32);
#pragma unroll
            for (int v4 = 0; v4 < 4; ++v4) {
              uint4 w;
              w.x = pack_bf16x2(o[8 * v4 + 0], o[8 * v4 + 1]);
              w.y = pack_bf16x2(o[8 * v4 + 2], o[8 * v4 + 3]);
              w.z = pack_bf16x2(o[8 * v4 + 4], o[8 * v4 + 5]);
              w.w = pack_bf16x2(o[8 * v4 + 6], o[8 * v4 + 7]);
              dst[v4] = w;
            }
          }
        }
        if (valid && a.lse != nullptr) a.lse[row] = lse2 * kLn2;
      } else {
        const int64_t prow = static_cast<int64_t>(split) * bd.T * a.Hq + row;
#pragma unroll 1
        for (int q = 0; q < D / 32; ++q) {
          float o[32];
          if (n > 0) tmem_ld32(lane_addr + kTmemO + q * 32, o);
          if (valid) {
            float4* dst = reinterpret_cast<float4*>(a.part_o + prow * D + q * 32);
#pragma unroll
            for (int v4 = 0; v4 < 8; ++v4)
              dst[v4] = (n > 0) ? make_float4(o[4 * v4] * inv_l, o[4 * v4 + 1] * inv_l,
                                              o[4 * v4 + 2] * inv_l, o[4 * v4 + 3] * inv_l)
                                : make_float4(0.f, 0.f, 0.f, 0.f);
          }
        }
        if (valid) a.part_lse[prow] = lse2;
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// Merge per-split partials (O_s normalised, lse_s in log2 units) of one
// (token, head) row, one warp per row: lane s holds split s's lse (two rounds
// past 32 splits), so every lse arrives in one round of loads; the O loads are
// unrolled so several splits are in flight.  Splits enter the sum in order
// 0, 1, ... (fixed per call).
template <int D>
__global__ void __launch_bounds__(256) combine_kernel(const float* __restrict__ part_o,
                                                      const float* __restrict__ part_lse, int S,
                                                      int T, int Hq, uint16_t* __restrict__ out,
                                                      float* __restrict__ lse) {
  constexpr int E = D / 32;
  const int64_t row = static_cast<int64_t>(blockIdx.x) * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  const int64_t rows = static_cast<int64_t>(T) * Hq;
  griddep_wait();
  griddep_launch_dependents();
  if (row >= rows) return;
  const float l0 = lane < S ? part_lse[lane * rows + row] : -INFINITY;
  const float l1 = lane + 32 < S ? part_lse[(lane + 32) * rows + row] : -INFINITY;
  float M = fmaxf(l0, l1);
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
  const float w0 = (M == -INFINITY) ? 0.f : fast_exp2(l0 - M);
  const float w1 = (M == -INFINITY) ? 0.f : fast_exp2(l1 - M);
  float acc[E];
#pragma unroll
  for (int e = 0; e < E; ++e) acc[e] = 0.f;
  float wsum = 0.f;
#pragma unroll 8
  for (int s = 0; s < S; ++s) {
    const float w = __shfl_sync(0xffffffffu, s < 32 ? w0 : w1, s & 31);
    wsum += w;
    const float* src = part_o + (s * rows + row) * D + lane * E;
    float v[E];
    if constexpr (E == 4) {
      const float4 x = *reinterpret_cast<const float4*>(src);
      v[0] = x.x; v[1] = x.y; v[2] = x.z; v[3] = x.w;
    } else {
      const float2 x = *reinterpret_cast<const float2*>(src);
      v[0] = x.x; v[1] = x.y;
    }
#pragma unroll
    for (int e = 0; e < E; ++e) acc[e] = fmaf(w, v[e], acc[e]);
  }
  const float inv = wsum > 0.f ? 1.f / wsum : 0.f;
  uint32_t packed[E / 2];
#pragma unroll
  for (int e = 0; e < E / 2; ++e) packed[e] = pack_bf16x2(acc[2 * e] * inv, acc[2 * e + 1] * inv);
  uint16_t* dst = out + row * D + lane * E;
  if constexpr (E == 4) {
    *reinterpret_cast<uint2*>(dst) = make_uint2(packed[0], packed[1]);
  } else {
    *reinterpret_cast<uint32_t*>(dst) = packed[0];
  }
  if (lse != nullptr && lane == 0) lse[row] = (wsum > 0.f) ? (M + log2f(wsum)) * kLn2 : -INFINITY;
}

}  // namespace

int attention_smem_bytes(int d) {
  return d == 64 ? Layout<64>::kAlloc : Layout<128>::kAlloc;
}

cudaError_t launch_attention(const AttnArgs& a, const BatchDesc& b, int d, cudaStream_t st) {
  const int grid = a.n_rb * a.Hkv * a.n_splits;
  if (grid == 0) return cudaSuccess;
  if (d == 64) {
    static bool configured = false;
    if (!configured) {
      cudaError_t e = cudaFuncSetAttribute(attn_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           Layout<64>::kAlloc);
      if (e != cudaSuccess) return e;
      configured = true;
    }
    return launch_kernel(attn_kernel<64>, dim3(grid), dim3(kThreads), Layout<64>::kAlloc, st, 0, a, b);
  } else {
    static bool configured = false;
    if (!configured) {
      cudaError_t e = cudaFuncSetAttribute(attn_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           Layout<128>::kAlloc);
      if (e != cudaSuccess) return e;
      configured = true;
    }
    return launch_kernel(attn_kernel<128>, dim3(grid), dim3(kThreads), Layout<128>::kAlloc, st, 0, a, b);
  }
}

cudaError_t launch_combine(const float* part_o, const float* part_lse, int n_splits, int T, int Hq,
                           int d, uint16_t* out, float* lse, cudaStream_t st) {
  const int64_t rows = static_cast<int64_t>(T) * Hq;
  if (rows == 0) return cudaSuccess;
  const unsigned grid = static_cast<unsigned>((rows + 7) / 8);
  if (d == 64)
    return launch_kernel(combine_kernel<64>, dim3(grid), dim3(256), 0, st, 0, part_o, part_lse, n_splits, T, Hq,
                         out, lse);
  return launch_kernel(combine_kernel<128>, dim3(grid), dim3(256), 0, st, 0, part_o, part_lse, n_splits, T, Hq,
                       out, lse);
}

}  // namespace kvr
