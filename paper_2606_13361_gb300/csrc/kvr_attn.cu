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
// CTA = one or two query tiles (128 packed rows each = 128/G tokens x the G
// query heads of one KV head) x one KV head x one key split.  Two tiles share
// every K/V tile staged in shared memory, which halves the TMA bytes per MMA:
// while the tensor core streams its operands, TMA writes into shared memory
// run at about half their idle rate, and 64 KB of K/V per 128-row tile (per
// 1024 MMA cycles) outpaces them.  Small, split-heavy batches use one tile.
// Warp roles:
//   0-7   softmax, warpgroup x for Q tile x: thread = row = TMEM lane;
//         causal/ownership mask, online softmax in the exp2 domain, P as bf16
//         pairs into TMEM over S, O rescale in TMEM; final normalisation, store
//   8     TMA producer: the Q tiles once, then the K tiles (2-stage ring)
//   9     TMEM owner and MMA issuer: S = Q K^T (128x128 fp32 in TMEM),
//         O += P V (P from TMEM, V from shared memory)
//   10    TMA producer of the V tiles (2-stage ring)
// Key tiles: first the pages shared by every sequence of the batch (a loaded
// prefix forked by many consumers: each such tile is staged once per CTA and
// serves every consumer row in it), then each sequence's own pages; a row sees
// key c iff the tile is shared or its own, and c <= its position.
#include <math.h>

#include "kvr_internal.h"
#include "kvr_ptx.cuh"

namespace kvr {
#ifdef KVR_STAGE_TRACE
KVR_STAGE_BUFFER(g_stage_attn);
#endif
namespace {

constexpr int kStages = 2;  // depth of the K ring and of the V ring
constexpr int kThreads = 32 * 11;
constexpr int kKWarp = 8, kMmaWarp = 9, kVWarp = 10;
constexpr uint32_t kTmemCols = 512;
// TMEM columns: S buffers at 0 and 128, O_x at 256 + 128 x (fp32); the P of
// an S buffer as bf16 pairs over its last 64 columns.
constexpr uint32_t kTmemS = 0, kTmemO = 256, kTmemPOff = 64;
constexpr float kLn2 = 0.69314718055994530942f;

template <int D>
struct Layout {
  static constexpr int kSub = kBlockRows * 64 * 2;      // one 64-column swizzled sub-tile
  static constexpr int kTile = kBlockRows * D * 2;      // 128 rows x D bf16
  static constexpr int kQ = 0;                          // Q tiles A, B
  static constexpr int kK = kQ + kQTiles * kTile;
  static constexpr int kV = kK + kStages * kTile;
  static constexpr int kBar = kV + kStages * kTile;
  static constexpr int kMisc = kBar + 256;
  static constexpr int kMiscInts = 16 + kQTiles * kBlockRows;
  static constexpr int kXch = kMisc + kMiscInts * 4;      // fp32 [6][128]: one-tile key-half exchange
  static constexpr int kEnd = kXch + 6 * kBlockRows * 4;
  // 1 KB of slack to align the dynamic buffer to the 1024-byte swizzle atom;
  // small layouts pad to keep one CTA per SM (each CTA allocates all 512 TMEM columns).
  static constexpr int kAlloc = (kEnd + 1024) > 120 * 1024 ? (kEnd + 1024) : 120 * 1024;
};

enum {
  kBarQ = 0,  // Q tiles landed
  kBarKFull = 1,
  kBarVFull = kBarKFull + kStages,
  kBarKEmpty = kBarVFull + kStages,
  kBarVEmpty = kBarKEmpty + kStages,
  kBarSFull = kBarVEmpty + kStages,  // per S buffer
  kBarPFull = kBarSFull + 2,         // per S buffer
  kBarODone = kBarPFull + 2,         // per O
  kBarDrain = kBarODone + 2,
  kBarPair = kBarDrain + 1,          // one Q tile: key-half exchange per TMEM lane quarter
  kNumBars = kBarPair + 4
};
static_assert(kNumBars * 8 <= 256, "barrier area");
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

// SINGLE: one Q tile per CTA (a.q_tiles == 1), else kQTiles.
template <int D, bool SINGLE>
__global__ void __launch_bounds__(kThreads, 1)
attn_kernel(const __grid_constant__ AttnArgs a, const __grid_constant__ BatchDesc bd) {
  using Lay = Layout<D>;
  static_assert(Lay::kAlloc <= 227 * 1024, "shared memory per CTA");
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + Lay::kBar);
  int* misc = reinterpret_cast<int*>(smem + Lay::kMisc);
  volatile int* abort_flag = misc + kMiscAbort;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // stage slots: 0 entry, 1 grid dependency resolved, 2 Q and the first K tile
  // landed, 3 first P stored, 4 last P stored, 5 waiting for the last P V,
  // 6 output stored, 7 end; 8 + j (20 + j): warpgroup 0 (1) stored P of key
  // tile j < 12
  if (threadIdx.x == 0) KVR_STAGE(g_stage_attn, a.layer, 0);
  const int G = a.G, TB = kBlockRows / G;
  // (the two-tile instantiation keeps the one-tile paths reachable: with
  // them folded away its register allocation spills)
  const bool single = SINGLE || a.q_tiles == 1;
  int bid = blockIdx.x;
  const int split = bid % a.n_splits;
  bid /= a.n_splits;
  const int g = bid % a.Hkv;
  bid /= a.Hkv;
  const int n_groups = (a.n_rb + a.q_tiles - 1) / a.q_tiles;
  const int pr = n_groups - 1 - bid;  // late (longest) query blocks first
  const int tok0 = pr * a.q_tiles * TB;
  const int tok1 = min(bd.T, tok0 + a.q_tiles * TB);
  const bool has_b = !single && tok0 + TB < bd.T;  // Q tile B holds at least one token

  if (threadIdx.x == 0) {
    mbar_init(&bars[kBarQ], 1);
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&bars[kBarKFull + s], 1);
      mbar_init(&bars[kBarKEmpty + s], 1);
      mbar_init(&bars[kBarVFull + s], 1);
      mbar_init(&bars[kBarVEmpty + s], 1);
    }
    for (int x = 0; x < 2; ++x) {
      mbar_init(&bars[kBarSFull + x], 1);
      mbar_init(&bars[kBarPFull + x], single ? 256 : 128);  // one Q tile: both warpgroups
      mbar_init(&bars[kBarODone + x], 1);
    }
    mbar_init(&bars[kBarDrain], 1);
    for (int qq = 0; qq < 4; ++qq) mbar_init(&bars[kBarPair + qq], 64);
    fence_barrier_init();
    misc[kMiscAbort] = 0;
    // Key-tile plan of the CTA's query rows and this split's share of it.
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
  if (warp == kMmaWarp) {
    tmem_alloc(reinterpret_cast<uint32_t*>(misc + kMiscTmem), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  griddep_wait();  // global memory from here on
  griddep_launch_dependents();
  if (threadIdx.x == 0) KVR_STAGE(g_stage_attn, a.layer, 1);

  const uint32_t tmem = static_cast<uint32_t>(misc[kMiscTmem]);
  const int b_lo = misc[kMiscBLo], b_hi = misc[kMiscBHi];
  const int t_begin = misc[kMiscBegin];
  const int n = misc[kMiscEnd] - t_begin;
  const int* ntile = misc + kMiscNTile;

  if (warp == kKWarp || warp == kVWarp) {
    // ----------------------------------------------------------- producers --
    // One warp streams the Q tiles and the K tiles, another the V tiles, so a
    // K load never queues behind a V slot that a P V still holds.  The issuing
    // thread stalls while the TMA unit takes each copy, so its loop carries no
    // memory latency: the 32 lanes look up the pages of the next 32 tiles (one
    // page-table load each) while lane 0 issues the current 32.
    const int kind = warp == kKWarp ? 0 : 1;
    auto lookup_page = [&](int chunk) -> int {  // page of tile chunk*32 + lane, -2 past the end
      const int ti = chunk * 32 + lane;
      if (ti >= n) return -2;
      TileCursor lc;
      lc.init(t_begin + ti, b_lo, b_hi, bd.shared_pages, ntile);
      int slot;
      const int pidx = lc.page_slot_index(bd, &slot);
      return (pidx >= 0 && pidx < bd.max_pages) ? bd.page_table[slot * bd.max_pages + pidx] : -1;
    };
    auto page_row = [&](int page) -> int {  // first pool row of this kind's tile; bad pages read row 0
      if (page == -2) return 0;
      const int64_t r = kv_row(page, a.layer, kind, g, a.layers, a.Hkv);
      if (page < 0 || r < 0 || r + kPageTokens > a.n_pool_rows) {
        atomicOr(a.err, kDevErrBounds);
        return 0;
      }
      return static_cast<int>(r);
    };
    if (n > 0) {
      uint64_t* full = &bars[kind ? kBarVFull : kBarKFull];
      uint64_t* empty = &bars[kind ? kBarVEmpty : kBarKEmpty];
      uint8_t* ring = smem + (kind ? Lay::kV : Lay::kK);
      int page_next = lookup_page(0);
      if (lane == 0) {
        tma_prefetch_desc(&a.tm_kv);
        if (kind == 0) {
          tma_prefetch_desc(&a.tm_q);
          const int nq = has_b ? 2 : 1;
          mbar_arrive_expect_tx(&bars[kBarQ], nq * Lay::kTile);
          for (int x = 0; x < nq; ++x)
#pragma unroll
            for (int c = 0; c < D / 64; ++c)
              tma_load_3d(smem + Lay::kQ + x * Lay::kTile + c * Lay::kSub, &a.tm_q, &bars[kBarQ], c * 64,
                          g * G, tok0 + x * TB);
        }
      }
      bool ok = true;
      int issued = 0, st = 0;
      uint32_t phase = 0;  // parity of the current pass over the ring
      for (int c0 = 0; c0 < n && ok; c0 += 32) {
        const int row_cur = page_row(page_next);
        if (c0 + 32 < n) page_next = lookup_page(c0 / 32 + 1);
        const int cnt = min(32, n - c0);
        for (int i = 0; i < cnt; ++i) {
          const int row = __shfl_sync(0xffffffffu, row_cur, i);
          const int j = c0 + i;
          if (lane == 0) {
            if (j >= kStages) ok = mbar_wait(&empty[st], phase ^ 1u, abort_flag, a.err);
            if (ok) {
              mbar_arrive_expect_tx(&full[st], Lay::kTile);
#pragma unroll
              for (int c = 0; c < D / 64; ++c)
                tma_load_2d(ring + st * Lay::kTile + c * Lay::kSub, &a.tm_kv, &full[st], c * 64, row);
              issued = j + 1;
              if (++st == kStages) {
                st = 0;
                phase ^= 1u;
              }
            }
          }
          ok = __shfl_sync(0xffffffffu, ok, 0);
          if (!ok) break;
        }
      }
      if (!ok && lane == 0) {
        // Unwinding: let the copies already in flight land before the CTA exits.
        volatile int no_abort = 0;
        if (kind == 0) mbar_wait(&bars[kBarQ], 0, &no_abort, a.err);
        for (int j = max(0, issued - kStages); j < issued; ++j)
          mbar_wait(&full[j % kStages], (j / kStages) & 1, &no_abort, a.err);
      }
    }
  } else if (warp == kMmaWarp) {
    // ---------------------------------------------------------------- MMA --
    // The tensor pipe runs one issuer's MMAs in order.  Two Q tiles (x = A, B,
    // S buffer x, O_x): per key tile j the stream is P_A V_j, S_A = Q_A K_{j+1}^T,
    // P_B V_j, S_B(j+1), so S_x(j+1) completing also means P_x V_j has
    // completed: the softmax of tile j+1 may then rescale O_x and overwrite
    // P_x.  One Q tile: S alternates between both buffers, S(j+2) follows P V_j
    // into buffer j&1; every P V commits its own O-done phase, and the P-full
    // barrier of a buffer has one phase per use of that buffer (the softmax
    // may finish tile j+1 before P V_j is issued).
    if (lane == 0 && n > 0) {
      constexpr uint32_t kIdS = make_idesc_bf16(128, kPageTokens, 0);
      constexpr uint32_t kIdO = make_idesc_bf16(128, D, 1);
      const uint32_t sQ = smem_u32(smem + Lay::kQ);
      const uint32_t sK = smem_u32(smem + Lay::kK);
      const uint32_t sV = smem_u32(smem + Lay::kV);
      // S buffer `buf` = Q_qx K_j^T
      auto issue_s = [&](int qx, int buf, int j) {
        const int st = j % kStages;
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint32_t off = (kk >> 2) * Lay::kSub + (kk & 3) * 32;
          const uint64_t ad = make_sdesc_sw128(sQ + qx * Lay::kTile + off, 16, 1024);
          const uint64_t bd2 = make_sdesc_sw128(sK + st * Lay::kTile + off, 16, 1024);
          umma_bf16_ss(tmem + kTmemS + buf * 128, ad, bd2, kIdS, kk > 0 ? 1u : 0u);
        }
        umma_commit(&bars[kBarSFull + buf]);
      };
      // O_ox += P (over S buffer `buf`) V_j once that P is complete
      auto issue_pv = [&](int buf, int ox, int j) -> bool {
        const uint32_t par = single ? ((j >> 1) & 1) : (j & 1);
        if (!mbar_wait(&bars[kBarPFull + buf], par, abort_flag, a.err)) return false;
        if (!single && j == 4 && ox == 0) KVR_STAGE(g_stage_attn, a.layer, 29);
        tc_fence_after();
        const int st = j % kStages;
#pragma unroll
        for (int kk = 0; kk < kPageTokens / 16; ++kk) {
          const uint64_t bd2 = make_sdesc_sw128(sV + st * Lay::kTile + kk * 2048, Lay::kSub, 1024);
          umma_bf16_ts(tmem + kTmemO + ox * 128, tmem + kTmemS + buf * 128 + kTmemPOff + kk * 8, bd2, kIdO,
                       (j > 0 || kk > 0) ? 1u : 0u);
        }
        if (single || j == n - 1) umma_commit(&bars[kBarODone + ox]);
        return true;
      };
      auto wait_k = [&](int j) {
        return mbar_wait(&bars[kBarKFull + j % kStages], (j / kStages) & 1, abort_flag, a.err);
      };
      auto wait_v = [&](int j) {
        return mbar_wait(&bars[kBarVFull + j % kStages], (j / kStages) & 1, abort_flag, a.err);
      };
      bool issued_any = false;
      bool ok = mbar_wait(&bars[kBarQ], 0, abort_flag, a.err) && wait_k(0);
      KVR_STAGE(g_stage_attn, a.layer, 2);
      if (single) {
        if (ok) {
          tc_fence_after();
          issue_s(0, 0, 0);
          umma_commit(&bars[kBarKEmpty]);
          issued_any = true;
        }
        if (ok && n > 1 && (ok = wait_k(1))) {
          tc_fence_after();
          issue_s(0, 1, 1);
          umma_commit(&bars[kBarKEmpty + 1 % kStages]);
        }
        for (int j = 0; j < n && ok; ++j) {
          if (!(ok = wait_v(j) && issue_pv(j & 1, 0, j))) break;
          umma_commit(&bars[kBarVEmpty + j % kStages]);
          if (j + 2 < n) {
            if (!(ok = wait_k(j + 2))) break;
            tc_fence_after();
            issue_s(0, j & 1, j + 2);
            umma_commit(&bars[kBarKEmpty + (j + 2) % kStages]);
          }
        }
      } else {
        const int nq = has_b ? 2 : 1;
        if (ok) {
          tc_fence_after();
          for (int x = 0; x < nq; ++x) issue_s(x, x, 0);
          umma_commit(&bars[kBarKEmpty]);
          issued_any = true;
        }
        for (int j = 0; j < n && ok; ++j) {
          const bool more = j + 1 < n;
          // P V_j waits only for V_j (and its P); K_{j+1} is waited for just
          // before the first S of tile j+1, so a late K tile delays no P V
          if (!(ok = wait_v(j))) break;
          if (j == 4) KVR_STAGE(g_stage_attn, a.layer, 28);
          bool k_ready = !more;
          for (int x = 0; x < nq && ok; ++x) {
            ok = issue_pv(x, x, j);
            if (j == 4 && x == 0) KVR_STAGE(g_stage_attn, a.layer, 30);
            if (ok && more) {
              if (!k_ready) ok = k_ready = wait_k(j + 1);
              if (ok) issue_s(x, x, j + 1);
            }
          }
          if (!ok) break;
          umma_commit(&bars[kBarVEmpty + j % kStages]);
          if (more) umma_commit(&bars[kBarKEmpty + (j + 1) % kStages]);
        }
      }
      if (!ok && issued_any) {
        // Unwinding: wait for the MMAs in flight before TMEM is released.
        volatile int no_abort = 0;
        umma_commit(&bars[kBarDrain]);
        mbar_wait(&bars[kBarDrain], 0, &no_abort, a.err);
      }
    }
  } else if (warp < kKWarp) {
    if constexpr (SINGLE) {
      // ------------------------------------------------------------ softmax --
      // Warp w serves TMEM lane quarter w % 4 (rows 32*(w%4) + lane; a warp
      // reaches only its own quarter of TMEM lanes).  Two Q tiles: warpgroup
      // x = w / 4 owns Q tile x.  One Q tile: both warpgroups serve its rows and
      // warpgroup x takes keys 64x .. 64x + 63 of every key tile (the two halves
      // of a row meet through shared memory for the row maximum and the final
      // row sum; O columns 64x .. 64x + 63 are warpgroup x's to rescale and
      // store), which halves the per-tile chain of a row.
      const int x = warp >> 2;
      const int quarter = warp & 3;
      const int r = quarter * 32 + lane;
      const int xt = single ? 0 : x;  // Q tile of this warpgroup
      const uint32_t lane_addr = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
      const uint32_t o_addr = lane_addr + kTmemO + xt * 128;
      const int nx = (x == 0 || has_b || single) ? n : 0;  // tiles this warpgroup walks
      const int t = tok0 + xt * TB + r / G;
      const int h = g * G + r % G;
      const bool valid = t < tok1;
      // one Q tile: per-row maxima of each key half ([tile parity][half][row]),
      // then the halves' row sums ([half][row])
      float* xm = reinterpret_cast<float*>(smem + Lay::kXch);
      // warps quarter and quarter + 4 meet on an mbarrier of 64 arrivals (a
      // bounded wait: a partner that gave up cannot hang this warp)
      uint32_t pair_uses = 0;
      auto pair_sync = [&]() -> bool {
        mbar_arrive(&bars[kBarPair + quarter]);
        return mbar_wait(&bars[kBarPair + quarter], (pair_uses++) & 1, abort_flag, a.err);
      };
      // O columns this warpgroup rescales and stores
      const int oc0 = single ? x * (D / 2) : 0, ocn = single ? D / 2 : D;
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
      for (int j = 0; j < nx; ++j, cur.next()) {
        const int sb = single ? (j & 1) : x;  // S buffer of this tile
        const uint32_t sp = single ? ((j >> 1) & 1) : (j & 1);
        ok = __all_sync(0xffffffffu, ok && mbar_wait(&bars[kBarSFull + sb], sp, abort_flag, a.err));
        if (!ok) break;
        tc_fence_after();
        const uint32_t s_addr = lane_addr + kTmemS + sb * 128;
        // Scores in 64-key halves (never all 128 live).  Two Q tiles: the row
        // maximum needs both halves; the second half stays in registers and its
        // P goes over its own columns, then the first half is read again for its
        // P.  One Q tile: this warpgroup's half only.
        const int owner = cur.owner();
        int nvis = 0;
        if (owner == -1 || owner == my_b) nvis = min(max(pos - cur.key_base() + 1, 0), kPageTokens);
        const bool masked = __any_sync(0xffffffffu, nvis < kPageTokens);
        float hs[64];
        auto load_half = [&](int half) {
          tmem_ld64(s_addr + half * 64, hs);
          if (masked) {
  #pragma unroll
            for (int k = 0; k < 64; ++k) hs[k] = (half * 64 + k < nvis) ? hs[k] : -INFINITY;
          }
        };
        auto half_max = [&]() {  // 8 independent chains of three-input maxima
          float mx[8];
  #pragma unroll
          for (int i = 0; i < 8; ++i) {
            mx[i] = fmax3(hs[i], hs[8 + i], hs[16 + i]);
            mx[i] = fmax3(mx[i], hs[24 + i], hs[32 + i]);
            mx[i] = fmax3(mx[i], hs[40 + i], hs[48 + i]);
            mx[i] = fmaxf(mx[i], hs[56 + i]);
          }
          return fmax3(fmax3(mx[0], mx[1], mx[2]), fmax3(mx[3], mx[4], mx[5]), fmaxf(mx[6], mx[7]));
        };
        float tmax;
        if (single) {
          load_half(x);
          const float hm = half_max();
          // both halves are read (and in registers) before either warpgroup
          // overwrites columns 64..127 with P below
          float* xb = xm + (j & 1) * 2 * kBlockRows;
          xb[x * kBlockRows + r] = hm;
          if (!__all_sync(0xffffffffu, pair_sync())) {
            ok = false;
            break;
          }
          tmax = fmaxf(xb[r], xb[kBlockRows + r]);
        } else {
          load_half(0);
          const float max0 = half_max();
          load_half(1);
          tmax = fmaxf(max0, half_max());
        }
        float alpha = 1.f;
        if (tmax != -INFINITY && (m == -INFINITY || (tmax - m) * c > kLazy)) {
          alpha = fast_exp2((m - tmax) * c);  // 0 when nothing was accumulated yet
          m = tmax;
        }
        const float mc = (m == -INFINITY) ? 0.f : m * c;
        // exponentials (packed argument), row sum over 4 packed chains; P as
        // bf16 pairs (key 2i in the low half of column i) over columns 64..127
        float2 acc[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f),
                         make_float2(0.f, 0.f)};
        // One Q tile: the softmax may start tile j before P V_{j-1} has finished
        // (S(j) was computed ahead), and a tcgen05.st into the tile's TMEM while
        // that P V runs gave nondeterministic results on this GPU although the
        // columns differ, so the P stores and the O rescale wait for its O-done
        // phase.  Two Q tiles: S_x(j) completing already implies it.
        bool pv_done = true;
        auto exp_half = [&](int half, bool wait_pv) {
          uint32_t pw[32];
  #pragma unroll
          for (int k = 0; k < 64; k += 2) {
            const float2 xx = ffma2(make_float2(hs[k], hs[k + 1]), make_float2(c, c), make_float2(-mc, -mc));
            const float e0 = fast_exp2(xx.x), e1 = fast_exp2(xx.y);
            acc[(k >> 1) & 3] = fadd2(acc[(k >> 1) & 3], make_float2(e0, e1));
            pw[k >> 1] = pack_bf16x2(e0, e1);
          }
          if (wait_pv) {
            pv_done = __all_sync(0xffffffffu, mbar_wait(&bars[kBarODone], (j - 1) & 1, abort_flag, a.err));
            if (!pv_done) return;
            tc_fence_after();
          }
          tmem_st32_u32(s_addr + kTmemPOff + half * 32, pw);
        };
        if (single) {
          exp_half(x, j > 0);  // keys 64x.. -> columns 64 + 32x ..
        } else {
          exp_half(1, false);  // keys 64..127 -> columns 96..127 (their own scores, already read)
          load_half(0);
          exp_half(0, false);  // keys 0..63 -> columns 64..95 (keys 64..95's scores, already read)
        }
        if (!pv_done) {  // a failed wait skips this tile's P; the next tile's wait ends the loop
          ok = false;
          continue;
        }
        const float2 a01 = fadd2(acc[0], acc[1]), a23 = fadd2(acc[2], acc[3]);
        const float2 a03 = fadd2(a01, a23);
        l = l * alpha + (a03.x + a03.y);
        // O rescale (P V_{j-1} is complete: see above)
        if (j > 0 && __any_sync(0xffffffffu, alpha != 1.f)) {
  #pragma unroll 1
          for (int q = oc0 / 32; q < (oc0 + ocn) / 32; ++q) {
            float o[32];
            tmem_ld32(o_addr + q * 32, o);
  #pragma unroll
            for (int i = 0; i < 32; ++i) o[i] *= alpha;
            tmem_st32(o_addr + q * 32, o);
          }
        }
        tc_fence_before();
        mbar_arrive(&bars[kBarPFull + sb]);
        if (threadIdx.x == 0) {
          if (j == 0) KVR_STAGE(g_stage_attn, a.layer, 3);
          KVR_STAGE(g_stage_attn, a.layer, 4);
        }
        if ((threadIdx.x & 127) == 0 && j < 10) KVR_STAGE(g_stage_attn, a.layer, 8 + 10 * (threadIdx.x >> 7) + j);
      }
      if (threadIdx.x == 0) KVR_STAGE(g_stage_attn, a.layer, 5);
      if (ok && nx > 0)
        ok = __all_sync(0xffffffffu, mbar_wait(&bars[kBarODone + xt], single ? (nx - 1) & 1 : 0, abort_flag, a.err));
      if (threadIdx.x == 0) KVR_STAGE(g_stage_attn, a.layer, 28);
      if (single) {  // the row sum over both key halves, in half order
        float* xl = xm + 4 * kBlockRows;
        xl[x * kBlockRows + r] = l;
        ok = __all_sync(0xffffffffu, pair_sync()) && ok;
        l = xl[r] + xl[kBlockRows + r];
      }
      if (threadIdx.x == 0) KVR_STAGE(g_stage_attn, a.layer, 29);
      if (ok) {
        tc_fence_after();
        const float inv_l = (l > 0.f) ? 1.f / l : 0.f;
        const float lse2 = (l > 0.f) ? (m * c + log2f(l)) : -INFINITY;
        const int64_t row = static_cast<int64_t>(t) * a.Hq + h;
        const bool lse_writer = !single || x == 0;
        if (a.n_splits == 1) {
  #pragma unroll 1
          for (int q = oc0 / 32; q < (oc0 + ocn) / 32; ++q) {
            float o[32];
            if (nx > 0) tmem_ld32(o_addr + q * 32, o);
  #pragma unroll
            for (int i = 0; i < 32; ++i) o[i] = (nx > 0) ? o[i] * inv_l : 0.f;
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
          if (valid && lse_writer && a.lse != nullptr) a.lse[row] = lse2 * kLn2;
        } else {
          // The warp's 32 rows x this warpgroup's columns go through shared
          // memory (the K/V rings are free: the last P V has completed) so that
          // the stores of the partial are whole row segments: a row per lane
          // would make every store instruction touch 32 separate rows.
          constexpr int kHalf = D / 2, kPitch = kHalf + 4;  // padded rows: conflict-free 16-byte accesses
          float* stg = reinterpret_cast<float*>(smem + Lay::kK) + warp * 32 * kPitch;
          if constexpr (kHalf == 64) {  // this warpgroup's 64 columns in one TMEM load
            float o[64];
            if (nx > 0) tmem_ld64(o_addr + oc0, o);
  #pragma unroll
            for (int v4 = 0; v4 < 16; ++v4)
              *reinterpret_cast<float4*>(stg + lane * kPitch + 4 * v4) =
                  (nx > 0) ? make_float4(o[4 * v4] * inv_l, o[4 * v4 + 1] * inv_l, o[4 * v4 + 2] * inv_l,
                                         o[4 * v4 + 3] * inv_l)
                           : make_float4(0.f, 0.f, 0.f, 0.f);
          } else {
  #pragma unroll 1
            for (int q = oc0 / 32; q < (oc0 + ocn) / 32; ++q) {
              float o[32];
              if (nx > 0) tmem_ld32(o_addr + q * 32, o);
  #pragma unroll
              for (int v4 = 0; v4 < 8; ++v4)
                *reinterpret_cast<float4*>(stg + lane * kPitch + (q * 32 - oc0) + 4 * v4) =
                    (nx > 0) ? make_float4(o[4 * v4] * inv_l, o[4 * v4 + 1] * inv_l, o[4 * v4 + 2] * inv_l,
                                           o[4 * v4 + 3] * inv_l)
                             : make_float4(0.f, 0.f, 0.f, 0.f);
            }
          }
          __syncwarp();
          if (threadIdx.x == 0) KVR_STAGE(g_stage_attn, a.layer, 30);
          constexpr int kRowsPer = 32 / (kHalf / 4);  // rows stored per instruction
          const int sub = lane / (kHalf / 4), c4 = lane % (kHalf / 4);
  #pragma unroll 4
          for (int rr = sub; rr < 32; rr += kRowsPer) {
            const int r2 = quarter * 32 + rr;
            const int t2 = tok0 + r2 / G, h2 = g * G + r2 % G;
            if (t2 < tok1) {
              const int64_t prow2 = static_cast<int64_t>(split) * bd.T * a.Hq + static_cast<int64_t>(t2) * a.Hq + h2;
              *reinterpret_cast<float4*>(a.part_o + prow2 * D + oc0 + 4 * c4) =
                  *reinterpret_cast<const float4*>(stg + rr * kPitch + 4 * c4);
            }
          }
          if (valid && lse_writer) a.part_lse[static_cast<int64_t>(split) * bd.T * a.Hq + row] = lse2;
        }
      }
    } else {
      // ------------------------------------------------------------ softmax --
      // Warpgroup x = w / 4 owns Q tile x; warp w serves TMEM lane quarter w % 4
      // (rows 32*(w%4) + lane; a warp reaches only its own quarter of TMEM lanes).
      const int x = warp >> 2;
      const int quarter = warp & 3;
      const int r = quarter * 32 + lane;
      const uint32_t lane_addr = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
      const uint32_t o_addr = lane_addr + kTmemO + x * 128;
      const int nx = (x == 0 || has_b) ? n : 0;  // tiles this warpgroup walks
      const int t = tok0 + x * TB + r / G;
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
      for (int j = 0; j < nx; ++j, cur.next()) {
        const int sb = single ? (j & 1) : x;  // S buffer of this tile
        const uint32_t sp = single ? ((j >> 1) & 1) : (j & 1);
        ok = __all_sync(0xffffffffu, ok && mbar_wait(&bars[kBarSFull + sb], sp, abort_flag, a.err));
        if (!ok) break;
        tc_fence_after();
        if (threadIdx.x == 0 && j == 5) KVR_STAGE(g_stage_attn, a.layer, 31);
        const uint32_t s_addr = lane_addr + kTmemS + sb * 128;
        // Scores in two 64-key halves (never all 128 live): the row maximum
        // needs both; the second half stays in registers and its P goes over its
        // own columns, then the first half is read again for its P.
        const int owner = cur.owner();
        int nvis = 0;
        if (owner == -1 || owner == my_b) nvis = min(max(pos - cur.key_base() + 1, 0), kPageTokens);
        const bool masked = __any_sync(0xffffffffu, nvis < kPageTokens);
        float hs[64];
        auto load_half = [&](int half) {
          tmem_ld64(s_addr + half * 64, hs);
          if (masked) {
  #pragma unroll
            for (int k = 0; k < 64; ++k) hs[k] = (half * 64 + k < nvis) ? hs[k] : -INFINITY;
          }
        };
        auto half_max = [&]() {  // 8 independent chains of three-input maxima
          float mx[8];
  #pragma unroll
          for (int i = 0; i < 8; ++i) {
            mx[i] = fmax3(hs[i], hs[8 + i], hs[16 + i]);
            mx[i] = fmax3(mx[i], hs[24 + i], hs[32 + i]);
            mx[i] = fmax3(mx[i], hs[40 + i], hs[48 + i]);
            mx[i] = fmaxf(mx[i], hs[56 + i]);
          }
          return fmax3(fmax3(mx[0], mx[1], mx[2]), fmax3(mx[3], mx[4], mx[5]), fmaxf(mx[6], mx[7]));
        };
        load_half(0);
        const float max0 = half_max();
        load_half(1);
        const float tmax = fmaxf(max0, half_max());
        float alpha = 1.f;
        if (tmax != -INFINITY && (m == -INFINITY || (tmax - m) * c > kLazy)) {
          alpha = fast_exp2((m - tmax) * c);  // 0 when nothing was accumulated yet
          m = tmax;
        }
        const float mc = (m == -INFINITY) ? 0.f : m * c;
        // exponentials (packed argument), row sum over 4 packed chains; P as
        // bf16 pairs (key 2i in the low half of column i) over columns 64..127
        float2 acc[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f),
                         make_float2(0.f, 0.f)};
        // One Q tile: the softmax may start tile j before P V_{j-1} has finished
        // (S(j) was computed ahead), and a tcgen05.st into the tile's TMEM while
        // that P V runs gave nondeterministic results on this GPU although the
        // columns differ, so the P stores and the O rescale wait for its O-done
        // phase.  Two Q tiles: S_x(j) completing already implies it.
        bool pv_done = true;
        auto exp_half = [&](int half, bool wait_pv) {
          uint32_t pw[32];
  #pragma unroll
          for (int k = 0; k < 64; k += 2) {
            const float2 xx = ffma2(make_float2(hs[k], hs[k + 1]), make_float2(c, c), make_float2(-mc, -mc));
            const float e0 = fast_exp2(xx.x), e1 = fast_exp2(xx.y);
            acc[(k >> 1) & 3] = fadd2(acc[(k >> 1) & 3], make_float2(e0, e1));
            pw[k >> 1] = pack_bf16x2(e0, e1);
          }
          if (wait_pv) {
            pv_done = __all_sync(0xffffffffu, mbar_wait(&bars[kBarODone], (j - 1) & 1, abort_flag, a.err));
            if (!pv_done) return;
            tc_fence_after();
          }
          tmem_st32_u32(s_addr + kTmemPOff + half * 32, pw);
        };
        exp_half(1, single && j > 0);  // keys 64..127 -> columns 96..127 (their own scores, already read)
        if (!pv_done) {  // a failed wait skips this tile's P; the next tile's wait ends the loop
          ok = false;
          continue;
        }
        load_half(0);
        exp_half(0, false);  // keys 0..63 -> columns 64..95 (keys 64..95's scores, already read)
        const float2 a01 = fadd2(acc[0], acc[1]), a23 = fadd2(acc[2], acc[3]);
        const float2 a03 = fadd2(a01, a23);
        l = l * alpha + (a03.x + a03.y);
        // O rescale (P V_{j-1} is complete: see above)
        if (j > 0 && __any_sync(0xffffffffu, alpha != 1.f)) {
  #pragma unroll 1
          for (int q = 0; q < D / 32; ++q) {
            float o[32];
            tmem_ld32(o_addr + q * 32, o);
  #pragma unroll
            for (int i = 0; i < 32; ++i) o[i] *= alpha;
            tmem_st32(o_addr + q * 32, o);
          }
        }
        tc_fence_before();
        mbar_arrive(&bars[kBarPFull + sb]);
        if (threadIdx.x == 0) {
          if (j == 0) KVR_STAGE(g_stage_attn, a.layer, 3);
          KVR_STAGE(g_stage_attn, a.layer, 4);
        }
        if ((threadIdx.x & 127) == 0 && j < 10 && (threadIdx.x >> 7) == 0) KVR_STAGE(g_stage_attn, a.layer, 8 + j);
        if (lane == 0 && warp < 4 && j == 4) KVR_STAGE(g_stage_attn, a.layer, 24 + warp);
      }
      if (threadIdx.x == 0) KVR_STAGE(g_stage_attn, a.layer, 5);
      if (ok && nx > 0)
        ok = __all_sync(0xffffffffu, mbar_wait(&bars[kBarODone + x], single ? (nx - 1) & 1 : 0, abort_flag, a.err));
      if (ok) {
        tc_fence_after();
        const float inv_l = (l > 0.f) ? 1.f / l : 0.f;
        const float lse2 = (l > 0.f) ? (m * c + log2f(l)) : -INFINITY;
        const int64_t row = static_cast<int64_t>(t) * a.Hq + h;
        if (a.n_splits == 1) {
  #pragma unroll 1
          for (int q = 0; q < D / 32; ++q) {
            float o[32];
            if (nx > 0) tmem_ld32(o_addr + q * 32, o);
  #pragma unroll
            for (int i = 0; i < 32; ++i) o[i] = (nx > 0) ? o[i] * inv_l : 0.f;
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
            if (nx > 0) tmem_ld32(o_addr + q * 32, o);
            if (valid) {
              float4* dst = reinterpret_cast<float4*>(a.part_o + prow * D + q * 32);
  #pragma unroll
              for (int v4 = 0; v4 < 8; ++v4)
                dst[v4] = (nx > 0) ? make_float4(o[4 * v4] * inv_l, o[4 * v4 + 1] * inv_l,
                                                 o[4 * v4 + 2] * inv_l, o[4 * v4 + 3] * inv_l)
                                   : make_float4(0.f, 0.f, 0.f, 0.f);
            }
          }
          if (valid) a.part_lse[prow] = lse2;
        }
      }
  
    }
  }

  if (threadIdx.x == 0) KVR_STAGE(g_stage_attn, a.layer, 6);
  tc_fence_before();
  __syncthreads();
  if (warp == kMmaWarp) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
  if (threadIdx.x == 0) KVR_STAGE(g_stage_attn, a.layer, 7);
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
  // up to kPre splits: every O vector of the row is loaded together with the
  // lse values (one round trip to L2 instead of two)
  constexpr int kPre = 16;
  float pre[kPre][E];
  if (S <= kPre) {
#pragma unroll
    for (int s = 0; s < kPre; ++s) {
      const float* src = part_o + (s * rows + row) * D + lane * E;
      if constexpr (E == 4) {
        const float4 x = s < S ? *reinterpret_cast<const float4*>(src) : make_float4(0.f, 0.f, 0.f, 0.f);
        pre[s][0] = x.x; pre[s][1] = x.y; pre[s][2] = x.z; pre[s][3] = x.w;
      } else {
        const float2 x = s < S ? *reinterpret_cast<const float2*>(src) : make_float2(0.f, 0.f);
        pre[s][0] = x.x; pre[s][1] = x.y;
      }
    }
  }
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
  if (S <= kPre) {
#pragma unroll
    for (int s = 0; s < kPre; ++s) {
      if (s < S) {
        const float w = __shfl_sync(0xffffffffu, w0, s);
        wsum += w;
#pragma unroll
        for (int e = 0; e < E; ++e) acc[e] = fmaf(w, pre[s][e], acc[e]);
      }
    }
  }
#pragma unroll 8
  for (int s = S <= kPre ? S : 0; s < S; ++s) {
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

template <int D, bool SINGLE>
cudaError_t launch_attention_d(const AttnArgs& a, const BatchDesc& b, int grid, cudaStream_t st) {
  static PerDeviceOnce setup;
  const cudaError_t e = setup.run([] {
    return cudaFuncSetAttribute(attn_kernel<D, SINGLE>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                Layout<D>::kAlloc);
  });
  if (e != cudaSuccess) return e;
  return launch_kernel(attn_kernel<D, SINGLE>, dim3(grid), dim3(kThreads), Layout<D>::kAlloc, st, 0, a, b);
}

cudaError_t launch_attention(const AttnArgs& a, const BatchDesc& b, int d, cudaStream_t st) {
  if (a.q_tiles != 1 && a.q_tiles != kQTiles) return cudaErrorInvalidValue;
  const int grid = (a.n_rb + a.q_tiles - 1) / a.q_tiles * a.Hkv * a.n_splits;
  if (grid == 0) return cudaSuccess;
  if (d == 64)
    return a.q_tiles == 1 ? launch_attention_d<64, true>(a, b, grid, st) : launch_attention_d<64, false>(a, b, grid, st);
  return a.q_tiles == 1 ? launch_attention_d<128, true>(a, b, grid, st) : launch_attention_d<128, false>(a, b, grid, st);
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

#ifdef KVR_STAGE_TRACE
extern "C" __attribute__((visibility("default"))) int kvr_stage_read_attn(void* host, int bytes) {
  return static_cast<int>(cudaMemcpyFromSymbol(host, kvr::g_stage_attn, static_cast<size_t>(bytes)));
}
#endif
