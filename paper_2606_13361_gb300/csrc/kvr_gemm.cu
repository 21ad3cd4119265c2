// kvr_gemm.cu -- the projections of the whole decoder layer (the paper times
// whole-model forwards, Sec. 5 Table 1): D[T][N] = X[T][K] W[N][K]^T (+ C) in
// bf16 with fp32 accumulation, on tcgen05 tensor cores.
//
// Persistent kernel, one CTA per SM, 128 x BN output tiles (BN = 256, or 128
// for short batches so that more SMs share the weight stream).  Warp roles:
//   0     TMA producer: the X tile (128 rows x 64 K) and the W tile (BN rows x
//         64 K) of each K step into a 4- or 6-stage ring, 128-byte swizzle
//   1     TMEM owner and MMA issuer: tcgen05.mma M128 N=BN K16 per 16 of K,
//         accumulating in TMEM; two accumulators, so the epilogue of one tile
//         overlaps the main loop of the next
//   2-5   epilogue: warp w reads TMEM lanes 32 (w % 4) .. + 31 (one output
//         row per thread), adds the residual, rounds once to bf16, stores
// Operands are both K-major (X rows and W rows are contiguous in K), so no
// operand is transposed anywhere.  Up to three weight matrices that share the
// input (the q, k and v projections) run as one launch over their
// concatenated output columns.  The SwiGLU variant loads, per tile, BN/2
// gate rows and the matching BN/2 up rows of W = [W_gate; W_up] and writes
// silu(g) * u (g and u rounded to bf16 first: the arithmetic of the separate
// SwiGLU pass), so the gate/up activations never reach HBM.
#include "kvr_internal.h"
#include "kvr_ptx.cuh"

namespace kvr {
namespace {

constexpr int kBM = 128, kBK = 64;
constexpr int kThreads = 6 * 32;  // producer, MMA, four epilogue warps

template <int BN>
struct GemmLayout {
  static constexpr int kStages = BN == 256 ? 4 : 6;
  static constexpr int kA = kBM * kBK * 2;   // 16 KB
  static constexpr int kB = BN * kBK * 2;    // 32 KB (BN = 256) or 16 KB
  static constexpr int kStage = kA + kB;
  static constexpr int kBar = kStages * kStage;
  static constexpr int kMisc = kBar + 256;
  static constexpr int kEnd = kMisc + 64;
  static constexpr int kAlloc = kEnd + 1024;  // 1 KB to align to the swizzle atom
  static constexpr uint32_t kTmemCols = 2 * BN;
};

enum { kBarFull = 0, kBarEmpty = 8, kBarAccFull = 16, kBarAccEmpty = 18, kBarDrain = 20, kNumBars = 21 };
static_assert(kNumBars * 8 <= 256, "barrier area");

struct TileMap {
  int m_tiles, n_tiles;
  int nseg;
  int seg_tiles[kMaxGemmSegs];  // output tiles of each segment along N
  __device__ void locate(int t, int* m0, int* seg, int* nt) const {
    *m0 = (t % m_tiles) * kBM;
    int nb = t / m_tiles, s = 0;
    while (s < nseg - 1 && nb >= seg_tiles[s]) nb -= seg_tiles[s++];
    *seg = s;
    *nt = nb;
  }
};

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }
__device__ __forceinline__ float bf16_round(float x) { return bf16_lo(pack_bf16x2(x, 0.f)); }
// silu(g) * u in fp32 from bf16 values (the SwiGLU pass's arithmetic)
__device__ __forceinline__ float silu_mul(float g, float u) { return g / (1.0f + expf(-g)) * u; }

template <int BN>
__global__ void __launch_bounds__(kThreads, 1) gemm_kernel(const __grid_constant__ GemmArgs g) {
  using Lay = GemmLayout<BN>;
  constexpr int S = Lay::kStages;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + Lay::kBar);
  int* misc = reinterpret_cast<int*>(smem + Lay::kMisc);
  volatile int* abort_flag = misc + 1;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int KT = (g.K + kBK - 1) / kBK;
  const int BNo = g.swiglu ? BN / 2 : BN;  // output columns per tile

  TileMap tm;
  tm.nseg = g.nseg;
  tm.m_tiles = (g.T + kBM - 1) / kBM;
  tm.n_tiles = 0;
  for (int s = 0; s < g.nseg; ++s) {
    tm.seg_tiles[s] = (g.seg[s].N + BNo - 1) / BNo;
    tm.n_tiles += tm.seg_tiles[s];
  }
  const int out_tiles = tm.m_tiles * tm.n_tiles;
  const int KS = g.ksplit;
  const int tiles = out_tiles * KS;  // work item t: output tile t % out_tiles, K range t / out_tiles

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&bars[kBarFull + s], 1);
      mbar_init(&bars[kBarEmpty + s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&bars[kBarAccFull + b], 1);
      mbar_init(&bars[kBarAccEmpty + b], 4);  // one arrival per epilogue warp
    }
    mbar_init(&bars[kBarDrain], 1);
    fence_barrier_init();
    misc[1] = 0;
  }
  if (warp == 1) {
    tmem_alloc(reinterpret_cast<uint32_t*>(misc), Lay::kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  griddep_wait();  // global memory from here on
  griddep_launch_dependents();
  const uint32_t tmem = static_cast<uint32_t>(misc[0]);

  if (warp == 0) {
    // ------------------------------------------------------------ producer --
    if (lane == 0) {
      tma_prefetch_desc(&g.tm_x);
      for (int s = 0; s < g.nseg; ++s) tma_prefetch_desc(&g.seg[s].tm_w);
      int st = 0, issued = 0;
      uint32_t phase = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x) {
        int m0, seg, nt;
        tm.locate(t % out_tiles, &m0, &seg, &nt);
        const int ks = t / out_tiles;
        const int k_begin = KT * ks / KS, k_end = KT * (ks + 1) / KS;
        const CUtensorMap* tw = &g.seg[seg].tm_w;
        // W rows of this tile: BN consecutive rows, or BN/2 gate rows and the
        // BN/2 up rows I further on
        const int r0 = nt * BNo;
        const int r1 = g.swiglu ? g.I + nt * BNo : r0 + BN / 2;
        for (int k = k_begin; k < k_end; ++k) {
          if (issued >= S && !(ok = mbar_wait(&bars[kBarEmpty + st], phase ^ 1u, abort_flag, g.err))) break;
          uint8_t* sa = smem + st * Lay::kStage;
          uint8_t* sb = sa + Lay::kA;
          mbar_arrive_expect_tx(&bars[kBarFull + st], Lay::kStage);
          tma_load_2d(sa, &g.tm_x, &bars[kBarFull + st], k * kBK, m0);
          tma_load_2d(sb, tw, &bars[kBarFull + st], k * kBK, r0);
          tma_load_2d(sb + Lay::kB / 2, tw, &bars[kBarFull + st], k * kBK, r1);
          ++issued;
          if (++st == S) {
            st = 0;
            phase ^= 1u;
          }
        }
      }
      if (!ok) {
        // unwinding: let the copies in flight land before the CTA exits
        volatile int no_abort = 0;
        for (int j = issued > S ? issued - S : 0; j < issued; ++j)
          mbar_wait(&bars[kBarFull + j % S], (j / S) & 1, &no_abort, g.err);
      }
    }
  } else if (warp == 1) {
    // ----------------------------------------------------------------- MMA --
    if (lane == 0) {
      constexpr uint32_t kIdesc = make_idesc_bf16(kBM, BN, 0);
      int st = 0, j = 0;
      uint32_t phase = 0;
      bool ok = true, issued_any = false;
      for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x, ++j) {
        const int buf = j & 1;
        if (!(ok = mbar_wait(&bars[kBarAccEmpty + buf], ((j >> 1) & 1) ^ 1u, abort_flag, g.err))) break;
        tc_fence_after();
        const uint32_t acc = tmem + static_cast<uint32_t>(buf * BN);
        const int ks = t / out_tiles;
        const int k_begin = KT * ks / KS, k_end = KT * (ks + 1) / KS;
        for (int k = k_begin; k < k_end; ++k) {
          if (!(ok = mbar_wait(&bars[kBarFull + st], phase, abort_flag, g.err))) break;
          tc_fence_after();
          const uint32_t sa = smem_u32(smem + st * Lay::kStage);
          const uint32_t sb = sa + Lay::kA;
#pragma unroll
          for (int kk = 0; kk < kBK / 16; ++kk) {
            const uint64_t ad = make_sdesc_sw128(sa + kk * 32, 16, 1024);
            const uint64_t bd = make_sdesc_sw128(sb + kk * 32, 16, 1024);
            umma_bf16_ss(acc, ad, bd, kIdesc, (k > k_begin || kk > 0) ? 1u : 0u);
          }
          issued_any = true;
          umma_commit(&bars[kBarEmpty + st]);  // the stage is free once these MMAs complete
          if (++st == S) {
            st = 0;
            phase ^= 1u;
          }
        }
        if (ok) umma_commit(&bars[kBarAccFull + buf]);
      }
      if (!ok && issued_any) {
        // unwinding: the MMAs in flight finish before TMEM is released
        volatile int no_abort = 0;
        umma_commit(&bars[kBarDrain]);
        mbar_wait(&bars[kBarDrain], 0, &no_abort, g.err);
      }
    }
  } else {
    // ------------------------------------------------------------ epilogue --
    const int quarter = warp & 3;  // warps 2, 3, 4, 5 -> TMEM lanes 64, 96, 0, 32 ..
    const int r = quarter * 32 + lane;
    const uint32_t lane_base = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
    int j = 0;
    for (int t = blockIdx.x; t < tiles; t += gridDim.x, ++j) {
      const int buf = j & 1;
      const bool ok = __all_sync(0xffffffffu, mbar_wait(&bars[kBarAccFull + buf], (j >> 1) & 1, abort_flag, g.err));
      if (!ok) break;
      tc_fence_after();
      int m0, seg, nt;
      tm.locate(t % out_tiles, &m0, &seg, &nt);
      const GemmSeg sg = g.seg[seg];
      const int row = m0 + r;
      const bool row_ok = row < g.T;
      const uint32_t acc = lane_base + static_cast<uint32_t>(buf * BN);
      if (KS > 1) {
        // fp32 partial sums of this K range: columns of the partial row are the
        // segments side by side (swiglu: gate columns, then the I up columns)
        int P = 0, off = 0;
        for (int s2 = 0; s2 < g.nseg; ++s2) {
          if (s2 == seg) off = P;
          P += g.seg[s2].N;
        }
        if (g.swiglu) P = 2 * g.I;
        float* prow = g.part + (static_cast<int64_t>(t / out_tiles) * g.T + row) * P;
#pragma unroll 1
        for (int c = 0; c < BN / 32; ++c) {
          float v[32];
          tmem_ld32(acc + c * 32, v);
          if (c == BN / 32 - 1) {
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&bars[kBarAccEmpty + buf]);
          }
          // output column of accumulator column c * 32 (+ i) and its bound
          int n, lim;
          if (g.swiglu) {
            const int half = (c * 32) / (BN / 2);
            n = nt * (BN / 2) + c * 32 - half * (BN / 2);
            lim = g.I;
            n += half * g.I;
            lim += half * g.I;
          } else {
            n = nt * BN + c * 32;
            lim = sg.N;
            n += off;
            lim += off;
          }
          if (!row_ok) continue;
#pragma unroll
          for (int q = 0; q < 8; ++q)
            if (n + 4 * q < lim)
              *reinterpret_cast<float4*>(prow + n + 4 * q) =
                  make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
        }
      } else if (!g.swiglu) {
        const int n0 = nt * BN;
        const uint16_t* crow = (seg == 0 && g.C != nullptr) ? g.C + static_cast<int64_t>(row) * sg.N : nullptr;
        uint16_t* drow = sg.D + static_cast<int64_t>(row) * sg.N;
#pragma unroll 1
        for (int c = 0; c < BN / 32; ++c) {
          float v[32];
          tmem_ld32(acc + c * 32, v);
          if (c == BN / 32 - 1) {
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&bars[kBarAccEmpty + buf]);
          }
          const int n = n0 + c * 32;
          if (!row_ok || n >= sg.N) continue;
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            if (n + 8 * q >= sg.N) break;
            float add[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
            if (crow != nullptr) {
              const uint4 cv = *reinterpret_cast<const uint4*>(crow + n + 8 * q);
              const uint32_t cw[4] = {cv.x, cv.y, cv.z, cv.w};
#pragma unroll
              for (int i = 0; i < 4; ++i) {
                add[2 * i] = bf16_lo(cw[i]);
                add[2 * i + 1] = bf16_hi(cw[i]);
              }
            }
            uint4 o;
            o.x = pack_bf16x2(v[8 * q + 0] + add[0], v[8 * q + 1] + add[1]);
            o.y = pack_bf16x2(v[8 * q + 2] + add[2], v[8 * q + 3] + add[3]);
            o.z = pack_bf16x2(v[8 * q + 4] + add[4], v[8 * q + 5] + add[5]);
            o.w = pack_bf16x2(v[8 * q + 6] + add[6], v[8 * q + 7] + add[7]);
            *reinterpret_cast<uint4*>(drow + n + 8 * q) = o;
          }
        }
      } else {
        // columns [0, BN/2) of the accumulator are gate outputs nt*BN/2 + c,
        // columns [BN/2, BN) the matching up outputs
        const int n0 = nt * (BN / 2);
        uint16_t* drow = sg.D + static_cast<int64_t>(row) * g.I;
#pragma unroll 1
        for (int c = 0; c < BN / 64; ++c) {
          float gv[32], uv[32];
          tmem_ld32(acc + c * 32, gv);
          tmem_ld32(acc + BN / 2 + c * 32, uv);
          if (c == BN / 64 - 1) {
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&bars[kBarAccEmpty + buf]);
          }
          const int n = n0 + c * 32;
          if (!row_ok || n >= g.I) continue;
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            if (n + 8 * q >= g.I) break;
            float a[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) a[i] = silu_mul(bf16_round(gv[8 * q + i]), bf16_round(uv[8 * q + i]));
            uint4 o;
            o.x = pack_bf16x2(a[0], a[1]);
            o.y = pack_bf16x2(a[2], a[3]);
            o.z = pack_bf16x2(a[4], a[5]);
            o.w = pack_bf16x2(a[6], a[7]);
            *reinterpret_cast<uint4*>(drow + n + 8 * q) = o;
          }
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, Lay::kTmemCols);
  }
}

// Split-K reduction: the ksplit partials of each output, added in split
// order, then the GEMM epilogue's arithmetic (residual, or SwiGLU of the
// bf16-rounded gate and up sums), one rounding, 8 outputs per thread.
__global__ void __launch_bounds__(256) gemm_reduce_kernel(const __grid_constant__ GemmArgs g) {
  griddep_wait();
  griddep_launch_dependents();
  int P = 0;
  for (int s = 0; s < g.nseg; ++s) P += g.seg[s].N;
  const int W = g.swiglu ? g.I : P;  // outputs per row
  if (g.swiglu) P = 2 * g.I;
  const int64_t per_row = W / 8;
  const int64_t total = static_cast<int64_t>(g.T) * per_row;
  const int64_t split_stride = static_cast<int64_t>(g.T) * P;
  for (int64_t e = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; e < total;
       e += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t row = e / per_row;
    const int col = static_cast<int>(e % per_row) * 8;
    float a[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f}, b[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    const float* src = g.part + row * P + col;
    for (int ks = 0; ks < g.ksplit; ++ks) {
      const float4 x0 = *reinterpret_cast<const float4*>(src + ks * split_stride);
      const float4 x1 = *reinterpret_cast<const float4*>(src + ks * split_stride + 4);
      a[0] += x0.x; a[1] += x0.y; a[2] += x0.z; a[3] += x0.w;
      a[4] += x1.x; a[5] += x1.y; a[6] += x1.z; a[7] += x1.w;
      if (g.swiglu) {
        const float4 y0 = *reinterpret_cast<const float4*>(src + ks * split_stride + g.I);
        const float4 y1 = *reinterpret_cast<const float4*>(src + ks * split_stride + g.I + 4);
        b[0] += y0.x; b[1] += y0.y; b[2] += y0.z; b[3] += y0.w;
        b[4] += y1.x; b[5] += y1.y; b[6] += y1.z; b[7] += y1.w;
      }
    }
    uint16_t* dst;
    if (g.swiglu) {
#pragma unroll
      for (int i = 0; i < 8; ++i) a[i] = silu_mul(bf16_round(a[i]), bf16_round(b[i]));
      dst = g.seg[0].D + row * g.I + col;
    } else {
      int s = 0, c = col;
      while (s < g.nseg - 1 && c >= g.seg[s].N) c -= g.seg[s++].N;
      if (s == 0 && g.C != nullptr) {
        const uint4 cv = *reinterpret_cast<const uint4*>(g.C + row * g.seg[0].N + c);
        const uint32_t cw[4] = {cv.x, cv.y, cv.z, cv.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          a[2 * i] += bf16_lo(cw[i]);
          a[2 * i + 1] += bf16_hi(cw[i]);
        }
      }
      dst = g.seg[s].D + row * g.seg[s].N + c;
    }
    *reinterpret_cast<uint4*>(dst) =
        make_uint4(pack_bf16x2(a[0], a[1]), pack_bf16x2(a[2], a[3]), pack_bf16x2(a[4], a[5]), pack_bf16x2(a[6], a[7]));
  }
}

}  // namespace

int gemm_tile_n(int T) { return T <= 512 ? 128 : 256; }

cudaError_t launch_gemm_main(const GemmArgs& g, int BN, int grid, cudaStream_t st);

int gemm_tiles(const GemmArgs& g) {
  const int BN = gemm_tile_n(g.T);
  const int BNo = g.swiglu ? BN / 2 : BN;
  int n_tiles = 0;
  for (int s = 0; s < g.nseg; ++s) n_tiles += (g.seg[s].N + BNo - 1) / BNo;
  return (g.T + kBM - 1) / kBM * n_tiles;
}

int gemm_ksplit(int T, int K, int tiles, int num_sms, int max_split) {
  (void)T;
  if (tiles <= 0 || 2 * tiles > num_sms) return 1;
  const int KT = (K + kBK - 1) / kBK;
  int ks = num_sms / tiles;
  ks = ks < KT / 4 ? ks : KT / 4;  // at least four K steps per split
  ks = ks < max_split ? ks : max_split;
  return ks > 1 ? ks : 1;
}

cudaError_t launch_gemm(const GemmArgs& g, int num_sms, cudaStream_t st) {
  if (g.T <= 0) return cudaSuccess;
  if (g.ksplit < 1 || (g.ksplit > 1 && g.part == nullptr)) return cudaErrorInvalidValue;
  const int BN = gemm_tile_n(g.T);
  const int tiles = gemm_tiles(g) * g.ksplit;
  if (tiles == 0) return cudaSuccess;
  const int grid = tiles < num_sms ? tiles : num_sms;
  if (g.ksplit > 1) {
    cudaError_t e = launch_gemm_main(g, BN, grid, st);
    if (e != cudaSuccess) return e;
    int W = 0;
    for (int s = 0; s < g.nseg; ++s) W += g.seg[s].N;
    if (g.swiglu) W = g.I;
    const int64_t vec = static_cast<int64_t>(g.T) * (W / 8);
    const int blocks = static_cast<int>((vec + 255) / 256 < 4 * num_sms ? (vec + 255) / 256 : 4 * num_sms);
    return launch_kernel(gemm_reduce_kernel, dim3(blocks), dim3(256), 0, st, 0, g);
  }
  return launch_gemm_main(g, BN, grid, st);
}

cudaError_t launch_gemm_main(const GemmArgs& g, int BN, int grid, cudaStream_t st) {
  static PerDeviceOnce setup128, setup256;
  if (BN == 128) {
    const cudaError_t e = setup128.run([] {
      return cudaFuncSetAttribute(gemm_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  GemmLayout<128>::kAlloc);
    });
    if (e != cudaSuccess) return e;
    return launch_kernel(gemm_kernel<128>, dim3(grid), dim3(kThreads), GemmLayout<128>::kAlloc, st, 0, g);
  }
  const cudaError_t e = setup256.run([] {
    return cudaFuncSetAttribute(gemm_kernel<256>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                GemmLayout<256>::kAlloc);
  });
  if (e != cudaSuccess) return e;
  return launch_kernel(gemm_kernel<256>, dim3(grid), dim3(kThreads), GemmLayout<256>::kAlloc, st, 0, g);
}

}  // namespace kvr
