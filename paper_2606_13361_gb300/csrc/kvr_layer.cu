// kvr_layer.cu -- a whole Qwen3-style decoder layer around the hot path, so
// that the whole-layer costs of prefill and of a reuse step can be measured
// (the paper's Table 1 times whole-model forwards; Sec. 5).
//
//   x  = RMSNorm(h)                      rmsnorm_rows_kernel
//   q, k, v = x Wq^T, x Wk^T, x Wv^T     bf16 GEMMs, fp32 accumulation: the tcgen05 GEMM
//                                        (kvr_gemm.cu, one launch for all three); up to
//                                        8 rows gemv_pro_kernel, bound by the weight read
//   o  = attention(...)                  kvr_append_kv + kvr_prefill_attn, or
//                                        kvr_decode_step (reuse path)
//   h1 = h + o Wo^T                      GEMM, residual in the epilogue
//   x2 = RMSNorm(h1)                     rmsnorm_rows_kernel
//   a  = silu(x2 Wg^T) * (x2 Wu^T)       GEMM with SwiGLU in its epilogue (up to 8
//                                        rows: GEMV, then SwiGLU fused into the next GEMV)
//   h_out = h1 + a Wd^T                  GEMM, residual in the epilogue
//
// Every tensor between two operations is bf16 (the model runs in bf16); each
// operation computes in fp32 and rounds once.  The norms and SwiGLU are
// memory-bound streams (16-byte accesses, one row per CTA for the norm); the
// projections are this library's tcgen05 GEMM, except for a few rows (a
// decode step), where its weight-streaming GEMV reads each weight once.
#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>

#include "kvr_internal.h"
#include "kvr_ptx.cuh"

namespace kvr {

// Defined in kvr_api.cu.
const kvr_model_desc* ctx_desc(const kvr_ctx* c);
void ctx_add_launches(kvr_ctx* c, int n);
int* ctx_err(kvr_ctx* c);
kvr_status set_error(kvr_status s, const char* msg);

namespace {

kvr_status fail(kvr_status s, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  return set_error(s, buf);
}

constexpr int kNormThreads = 256;
constexpr size_t kAlignWs = 256;
// Split-K partials of one projection: ksplit x T x width fp32.  A split is
// only taken when the output tiles cover at most half of the SMs, which bounds
// this by SMs x 128 x 128 x 4 bytes (10 MB on 152 SMs); calls clamp ksplit to it.
constexpr size_t kSplitBytes = size_t(16) << 20;
constexpr int kMaxKSplit = 16;

size_t align_ws(size_t x) { return (x + kAlignWs - 1) / kAlignWs * kAlignWs; }

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

// y[t] = bf16(x[t] / sqrt(mean(x[t]^2) + eps) * w), one CTA per row, n % 8 == 0.
__global__ void __launch_bounds__(kNormThreads) rmsnorm_rows_kernel(const uint16_t* __restrict__ x,
                                                                    const uint16_t* __restrict__ w,
                                                                    uint16_t* __restrict__ y, int n, float eps) {
  __shared__ float red[kNormThreads / 32];
  griddep_wait();
  griddep_launch_dependents();
  const uint4* xr = reinterpret_cast<const uint4*>(x + static_cast<int64_t>(blockIdx.x) * n);
  const uint4* wr = reinterpret_cast<const uint4*>(w);
  uint4* yr = reinterpret_cast<uint4*>(y + static_cast<int64_t>(blockIdx.x) * n);
  const int nv = n / 8;
  float ss = 0.f;
  for (int i = threadIdx.x; i < nv; i += kNormThreads) {
    const uint4 v = xr[i];
    const uint32_t u[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float a = bf16_lo(u[j]), b = bf16_hi(u[j]);
      ss = fmaf(a, a, fmaf(b, b, ss));
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
  __syncthreads();
  float tot = 0.f;
#pragma unroll
  for (int i = 0; i < kNormThreads / 32; ++i) tot += red[i];
  const float inv = 1.0f / sqrtf(tot / static_cast<float>(n) + eps);
  for (int i = threadIdx.x; i < nv; i += kNormThreads) {
    const uint4 v = xr[i], g = wr[i];
    const uint32_t u[4] = {v.x, v.y, v.z, v.w}, gw[4] = {g.x, g.y, g.z, g.w};
    uint32_t o[4];
#pragma unroll
    for (int j = 0; j < 4; ++j)
      o[j] = pack_bf16x2(bf16_lo(u[j]) * inv * bf16_lo(gw[j]), bf16_hi(u[j]) * inv * bf16_hi(gw[j]));
    yr[i] = make_uint4(o[0], o[1], o[2], o[3]);
  }
}

// silu(g) * u in fp32 from bf16 values (the SwiGLU step's arithmetic; the
// decode-size path applies it in the down projection's prologue)
__device__ __forceinline__ float silu_mul(float g, float u) { return g / (1.0f + expf(-g)) * u; }

// ---- few rows: D[T][N] = X[T][K] W[N][K]^T (+ C[T][N]), T <= kGemvRows ----
// A decode step multiplies one row per sequence by every weight matrix: the
// weights are read once and the call is bound by HBM.  One warp per output
// column n (a row of W): 16-byte streaming loads of W, eight in flight per
// lane, the T rows of X through L1, fp32 sums reduced across the warp, one
// rounding of sum (+ C) to bf16 (the GEMM epilogue's arithmetic).
constexpr int kGemvRows = 8;
constexpr int kGemvWarps = 8;
constexpr int kGemvUnroll = 8;  // 16-byte weight loads in flight per lane

__device__ __forceinline__ float dot8(const uint4& w, const uint4& x) {
  const uint32_t a[4] = {w.x, w.y, w.z, w.w}, b[4] = {x.x, x.y, x.z, x.w};
  float s = 0.f;
#pragma unroll
  for (int i = 0; i < 4; ++i) s = fmaf(bf16_lo(a[i]), bf16_lo(b[i]), fmaf(bf16_hi(a[i]), bf16_hi(b[i]), s));
  return s;
}

template <int TM>
__global__ void __launch_bounds__(kGemvWarps * 32) gemv_kernel(const uint16_t* __restrict__ W,
                                                               const uint16_t* __restrict__ X,
                                                               const uint16_t* __restrict__ C,
                                                               uint16_t* __restrict__ D, int N, int K, int T) {
  const int lane = threadIdx.x & 31;
  const int n = blockIdx.x * kGemvWarps + (threadIdx.x >> 5);
  // The weight row starts moving into L2 before the dependency: a prefetch is
  // only a hint, so it is right whatever the previous kernel writes, and the
  // weights stream while that kernel finishes.
  if (n < N && lane == 0) l2_prefetch(W + static_cast<int64_t>(n) * K, static_cast<uint32_t>(K) * 2);
  griddep_wait();
  griddep_launch_dependents();
  if (n >= N) return;
  const uint4* w = reinterpret_cast<const uint4*>(W + static_cast<int64_t>(n) * K);
  const int nv = K / 8;
  float acc[TM];
#pragma unroll
  for (int t = 0; t < TM; ++t) acc[t] = 0.f;
  for (int i = lane; i < nv; i += 32 * kGemvUnroll) {
    uint4 wv[kGemvUnroll];
#pragma unroll
    for (int u = 0; u < kGemvUnroll; ++u)
      if (i + u * 32 < nv) wv[u] = __ldcs(w + i + u * 32);
#pragma unroll
    for (int u = 0; u < kGemvUnroll; ++u) {
      const int idx = i + u * 32;
      if (idx >= nv) break;
#pragma unroll
      for (int t = 0; t < TM; ++t)
        if (t < T) acc[t] += dot8(wv[u], __ldg(reinterpret_cast<const uint4*>(X + static_cast<int64_t>(t) * K) + idx));
    }
  }
  float mine = 0.f;
#pragma unroll
  for (int t = 0; t < TM; ++t) {
    float v = acc[t];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if (lane == t) mine = v;
  }
  if (lane < T) {
    const int64_t e = static_cast<int64_t>(lane) * N + n;
    const float c = C != nullptr ? __uint_as_float(static_cast<uint32_t>(C[e]) << 16) : 0.f;
    D[e] = static_cast<uint16_t>(pack_bf16x2(mine + c, 0.f) & 0xffffu);
  }
}

// ---- few rows, fused: the operation before a projection feeds it directly ----
// One launch computes its block's bf16 input rows into shared memory (RMSNorm
// of the residual stream with the arithmetic of rmsnorm_rows_kernel, or
// SwiGLU of the gate/up rows with that of the GEMM's SwiGLU epilogue) and then
// the projection as above, over up to three weight matrices that share that
// input (q, k, v).  A decode step's layer is then five launches.
enum { kProNorm = 1, kProSwiglu = 2 };

struct GemvSeg {
  const uint16_t* W;
  uint16_t* D;
  int N;
};

struct GemvArgs {
  GemvSeg seg[3];
  int nseg;
  int K;                // input width (hidden for the norm, the MLP width for SwiGLU)
  int T;
  const uint16_t* X;    // norm: rows [T][K]; SwiGLU: gate/up rows [T][2K]
  const uint16_t* C;    // residual added to segment 0, or null
  const uint16_t* nw;   // norm weight [K]
  float eps;
};

template <int TM, int PRO>
__global__ void __launch_bounds__(kGemvWarps * 32) gemv_pro_kernel(const __grid_constant__ GemvArgs g) {
  extern __shared__ uint4 xs_raw[];
  __shared__ float red[kGemvWarps];
  const int T = g.T, K = g.K, nv = K / 8;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  // this warp's output column over the concatenated segments; its weight row
  // starts moving into L2 before the dependency (a hint: right whatever the
  // previous kernel writes), so the weights stream while that kernel and the
  // prologue below run
  int n = blockIdx.x * kGemvWarps + warp, s = 0;
  while (s < g.nseg && n >= g.seg[s].N) n -= g.seg[s++].N;
  if (s < g.nseg && lane == 0) l2_prefetch(g.seg[s].W + static_cast<int64_t>(n) * K, static_cast<uint32_t>(K) * 2);
  griddep_wait();
  griddep_launch_dependents();
  if constexpr (PRO == kProNorm) {
    for (int t = 0; t < T; ++t) {
      const uint4* xr = reinterpret_cast<const uint4*>(g.X + static_cast<int64_t>(t) * K);
      float ss = 0.f;
      for (int i = threadIdx.x; i < nv; i += kGemvWarps * 32) {
        const uint4 v = xr[i];
        const uint32_t u[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const float a = bf16_lo(u[j]), b = bf16_hi(u[j]);
          ss = fmaf(a, a, fmaf(b, b, ss));
        }
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
      if (lane == 0) red[warp] = ss;
      __syncthreads();
      float tot = 0.f;
#pragma unroll
      for (int i = 0; i < kGemvWarps; ++i) tot += red[i];
      const float inv = 1.0f / sqrtf(tot / static_cast<float>(K) + g.eps);
      const uint4* wr = reinterpret_cast<const uint4*>(g.nw);
      for (int i = threadIdx.x; i < nv; i += kGemvWarps * 32) {
        const uint4 v = xr[i], ww = wr[i];
        const uint32_t u[4] = {v.x, v.y, v.z, v.w}, gw[4] = {ww.x, ww.y, ww.z, ww.w};
        uint32_t o[4];
#pragma unroll
        for (int j = 0; j < 4; ++j)
          o[j] = pack_bf16x2(bf16_lo(u[j]) * inv * bf16_lo(gw[j]), bf16_hi(u[j]) * inv * bf16_hi(gw[j]));
        xs_raw[t * nv + i] = make_uint4(o[0], o[1], o[2], o[3]);
      }
      __syncthreads();  // red[] is rewritten by the next row
    }
  } else {
    for (int e = threadIdx.x; e < T * nv; e += kGemvWarps * 32) {
      const int t = e / nv, c = (e % nv) * 8;
      const uint4 gg = *reinterpret_cast<const uint4*>(g.X + static_cast<int64_t>(t) * 2 * K + c);
      const uint4 uu = *reinterpret_cast<const uint4*>(g.X + static_cast<int64_t>(t) * 2 * K + K + c);
      const uint32_t gw[4] = {gg.x, gg.y, gg.z, gg.w}, uw[4] = {uu.x, uu.y, uu.z, uu.w};
      uint32_t o[4];
#pragma unroll
      for (int j = 0; j < 4; ++j)
        o[j] = pack_bf16x2(silu_mul(bf16_lo(gw[j]), bf16_lo(uw[j])), silu_mul(bf16_hi(gw[j]), bf16_hi(uw[j])));
      xs_raw[e] = make_uint4(o[0], o[1], o[2], o[3]);
    }
    __syncthreads();
  }
  // the projection: one warp per output column over the concatenated segments
  if (s >= g.nseg) return;
  const GemvSeg sg = g.seg[s];
  const uint4* w = reinterpret_cast<const uint4*>(sg.W + static_cast<int64_t>(n) * K);
  float acc[TM];
#pragma unroll
  for (int t = 0; t < TM; ++t) acc[t] = 0.f;
  for (int i = lane; i < nv; i += 32 * kGemvUnroll) {
    uint4 wv[kGemvUnroll];
#pragma unroll
    for (int u = 0; u < kGemvUnroll; ++u)
      if (i + u * 32 < nv) wv[u] = __ldcs(w + i + u * 32);
#pragma unroll
    for (int u = 0; u < kGemvUnroll; ++u) {
      const int idx = i + u * 32;
      if (idx >= nv) break;
#pragma unroll
      for (int t = 0; t < TM; ++t)
        if (t < T) acc[t] += dot8(wv[u], xs_raw[t * nv + idx]);
    }
  }
  float mine = 0.f;
#pragma unroll
  for (int t = 0; t < TM; ++t) {
    float v = acc[t];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if (lane == t) mine = v;
  }
  if (lane < T) {
    const int64_t e = static_cast<int64_t>(lane) * sg.N + n;
    const float c = (s == 0 && g.C != nullptr) ? __uint_as_float(static_cast<uint32_t>(g.C[e]) << 16) : 0.f;
    sg.D[e] = static_cast<uint16_t>(pack_bf16x2(mine + c, 0.f) & 0xffffu);
  }
}

template <int TM, int PRO>
cudaError_t launch_gemv_pro(const GemvArgs& g, cudaStream_t st) {
  const size_t smem = static_cast<size_t>(g.T) * g.K * 2;
  if (smem > 48 * 1024) {
    // the largest size set so far on each device (cudaFuncSetAttribute acts on
    // the current device only)
    static std::mutex mu;
    static size_t configured[kMaxDevices] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(mu);
    if (smem > configured[dev]) {
      e = cudaFuncSetAttribute(gemv_pro_kernel<TM, PRO>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               static_cast<int>(smem));
      if (e != cudaSuccess) return e;
      configured[dev] = smem;
    }
  }
  int rows = 0;
  for (int s = 0; s < g.nseg; ++s) rows += g.seg[s].N;
  return launch_kernel(gemv_pro_kernel<TM, PRO>, dim3((rows + kGemvWarps - 1) / kGemvWarps), dim3(kGemvWarps * 32),
                       smem, st, 0, g);
}

template <int PRO>
cudaError_t gemv_pro(const GemvArgs& g, cudaStream_t st) {
  return g.T == 1 ? launch_gemv_pro<1, PRO>(g, st) : launch_gemv_pro<kGemvRows, PRO>(g, st);
}

// ---- projections: D[T][N] = X[T][K] W[N][K]^T (+ C[T][N]) in bf16 ----
// Up to kGemvRows rows: the weight-streaming GEMV above.  More rows: the
// tcgen05 GEMM (kvr_gemm.cu), several weight matrices sharing X in one launch,
// or the gate/up projection with SwiGLU in its epilogue.
struct Proj {
  const void* W;
  void* D;
  int N;
};

int sm_count() {
  static int counts[kMaxDevices] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return 148;
  if (counts[dev] == 0) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 148;
    counts[dev] = n;
  }
  return counts[dev];
}

bool al16(const void* p) { return p && (reinterpret_cast<uintptr_t>(p) & 15) == 0; }

// The tcgen05 GEMM over `n` projections of X (any T >= 1); swiglu: one W of
// [2 I][K] rows whose output is silu(gate) * up, [T][I].
kvr_status tc_linear(int T, int K, const void* X, const Proj* p, int n, const void* C, bool swiglu, int* err,
                     cudaStream_t st, float* part = nullptr, size_t part_bytes = 0, int* launches = nullptr) {
  if (T <= 0) return KVR_OK;
  if (n < 1 || n > kMaxGemmSegs || (swiglu && n != 1)) return fail(KVR_ERR_INVALID_ARG, "bad projection count");
  if (K <= 0 || K % 8 || !al16(X) || (C != nullptr && !al16(C)))
    return fail(KVR_ERR_INVALID_ARG, "K must be a positive multiple of 8 and X, C 16-byte aligned");
  GemmArgs g{};
  const int BN = gemm_tile_n(T);
  if (encode_bf16_2d(&g.tm_x, X, static_cast<uint64_t>(K), static_cast<uint64_t>(T), 64, 128) != 0)
    return fail(KVR_ERR_CUDA, "cuTensorMapEncodeTiled(X) failed");
  for (int s = 0; s < n; ++s) {
    if (p[s].N <= 0 || p[s].N % 8 || !al16(p[s].W) || !al16(p[s].D))
      return fail(KVR_ERR_INVALID_ARG, "output widths must be positive multiples of 8, W and D 16-byte aligned");
    const uint64_t rows = static_cast<uint64_t>(p[s].N) * (swiglu ? 2 : 1);
    if (encode_bf16_2d(&g.seg[s].tm_w, p[s].W, static_cast<uint64_t>(K), rows, 64, static_cast<uint32_t>(BN / 2)) != 0)
      return fail(KVR_ERR_CUDA, "cuTensorMapEncodeTiled(W) failed");
    g.seg[s].D = static_cast<uint16_t*>(p[s].D);
    g.seg[s].N = p[s].N;
  }
  g.nseg = n;
  g.T = T;
  g.K = K;
  g.C = static_cast<const uint16_t*>(C);
  g.swiglu = swiglu ? 1 : 0;
  g.I = swiglu ? p[0].N : 0;
  g.err = err;
  // split K when the output tiles alone would leave most SMs idle, as far as
  // the partial sums fit the caller's scratch
  size_t P = 0;
  for (int s = 0; s < n; ++s) P += static_cast<size_t>(p[s].N);
  if (swiglu) P = 2 * static_cast<size_t>(p[0].N);
  int ks = part != nullptr ? gemm_ksplit(T, K, gemm_tiles(g), sm_count(), kMaxKSplit) : 1;
  while (ks > 1 && static_cast<size_t>(ks) * T * P * sizeof(float) > part_bytes) --ks;
  g.ksplit = ks;
  g.part = ks > 1 ? part : nullptr;
  const cudaError_t e = launch_gemm(g, sm_count(), st);
  if (e != cudaSuccess) return fail(KVR_ERR_CUDA, "gemm launch: %s", cudaGetErrorString(e));
  if (launches) *launches += ks > 1 ? 2 : 1;
  return KVR_OK;
}

// One projection with the layer's dispatch: GEMV up to kGemvRows rows.
kvr_status linear(int T, int N, int K, const void* W, const void* X, const void* C, void* D, int* err,
                  cudaStream_t st) {
  if (T <= kGemvRows && K % 8 == 0) {
    const dim3 grid((N + kGemvWarps - 1) / kGemvWarps), block(kGemvWarps * 32);
    const uint16_t *w16 = static_cast<const uint16_t*>(W), *x16 = static_cast<const uint16_t*>(X),
                   *c16 = static_cast<const uint16_t*>(C);
    uint16_t* d16 = static_cast<uint16_t*>(D);
    const cudaError_t e = T == 1 ? launch_kernel(gemv_kernel<1>, grid, block, 0, st, 0, w16, x16, c16, d16, N, K, T)
                                 : launch_kernel(gemv_kernel<kGemvRows>, grid, block, 0, st, 0, w16, x16, c16, d16, N,
                                                 K, T);
    if (e != cudaSuccess) return fail(KVR_ERR_CUDA, "gemv launch: %s", cudaGetErrorString(e));
    return KVR_OK;
  }
  const Proj p{W, D, N};
  return tc_linear(T, K, X, &p, 1, C, false, err, st);
}

// Workspace regions for T tokens.
struct LayerWs {
  uint16_t *x, *q, *k, *v, *qr, *o, *h1, *x2, *gu, *a;
  float* part;  // split-K partial sums of the projections (short batches)
  size_t bytes;
};

LayerWs carve(char* base, const kvr_model_desc& d, const kvr_layer_desc& l, size_t T) {
  LayerWs w{};
  size_t off = 0;
  auto take = [&](size_t elems) {
    char* p = base ? base + off : nullptr;
    off += align_ws(elems * 2);
    return reinterpret_cast<uint16_t*>(p);
  };
  const size_t qd = static_cast<size_t>(d.n_q_heads) * d.head_dim, kd = static_cast<size_t>(d.n_kv_heads) * d.head_dim;
  w.x = take(T * l.hidden);
  w.q = take(T * qd);
  w.k = take(T * kd);
  w.v = take(T * kd);
  w.qr = take(T * qd);
  w.o = take(T * qd);
  w.h1 = take(T * l.hidden);
  w.x2 = take(T * l.hidden);
  // gate/up rows reach memory only at decode sizes (the GEMV path); above
  // that the gate/up GEMM applies SwiGLU in its epilogue
  w.gu = T <= static_cast<size_t>(kGemvRows) ? take(T * 2 * static_cast<size_t>(l.intermediate)) : nullptr;
  w.a = take(T * static_cast<size_t>(l.intermediate));
  w.part = T > static_cast<size_t>(kGemvRows) ? reinterpret_cast<float*>(take(kSplitBytes / 2)) : nullptr;
  w.bytes = off;
  return w;
}

bool ldesc_ok(const kvr_layer_desc* l) {
  return l && l->hidden > 0 && l->intermediate > 0 && l->hidden % 8 == 0 && l->intermediate % 8 == 0;
}

}  // namespace
}  // namespace kvr

using namespace kvr;

extern "C" {

size_t kvr_layer_workspace_bytes(const kvr_model_desc* desc, const kvr_layer_desc* ldesc, uint32_t max_tokens) {
  if (!desc || !ldesc_ok(ldesc) || kvr_artifact_bytes(desc, 1) == 0) return 0;
  const size_t big = carve(nullptr, *desc, *ldesc, max_tokens).bytes;
  const size_t small = carve(nullptr, *desc, *ldesc, std::min<uint32_t>(max_tokens, kGemvRows)).bytes;
  return std::max(big, small);
}

kvr_status kvr_layer_forward(kvr_ctx* c, int layer, const kvr_layer_desc* ldesc, const kvr_layer_weights* w,
                             int n_seqs, const kvr_seq* seqs, const int32_t* start_pos, const int32_t* cu_q,
                             const void* h_in, void* h_out, void* workspace, size_t workspace_bytes,
                             kvr_stream stream) {
  if (!c || !w || !seqs || !start_pos || !cu_q || n_seqs <= 0) return fail(KVR_ERR_INVALID_ARG, "null argument");
  if (!ldesc_ok(ldesc)) return fail(KVR_ERR_INVALID_ARG, "hidden and intermediate must be positive multiples of 8");
  const kvr_model_desc& d = *ctx_desc(c);
  const int T = cu_q[n_seqs];
  if (T <= 0) return T == 0 ? KVR_OK : fail(KVR_ERR_INVALID_ARG, "cu_q must be non-decreasing from 0");
  const void* ptrs[] = {w->input_norm, w->wq, w->wk, w->wv, w->q_norm, w->k_norm, w->wo, w->post_norm,
                        w->w_gate_up, w->w_down, h_in, h_out, workspace};
  for (const void* p : ptrs)
    if (!al16(p)) return fail(KVR_ERR_INVALID_ARG, "weights, activations and workspace must be 16-byte aligned");
  if (h_in == h_out) return fail(KVR_ERR_INVALID_ARG, "h_out may not alias h_in");
  if (reinterpret_cast<uintptr_t>(workspace) % kAlignWs) return fail(KVR_ERR_INVALID_ARG, "workspace must be 256-byte aligned");
  const LayerWs ws = carve(static_cast<char*>(workspace), d, *ldesc, static_cast<size_t>(T));
  if (workspace_bytes < ws.bytes)
    return fail(KVR_ERR_INVALID_ARG, "workspace of %zu bytes < %zu needed for %d tokens", workspace_bytes, ws.bytes, T);
  int* err = ctx_err(c);
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const int H = static_cast<int>(ldesc->hidden), I = static_cast<int>(ldesc->intermediate);
  const int qd = static_cast<int>(d.n_q_heads * d.head_dim), kd = static_cast<int>(d.n_kv_heads * d.head_dim);
  const float eps = static_cast<float>(d.rms_eps);
  const uint16_t* hin = static_cast<const uint16_t*>(h_in);
  uint16_t* hout = static_cast<uint16_t*>(h_out);

  if (T <= kGemvRows) {
    // A decode-sized batch: RMSNorm + q/k/v projections, the decode step,
    // the output projection + residual, RMSNorm + gate/up, SwiGLU + down +
    // residual -- five launches, each projection reading its weights once.
    GemvArgs ga{};
    ga.K = H;
    ga.T = T;
    ga.eps = eps;
    ga.X = hin;
    ga.nw = static_cast<const uint16_t*>(w->input_norm);
    ga.nseg = 3;
    ga.seg[0] = {static_cast<const uint16_t*>(w->wq), ws.q, qd};
    ga.seg[1] = {static_cast<const uint16_t*>(w->wk), ws.k, kd};
    ga.seg[2] = {static_cast<const uint16_t*>(w->wv), ws.v, kd};
    cudaError_t e = gemv_pro<kProNorm>(ga, st);
    if (e != cudaSuccess) return fail(KVR_ERR_CUDA, "norm + qkv launch: %s", cudaGetErrorString(e));
    kvr_status r = kvr_decode_step(c, layer, n_seqs, seqs, start_pos, cu_q, ws.q, ws.k, ws.v, w->q_norm, w->k_norm,
                                   ws.qr, ws.o, nullptr, nullptr, stream);
    if (r != KVR_OK) return r;
    if ((r = linear(T, H, qd, w->wo, ws.o, hin, ws.h1, err, st)) != KVR_OK) return r;
    GemvArgs gb{};
    gb.K = H;
    gb.T = T;
    gb.eps = eps;
    gb.X = ws.h1;
    gb.nw = static_cast<const uint16_t*>(w->post_norm);
    gb.nseg = 1;
    gb.seg[0] = {static_cast<const uint16_t*>(w->w_gate_up), ws.gu, 2 * I};
    if ((e = gemv_pro<kProNorm>(gb, st)) != cudaSuccess)
      return fail(KVR_ERR_CUDA, "norm + gate/up launch: %s", cudaGetErrorString(e));
    GemvArgs gd{};
    gd.K = I;
    gd.T = T;
    gd.X = ws.gu;
    gd.C = ws.h1;
    gd.nseg = 1;
    gd.seg[0] = {static_cast<const uint16_t*>(w->w_down), hout, H};
    if ((e = gemv_pro<kProSwiglu>(gd, st)) != cudaSuccess)
      return fail(KVR_ERR_CUDA, "swiglu + down launch: %s", cudaGetErrorString(e));
    ctx_add_launches(c, 4);  // three fused projections and the output projection
    return KVR_OK;
  }
  cudaError_t e = launch_kernel(rmsnorm_rows_kernel, dim3(T), dim3(kNormThreads), 0, st, 0, hin,
                                static_cast<const uint16_t*>(w->input_norm), ws.x, H, eps);
  if (e != cudaSuccess) return fail(KVR_ERR_CUDA, "rmsnorm launch: %s", cudaGetErrorString(e));
  kvr_status r;
  int nl = 2;  // the two norms; the projections add theirs, the attention calls count their own
  const Proj qkv[3] = {{w->wq, ws.q, qd}, {w->wk, ws.k, kd}, {w->wv, ws.v, kd}};
  if ((r = tc_linear(T, H, ws.x, qkv, 3, nullptr, false, err, st, ws.part, kSplitBytes, &nl)) != KVR_OK) return r;
  if (n_seqs == 1 && start_pos[0] == 0) {
    r = kvr_append_kv(c, layer, 1, seqs, start_pos, cu_q, ws.q, ws.k, ws.v, w->q_norm, w->k_norm, ws.qr, stream);
    if (r == KVR_OK) r = kvr_prefill_attn(c, layer, seqs[0], T, ws.qr, ws.o, nullptr, nullptr, stream);
  } else {
    r = kvr_decode_step(c, layer, n_seqs, seqs, start_pos, cu_q, ws.q, ws.k, ws.v, w->q_norm, w->k_norm, ws.qr,
                        ws.o, nullptr, nullptr, stream);
  }
  if (r != KVR_OK) return r;
  const Proj po{w->wo, ws.h1, H};
  if ((r = tc_linear(T, qd, ws.o, &po, 1, hin, false, err, st, ws.part, kSplitBytes, &nl)) != KVR_OK) return r;
  e = launch_kernel(rmsnorm_rows_kernel, dim3(T), dim3(kNormThreads), 0, st, 0, static_cast<const uint16_t*>(ws.h1),
                    static_cast<const uint16_t*>(w->post_norm), ws.x2, H, eps);
  if (e != cudaSuccess) return fail(KVR_ERR_CUDA, "rmsnorm launch: %s", cudaGetErrorString(e));
  const Proj pgu{w->w_gate_up, ws.a, I};
  if ((r = tc_linear(T, H, ws.x2, &pgu, 1, nullptr, true, err, st, ws.part, kSplitBytes, &nl)) != KVR_OK) return r;
  const Proj pd{w->w_down, hout, H};
  if ((r = tc_linear(T, I, ws.a, &pd, 1, ws.h1, false, err, st, ws.part, kSplitBytes, &nl)) != KVR_OK) return r;
  ctx_add_launches(c, nl);
  return KVR_OK;
}

kvr_status kvr_linear(kvr_ctx* c, int T, int N, int K, const void* x, const void* w, const void* bias_c, void* d,
                      void* workspace, size_t workspace_bytes, kvr_stream stream) {
  if (!c) return fail(KVR_ERR_INVALID_ARG, "null ctx");
  if (T < 0) return fail(KVR_ERR_INVALID_ARG, "T must be >= 0");
  if (workspace != nullptr && !al16(workspace)) return fail(KVR_ERR_INVALID_ARG, "workspace must be 16-byte aligned");
  const Proj p{w, d, N};
  int nl = 0;
  kvr_status r = tc_linear(T, K, x, &p, 1, bias_c, false, ctx_err(c), reinterpret_cast<cudaStream_t>(stream),
                           static_cast<float*>(workspace), workspace != nullptr ? workspace_bytes : 0, &nl);
  ctx_add_launches(c, nl);
  return r;
}

kvr_status kvr_linear_swiglu(kvr_ctx* c, int T, int I, int K, const void* x, const void* w_gate_up, void* a,
                             void* workspace, size_t workspace_bytes, kvr_stream stream) {
  if (!c) return fail(KVR_ERR_INVALID_ARG, "null ctx");
  if (T < 0) return fail(KVR_ERR_INVALID_ARG, "T must be >= 0");
  if (workspace != nullptr && !al16(workspace)) return fail(KVR_ERR_INVALID_ARG, "workspace must be 16-byte aligned");
  const Proj p{w_gate_up, a, I};
  int nl = 0;
  kvr_status r = tc_linear(T, K, x, &p, 1, nullptr, true, ctx_err(c), reinterpret_cast<cudaStream_t>(stream),
                           static_cast<float*>(workspace), workspace != nullptr ? workspace_bytes : 0, &nl);
  ctx_add_launches(c, nl);
  return r;
}

}  // extern "C"
