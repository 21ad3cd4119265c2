// kvr_layer.cu -- a whole Qwen3-style decoder layer around the hot path, so
// that the whole-layer costs of prefill and of a reuse step can be measured
// (the paper's Table 1 times whole-model forwards; Sec. 5).
//
//   x  = RMSNorm(h)                      rmsnorm_rows_kernel
//   q, k, v = x Wq^T, x Wk^T, x Wv^T     bf16 GEMMs, fp32 accumulation (cuBLASLt; up to
//                                        8 rows gemv_kernel, bound by the weight read)
//   o  = attention(...)                  kvr_append_kv + kvr_prefill_attn, or
//                                        kvr_decode_step (reuse path)
//   h1 = h + o Wo^T                      GEMM, residual in the epilogue
//   x2 = RMSNorm(h1)                     rmsnorm_rows_kernel
//   gu = x2 [Wg; Wu]^T                   GEMM
//   a  = silu(g) * u                     swiglu_kernel
//   h_out = h1 + a Wd^T                  GEMM, residual in the epilogue
//
// Every tensor between two operations is bf16 (the model runs in bf16); each
// operation computes in fp32 and rounds once.  The norms and SwiGLU are
// memory-bound streams (16-byte accesses, one row per CTA for the norm); the
// projections are plain library GEMMs, except for a few rows (a decode step),
// where this library's weight-streaming gemv_kernel reads each weight once.
#include <cublasLt.h>

#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <map>
#include <mutex>
#include <tuple>

#include "kvr_internal.h"
#include "kvr_ptx.cuh"

namespace kvr {

// Defined in kvr_api.cu.
const kvr_model_desc* ctx_desc(const kvr_ctx* c);
void ctx_add_launches(kvr_ctx* c, int n);
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
constexpr size_t kGemmWorkspace = size_t(32) << 20;
constexpr size_t kAlignWs = 256;

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

__device__ __forceinline__ float silu_mul(float g, float u) { return g / (1.0f + expf(-g)) * u; }

// a[t][i] = bf16(silu(gu[t][i]) * gu[t][I + i]); 8 outputs per thread, I % 8 == 0.
__global__ void __launch_bounds__(256) swiglu_kernel(const uint16_t* __restrict__ gu, uint16_t* __restrict__ a,
                                                     int T, int I) {
  griddep_wait();
  griddep_launch_dependents();
  const int per_row = I / 8;
  const int64_t total = static_cast<int64_t>(T) * per_row;
  for (int64_t e = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; e < total;
       e += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t t = e / per_row;
    const int c = static_cast<int>(e % per_row) * 8;
    const uint4 g = *reinterpret_cast<const uint4*>(gu + t * 2 * I + c);
    const uint4 u = *reinterpret_cast<const uint4*>(gu + t * 2 * I + I + c);
    const uint32_t gw[4] = {g.x, g.y, g.z, g.w}, uw[4] = {u.x, u.y, u.z, u.w};
    uint32_t o[4];
#pragma unroll
    for (int j = 0; j < 4; ++j)
      o[j] = pack_bf16x2(silu_mul(bf16_lo(gw[j]), bf16_lo(uw[j])), silu_mul(bf16_hi(gw[j]), bf16_hi(uw[j])));
    *reinterpret_cast<uint4*>(a + t * I + c) = make_uint4(o[0], o[1], o[2], o[3]);
  }
}

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
  griddep_wait();
  griddep_launch_dependents();
  const int lane = threadIdx.x & 31;
  const int n = blockIdx.x * kGemvWarps + (threadIdx.x >> 5);
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
// of the residual stream, or SwiGLU of the gate/up rows: the arithmetic of
// rmsnorm_rows_kernel / swiglu_kernel) and then the projection as above, over
// up to three weight matrices that share that input (q, k, v).  A decode
// step's layer is then five launches instead of ten.
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
  griddep_wait();
  griddep_launch_dependents();
  const int T = g.T, K = g.K, nv = K / 8;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
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
  int n = blockIdx.x * kGemvWarps + warp, s = 0;
  while (s < g.nseg && n >= g.seg[s].N) n -= g.seg[s++].N;
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
  static size_t configured = 0;
  if (smem > 48 * 1024 && smem > configured) {
    const cudaError_t e =
        cudaFuncSetAttribute(gemv_pro_kernel<TM, PRO>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    configured = smem;
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

// ---- cuBLASLt: D[T][N] = X[T][K] W[N][K]^T (+ C[T][N]) in bf16 ----
// Column-major view: D^T [N x T] = op(W_colmajor [K x N])^T * X^T [K x T].
struct GemmPlan {
  cublasLtMatmulDesc_t op = nullptr;
  cublasLtMatrixLayout_t a = nullptr, b = nullptr, c = nullptr;
  cublasLtMatmulAlgo_t algo{};
};

std::mutex g_lt_mu;
cublasLtHandle_t g_lt[64] = {};
std::map<std::tuple<int, int, int, int, int>, GemmPlan> g_plans;  // (device, N, T, K, residual)

cublasLtHandle_t lt_handle(int dev) {
  if (dev < 0 || dev >= 64) return nullptr;
  if (!g_lt[dev] && cublasLtCreate(&g_lt[dev]) != CUBLAS_STATUS_SUCCESS) g_lt[dev] = nullptr;
  return g_lt[dev];
}

kvr_status gemm(int dev, int N, int T, int K, const void* W, const void* X, const void* C, void* D, void* ws,
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
  std::lock_guard<std::mutex> lock(g_lt_mu);
  cublasLtHandle_t h = lt_handle(dev);
  if (!h) return fail(KVR_ERR_CUDA, "cublasLtCreate failed");
  const auto key = std::make_tuple(dev, N, T, K, C != nullptr ? 1 : 0);
  auto it = g_plans.find(key);
  if (it == g_plans.end()) {
    GemmPlan p;
    const cublasOperation_t ta = CUBLAS_OP_T, tb = CUBLAS_OP_N;
    bool ok = cublasLtMatmulDescCreate(&p.op, CUBLAS_COMPUTE_32F, CUDA_R_32F) == CUBLAS_STATUS_SUCCESS &&
              cublasLtMatmulDescSetAttribute(p.op, CUBLASLT_MATMUL_DESC_TRANSA, &ta, sizeof(ta)) ==
                  CUBLAS_STATUS_SUCCESS &&
              cublasLtMatmulDescSetAttribute(p.op, CUBLASLT_MATMUL_DESC_TRANSB, &tb, sizeof(tb)) ==
                  CUBLAS_STATUS_SUCCESS &&
              cublasLtMatrixLayoutCreate(&p.a, CUDA_R_16BF, K, N, K) == CUBLAS_STATUS_SUCCESS &&
              cublasLtMatrixLayoutCreate(&p.b, CUDA_R_16BF, K, T, K) == CUBLAS_STATUS_SUCCESS &&
              cublasLtMatrixLayoutCreate(&p.c, CUDA_R_16BF, N, T, N) == CUBLAS_STATUS_SUCCESS;
    cublasLtMatmulPreference_t pref = nullptr;
    cublasLtMatmulHeuristicResult_t res{};
    int found = 0;
    const size_t wsb = kGemmWorkspace;
    ok = ok && cublasLtMatmulPreferenceCreate(&pref) == CUBLAS_STATUS_SUCCESS &&
         cublasLtMatmulPreferenceSetAttribute(pref, CUBLASLT_MATMUL_PREF_MAX_WORKSPACE_BYTES, &wsb, sizeof(wsb)) ==
             CUBLAS_STATUS_SUCCESS &&
         cublasLtMatmulAlgoGetHeuristic(h, p.op, p.a, p.b, p.c, p.c, pref, 1, &res, &found) ==
             CUBLAS_STATUS_SUCCESS &&
         found > 0;
    if (pref) cublasLtMatmulPreferenceDestroy(pref);
    if (!ok) {
      if (p.op) cublasLtMatmulDescDestroy(p.op);
      if (p.a) cublasLtMatrixLayoutDestroy(p.a);
      if (p.b) cublasLtMatrixLayoutDestroy(p.b);
      if (p.c) cublasLtMatrixLayoutDestroy(p.c);
      return fail(KVR_ERR_CUDA, "no cuBLASLt bf16 GEMM for N=%d T=%d K=%d", N, T, K);
    }
    p.algo = res.algo;
    it = g_plans.emplace(key, p).first;
  }
  const GemmPlan& p = it->second;
  const float alpha = 1.0f, beta = C != nullptr ? 1.0f : 0.0f;
  const cublasStatus_t s = cublasLtMatmul(h, p.op, &alpha, W, p.a, X, p.b, &beta, C != nullptr ? C : D, p.c, D, p.c,
                                          &p.algo, ws, kGemmWorkspace, st);
  if (s != CUBLAS_STATUS_SUCCESS) return fail(KVR_ERR_CUDA, "cublasLtMatmul failed: %d", static_cast<int>(s));
  return KVR_OK;
}

// Workspace regions for T tokens.
struct LayerWs {
  char* gemm;
  uint16_t *x, *q, *k, *v, *qr, *o, *h1, *x2, *gu, *a;
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
  w.gemm = base;
  off = align_ws(kGemmWorkspace);
  const size_t qd = static_cast<size_t>(d.n_q_heads) * d.head_dim, kd = static_cast<size_t>(d.n_kv_heads) * d.head_dim;
  w.x = take(T * l.hidden);
  w.q = take(T * qd);
  w.k = take(T * kd);
  w.v = take(T * kd);
  w.qr = take(T * qd);
  w.o = take(T * qd);
  w.h1 = take(T * l.hidden);
  w.x2 = take(T * l.hidden);
  w.gu = take(T * 2 * static_cast<size_t>(l.intermediate));
  w.a = take(T * static_cast<size_t>(l.intermediate));
  w.bytes = off;
  return w;
}

bool ldesc_ok(const kvr_layer_desc* l) {
  return l && l->hidden > 0 && l->intermediate > 0 && l->hidden % 8 == 0 && l->intermediate % 8 == 0;
}

bool al16(const void* p) { return p && (reinterpret_cast<uintptr_t>(p) & 15) == 0; }

}  // namespace
}  // namespace kvr

using namespace kvr;

extern "C" {

size_t kvr_layer_workspace_bytes(const kvr_model_desc* desc, const kvr_layer_desc* ldesc, uint32_t max_tokens) {
  if (!desc || !ldesc_ok(ldesc) || kvr_artifact_bytes(desc, 1) == 0) return 0;
  return carve(nullptr, *desc, *ldesc, max_tokens).bytes;
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
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return fail(KVR_ERR_CUDA, "cudaGetDevice failed");
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
    if ((r = gemm(dev, H, T, qd, w->wo, ws.o, hin, ws.h1, ws.gemm, st)) != KVR_OK) return r;
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
  if ((r = gemm(dev, qd, T, H, w->wq, ws.x, nullptr, ws.q, ws.gemm, st)) != KVR_OK) return r;
  if ((r = gemm(dev, kd, T, H, w->wk, ws.x, nullptr, ws.k, ws.gemm, st)) != KVR_OK) return r;
  if ((r = gemm(dev, kd, T, H, w->wv, ws.x, nullptr, ws.v, ws.gemm, st)) != KVR_OK) return r;
  if (n_seqs == 1 && start_pos[0] == 0) {
    r = kvr_append_kv(c, layer, 1, seqs, start_pos, cu_q, ws.q, ws.k, ws.v, w->q_norm, w->k_norm, ws.qr, stream);
    if (r == KVR_OK) r = kvr_prefill_attn(c, layer, seqs[0], T, ws.qr, ws.o, nullptr, nullptr, stream);
  } else {
    r = kvr_decode_step(c, layer, n_seqs, seqs, start_pos, cu_q, ws.q, ws.k, ws.v, w->q_norm, w->k_norm, ws.qr,
                        ws.o, nullptr, nullptr, stream);
  }
  if (r != KVR_OK) return r;
  if ((r = gemm(dev, H, T, qd, w->wo, ws.o, hin, ws.h1, ws.gemm, st)) != KVR_OK) return r;
  e = launch_kernel(rmsnorm_rows_kernel, dim3(T), dim3(kNormThreads), 0, st, 0, static_cast<const uint16_t*>(ws.h1),
                    static_cast<const uint16_t*>(w->post_norm), ws.x2, H, eps);
  if (e != cudaSuccess) return fail(KVR_ERR_CUDA, "rmsnorm launch: %s", cudaGetErrorString(e));
  if ((r = gemm(dev, 2 * I, T, H, w->w_gate_up, ws.x2, nullptr, ws.gu, ws.gemm, st)) != KVR_OK) return r;
  const int64_t vec = static_cast<int64_t>(T) * (I / 8);
  const int blocks = static_cast<int>(std::min<int64_t>((vec + 255) / 256, 152 * 16));
  e = launch_kernel(swiglu_kernel, dim3(blocks), dim3(256), 0, st, 0, static_cast<const uint16_t*>(ws.gu), ws.a, T, I);
  if (e != cudaSuccess) return fail(KVR_ERR_CUDA, "swiglu launch: %s", cudaGetErrorString(e));
  ctx_add_launches(c, 3);  // the two norms and SwiGLU (the GEMMs are cuBLASLt's)
  return gemm(dev, H, T, I, w->w_down, ws.a, ws.h1, hout, ws.gemm, st);
}

}  // extern "C"
