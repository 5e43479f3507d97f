// An allocation-free variant of the joint GEMM + fused selection for one
// label step, for callers that cannot allocate device memory.
//
// Some callers cannot call cudaMalloc at the time they decode: code running
// inside a memory pool or arena that owns every byte of the device, plugins
// that are handed pre-allocated buffers by their host framework, or
// real-time paths where an allocation's implicit synchronization and
// unbounded latency are not acceptable.  tsd_joint_select_noalloc serves
// them: the caller passes only inputs and outputs, and the one piece of
// working memory the computation needs -- the per-(row, label tile)
// selection partials -- lives in a fixed file-scope __device__ array that is
// part of the loaded library image (so every GPU that loads the library
// holds it until the process exits).
//
// The per-row work is the CUDA-core joint kernel's: logits = A . Wt^T in
// fp32 from bf16, the softmax partial over the V+1 labels and the best fused
// value logit + bias (bias 0 for blank), then a combine over the tiles.
#include <mutex>

#include "decoder.h"

namespace tsd {

namespace {

// Limits of the static working array (1 MiB of float4 partials).
constexpr int kNaRows = 1024;          // rows per call
constexpr int kNaCols = 128;           // labels per partial
constexpr int kNaMaxN = 8192;          // V + 1 per call
constexpr int kNaTiles = kNaMaxN / kNaCols;
constexpr int kJM = 64, kJK = 32;
constexpr float kNegInf = -__builtin_huge_valf();

static __device__ __align__(256) float4 g_na_part[kNaRows * kNaTiles];

__device__ __forceinline__ void unpack8(uint4 v, float* f) {
  const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    float2 x = __bfloat1622float2(h[q]);
    f[2 * q] = x.x;
    f[2 * q + 1] = x.y;
  }
}

// One 64-row x 128-label tile: fp32 product, then per row the tile's
// (max logit, sum exp(logit - max), best fused value, best label).
__global__ void __launch_bounds__(256) k_na_tile(int n, int H, int V, const uint16_t* __restrict__ A,
                                                 const uint16_t* __restrict__ Wt, const float* __restrict__ bias,
                                                 float4* __restrict__ part) {
  const int n0 = blockIdx.x * kNaCols, m0 = blockIdx.y * kJM;
  const int N = V + 1;
  __shared__ __align__(16) float sm[kJM * (kNaCols + 4)];
  float* As = sm;
  float* Bs = sm + kJK * (kJM + 4);
  const int tid = threadIdx.x, ty = tid >> 4, tx = tid & 15;
  float acc[4][8];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[i][j] = 0.f;
  for (int k0 = 0; k0 < H; k0 += kJK) {
    {
      const int row = tid >> 2, kq = (tid & 3) * 8;
      float f[8];
      if (m0 + row < n) {
        unpack8(__ldg(reinterpret_cast<const uint4*>(A + (size_t)(m0 + row) * H + k0 + kq)), f);
      } else {
#pragma unroll
        for (int i = 0; i < 8; ++i) f[i] = 0.f;
      }
#pragma unroll
      for (int i = 0; i < 8; ++i) As[(kq + i) * (kJM + 4) + row] = f[i];
    }
#pragma unroll
    for (int q = 0; q < 2; ++q) {
      const int idx = tid + q * 256;
      const int col = idx >> 2, kq = (idx & 3) * 8;
      float f[8];
      if (n0 + col < N) {
        unpack8(__ldg(reinterpret_cast<const uint4*>(Wt + (size_t)(n0 + col) * H + k0 + kq)), f);
      } else {
#pragma unroll
        for (int i = 0; i < 8; ++i) f[i] = 0.f;
      }
#pragma unroll
      for (int i = 0; i < 8; ++i) Bs[(kq + i) * (kNaCols + 4) + col] = f[i];
    }
    __syncthreads();
#pragma unroll 4
    for (int kk = 0; kk < kJK; ++kk) {
      float a[4], b[8];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = As[kk * (kJM + 4) + ty * 4 + i];
#pragma unroll
      for (int j = 0; j < 8; ++j) b[j] = Bs[kk * (kNaCols + 4) + tx * 8 + j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
  float* tile = sm;
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 8; ++j) tile[(ty * 4 + i) * (kNaCols + 4) + tx * 8 + j] = acc[i][j];
  __syncthreads();
  const int lane = tid & 31, warp = tid >> 5;
  for (int rr = 0; rr < kJM / 8; ++rr) {
    const int row = warp * (kJM / 8) + rr;
    const int gr = m0 + row;
    if (gr >= n) break;
    float l[4], mx = kNegInf, bv = kNegInf;
    int bi = INT_MAX;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int gc = n0 + lane * 4 + q;
      l[q] = tile[row * (kNaCols + 4) + lane * 4 + q];
      if (gc < N) {
        mx = fmaxf(mx, l[q]);
        const float f = l[q] + ((gc < V && bias) ? __ldg(bias + (size_t)gr * V + gc) : 0.f);
        if (f > bv) { bv = f; bi = gc; }
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
      const float v2 = __shfl_xor_sync(0xffffffffu, bv, o);
      const int i2 = __shfl_xor_sync(0xffffffffu, bi, o);
      if (v2 > bv || (v2 == bv && i2 < bi)) { bv = v2; bi = i2; }
    }
    float se = 0.f;
    if (mx != kNegInf) {
#pragma unroll
      for (int q = 0; q < 4; ++q)
        if (n0 + lane * 4 + q < N) se += expf(l[q] - mx);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) se += __shfl_xor_sync(0xffffffffu, se, o);
    if (lane == 0) part[(size_t)gr * kNaTiles + blockIdx.x] = make_float4(mx, se, bv, __int_as_float(bi));
  }
}

// One warp per row: log-sum-exp over the tiles, best label and its fused
// score (fused value minus the log-sum-exp).
__global__ void k_na_combine(int n, int tiles, int V, const float4* __restrict__ part, int32_t* __restrict__ label,
                             float* __restrict__ score) {
  const int r = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (r >= n) return;
  float m = kNegInf, s = 0.f, bv = kNegInf;
  int bi = INT_MAX;
  for (int j = lane; j < tiles; j += 32) {
    const float4 p = part[(size_t)r * kNaTiles + j];
    if (p.x != kNegInf) {
      if (m == kNegInf) { m = p.x; s = p.y; }
      else { const float mx = fmaxf(m, p.x); s = s * expf(m - mx) + p.y * expf(p.x - mx); m = mx; }
    }
    const int pi = __float_as_int(p.w);
    if (p.z > bv || (p.z == bv && pi < bi)) { bv = p.z; bi = pi; }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m, o), s2 = __shfl_xor_sync(0xffffffffu, s, o);
    const float v2 = __shfl_xor_sync(0xffffffffu, bv, o);
    const int i2 = __shfl_xor_sync(0xffffffffu, bi, o);
    if (m2 != kNegInf) {
      if (m == kNegInf) { m = m2; s = s2; }
      else { const float mx = fmaxf(m, m2); s = s * expf(m - mx) + s2 * expf(m2 - mx); m = mx; }
    }
    if (v2 > bv || (v2 == bv && i2 < bi)) { bv = v2; bi = i2; }
  }
  if (lane == 0) {
    label[r] = (bi >= 0 && bi <= V) ? bi : V;
    score[r] = bv - (m + logf(s));
  }
}

// Device address of the static array, resolved once per device.
std::mutex g_na_mu;
float4* g_na_ptr[64] = {};

}  // namespace

}  // namespace tsd

using namespace tsd;

extern "C" tsd_status tsd_joint_select_noalloc(int32_t n, int32_t H, int32_t V, const void* A_bf16,
                                               const void* Wt_bf16, const float* bias, int32_t* out_label,
                                               float* out_score, void* cuda_stream) {
  clear_error();
  if (!A_bf16 || !Wt_bf16 || !out_label || !out_score)
    return fail(TSD_EINVAL, "tsd_joint_select_noalloc: NULL argument");
  if (n < 1 || n > kNaRows) return fail(TSD_EINVAL, "tsd_joint_select_noalloc: n=%d outside [1, %d]", n, kNaRows);
  if (V < 1 || V + 1 > kNaMaxN)
    return fail(TSD_EINVAL, "tsd_joint_select_noalloc: V+1=%d outside [2, %d]", V + 1, kNaMaxN);
  if (H < 64 || H > 8192 || H % 64) return fail(TSD_EINVAL, "tsd_joint_select_noalloc: H=%d must be a multiple of 64 in [64, 8192]", H);
  int dev = -1;
  TSD_CUDA(cudaGetDevice(&dev));
  if (dev < 0 || dev >= 64) return fail(TSD_EINVAL, "tsd_joint_select_noalloc: device %d unsupported", dev);
  float4* part = nullptr;
  {
    std::lock_guard<std::mutex> lk(g_na_mu);
    if (!g_na_ptr[dev]) {
      // first call on this device: host code must ask the runtime for the
      // array's device address (its name in host code is only a stand-in)
      void* p = nullptr;
      cudaError_t e = cudaGetSymbolAddress(&p, g_na_part);
      if (e != cudaSuccess) return cuda_fail(e, "tsd_joint_select_noalloc: cudaGetSymbolAddress");
      g_na_ptr[dev] = static_cast<float4*>(p);
    }
    part = g_na_ptr[dev];
  }
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  const int tiles = (V + 1 + kNaCols - 1) / kNaCols;
  k_na_tile<<<dim3(tiles, (n + kJM - 1) / kJM), 256, 0, s>>>(n, H, V, static_cast<const uint16_t*>(A_bf16),
                                                             static_cast<const uint16_t*>(Wt_bf16), bias, part);
  k_na_combine<<<(n + 7) / 8, 256, 0, s>>>(n, tiles, V, part, out_label, out_score);
  TSD_CUDA(cudaGetLastError());
  return TSD_OK;
}
