// Joint GEMM with the fused selection epilogue, CUDA-core version.
//
// logits[r][v] = sum_k A[r][k] * Wt[v][k]  (bf16 inputs, fp32 accumulation;
// the joint network's output projection), then per row and 128-label tile:
// the softmax partial (max logit, sum exp(logit - max)) over the V+1 real
// labels and the best fused value logit + bias (bias = lambda*LM +
// beta*boost, 0 for blank), ties to the lowest label.  With DecView::fused
// the fused value is logit + D[v] + lambda*dense0[u][v] (the call's defaults
// and the dense LM row of the row's unigram state u), and the labels on the
// row's correction list are no candidates: their raw logits are stored for
// the row pass.  With fusion_path 0 (DecView::fz_dense = 0) the row's logits
// plus the call's defaults are written out instead and the row pass fuses.
// This is the simple reference-grade kernel for small row counts; the
// tensor-core kernel in joint_tc.cu does the same contraction with tcgen05.
#include "decoder.h"

namespace tsd {

namespace {

constexpr int kJM = 64, kJN = 128, kJK = 32;
constexpr float kNegInf = -__builtin_huge_valf();

__device__ __forceinline__ void bf16x8_to_f32(uint4 v, float* f) {
  const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    float2 x = __bfloat1622float2(h[q]);
    f[2 * q] = x.x;
    f[2 * q + 1] = x.y;
  }
}

__global__ void __launch_bounds__(256) k_joint_simt(DecView d, int step) {
  const int n0 = blockIdx.x * kJN, m0 = blockIdx.y * kJM;
  const int M = d.params->n * d.K;
  if (m0 >= M) return;
  const int H = d.H;
  // launched without programmatic overlap; the wait is then a no-op
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  __shared__ __align__(16) float sm[kJM * (kJN + 4)];
  float* As = sm;                      // [kJK][kJM + 4]
  float* Bs = sm + kJK * (kJM + 4);    // [kJK][kJN + 4]
  const int tid = threadIdx.x, ty = tid >> 4, tx = tid & 15;
  float acc[4][8];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[i][j] = 0.f;

  for (int k0 = 0; k0 < H; k0 += kJK) {
    {
      int row = tid >> 2, kq = (tid & 3) * 8;
      uint4 v = *reinterpret_cast<const uint4*>(d.A + (size_t)(m0 + row) * H + k0 + kq);
      float f[8];
      bf16x8_to_f32(v, f);
#pragma unroll
      for (int i = 0; i < 8; ++i) As[(kq + i) * (kJM + 4) + row] = f[i];
    }
#pragma unroll
    for (int q = 0; q < 2; ++q) {
      int idx = tid + q * 256;
      int col = idx >> 2, kq = (idx & 3) * 8;
      uint4 v = __ldg(reinterpret_cast<const uint4*>(d.Wt + (size_t)(n0 + col) * H + k0 + kq));
      float f[8];
      bf16x8_to_f32(v, f);
#pragma unroll
      for (int i = 0; i < 8; ++i) Bs[(kq + i) * (kJN + 4) + col] = f[i];
    }
    __syncthreads();
#pragma unroll 4
    for (int kk = 0; kk < kJK; ++kk) {
      float a[4], b[8];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = As[kk * (kJM + 4) + ty * 4 + i];
#pragma unroll
      for (int j = 0; j < 8; ++j) b[j] = Bs[kk * (kJN + 4) + tx * 8 + j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
  float* tile = sm;  // [kJM][kJN + 4]
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 8; ++j) tile[(ty * 4 + i) * (kJN + 4) + tx * 8 + j] = acc[i][j];
  __syncthreads();

  const int lane = tid & 31, warp = tid >> 5;
  const int N = d.N, V = d.V;
  for (int rr = 0; rr < kJM / 8; ++rr) {
    const int row = warp * (kJM / 8) + rr;
    const int gr = m0 + row;
    if (gr >= M) break;
    const float* brow = d.bias + (size_t)gr * d.N_pad;
    const float* urow = nullptr;
    const uint32_t* mrow = nullptr;
    const float lam = d.params->lambda;
    const bool dense = d.fused && d.fz_dense;
    if (dense) {
      const int u = __ldcg(&d.c_info[gr].x);
      if (u >= 0 && u < d.lm.n_dense) urow = d.lm.dense0 + (size_t)u * d.V4;
      mrow = d.c_mask + (size_t)gr * d.mask_words;
    }
    float l[4];
    float mx = kNegInf, bv = kNegInf;
    int bi = INT_MAX;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int c = lane * 4 + q, gc = n0 + c;
      l[q] = tile[row * (kJN + 4) + c];
      if (gc < N) {
        mx = fmaxf(mx, l[q]);
        float f;
        if (d.fused && !dense) {
          f = l[q];  // the streaming form: the row pass takes the argmax
        } else if (dense) {
          if ((__ldcg(mrow + (gc >> 5)) >> (gc & 31)) & 1u) {  // listed: the row pass evaluates it
            d.logits[(size_t)gr * d.N_pad + gc] = l[q];
            continue;
          }
          f = l[q] + fmaf(lam, (urow && gc < V) ? __ldg(urow + gc) : 0.f, __ldcg(d.dvec + gc));
        } else {
          f = l[q] + (gc < V ? brow[gc] : 0.f);
        }
        if (f > bv) { bv = f; bi = gc; }
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
      float v2 = __shfl_xor_sync(0xffffffffu, bv, o);
      int i2 = __shfl_xor_sync(0xffffffffu, bi, o);
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
    if (lane == 0)
      d.part[(size_t)gr * d.n_ptiles + blockIdx.x] = make_float4(mx, se, bv, __int_as_float(bi));
    if (d.fused && !dense) {  // the streaming form: logit + D of every label
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int gc = n0 + lane * 4 + q;
        d.logits[(size_t)gr * d.N_pad + gc] = l[q] + __ldcg(d.dvec + gc);
      }
    }
    if (d.cap_logits && step < d.cap_steps) {
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int gc = n0 + lane * 4 + q;
        if (gc < N) d.cap_logits[((size_t)step * M + gr) * N + gc] = l[q];
      }
    }
  }
}

}  // namespace

void launch_joint(const DecView& d, int M, int step, cudaStream_t s) {
  dim3 grid(d.N_pad / kJN, (M + kJM - 1) / kJM);
  k_joint_simt<<<grid, 256, 0, s>>>(d, step);
}

}  // namespace tsd
