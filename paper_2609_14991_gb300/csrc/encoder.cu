// The cache-aware encoder chunk step (Sec. III-B: chunked, limited-context
// attention, causal convolutions and a cache carried across chunks; Sec.
// IV-A: 80 ms encoder frames, look-ahead = the chunk): host driver and the
// kernels that are not GEMMs.  See tsd.h for the computation.
//
// Per chunk of n streams x C frames (M = n C rows, row b C + t = frame t of
// the call's stream b), one CUDA graph runs: the subsampling GEMM into the
// fp32 residual stream x, then per block 15 launches (layer norms, the
// tensor-core GEMMs of encoder_gemm.cu with their fused epilogues, the
// attention kernel, the depthwise convolution), then a kernel that advances
// every stream's frame count.  Caches live per slot in device memory:
// k and v of the last `left` frames per block and head in a ring indexed by
// frame position mod left, and the last K-1 GLU outputs per block.
#include <cuda.h>
#include <cuda_bf16.h>

#include <algorithm>
#include <cmath>
#include <cstring>
#include <memory>

#include "encoder.h"

namespace tsd {

namespace {

constexpr float kLnEps = 1e-5f;

__device__ __forceinline__ uint16_t f2bf(float v) {
  const __nv_bfloat16 b = __float2bfloat16_rn(v);
  return *reinterpret_cast<const uint16_t*>(&b);
}
__device__ __forceinline__ float bf2f(uint16_t u) { return __uint_as_float((uint32_t)u << 16); }

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// v := LN(v) * g + b over a row held by one warp (lane j holds the float4
// groups j, j + 32, ..; nq groups per lane): mean, then the variance about
// it, in fp32.
template <int kMaxQ>
__device__ __forceinline__ void ln_regs(float4 (&v)[kMaxQ], int nq, int d, int lane, const float* g, const float* b) {
  float s = 0.f;
#pragma unroll
  for (int i = 0; i < kMaxQ; ++i)
    if (i < nq) s += (v[i].x + v[i].y) + (v[i].z + v[i].w);
  const float mean = warp_sum(s) / (float)d;
  float q = 0.f;
#pragma unroll
  for (int i = 0; i < kMaxQ; ++i)
    if (i < nq) {
      const float a0 = v[i].x - mean, a1 = v[i].y - mean, a2 = v[i].z - mean, a3 = v[i].w - mean;
      q += (a0 * a0 + a1 * a1) + (a2 * a2 + a3 * a3);
    }
  const float rstd = 1.f / sqrtf(warp_sum(q) / (float)d + kLnEps);
#pragma unroll
  for (int i = 0; i < kMaxQ; ++i)
    if (i < nq) {
      const int c = 128 * i + 4 * lane;
      const float4 gg = *reinterpret_cast<const float4*>(g + c);
      const float4 be = *reinterpret_cast<const float4*>(b + c);
      v[i] = make_float4((v[i].x - mean) * rstd * gg.x + be.x, (v[i].y - mean) * rstd * gg.y + be.y,
                         (v[i].z - mean) * rstd * gg.z + be.z, (v[i].w - mean) * rstd * gg.w + be.w);
    }
}

template <int kMaxQ>
__device__ __forceinline__ void store_bf16(uint16_t* yr, const float4 (&v)[kMaxQ], int nq, int lane) {
#pragma unroll
  for (int i = 0; i < kMaxQ; ++i)
    if (i < nq) {
      uint2 w;
      w.x = (uint32_t)f2bf(v[i].x) | ((uint32_t)f2bf(v[i].y) << 16);
      w.y = (uint32_t)f2bf(v[i].z) | ((uint32_t)f2bf(v[i].w) << 16);
      *reinterpret_cast<uint2*>(yr + 128 * i + 4 * lane) = w;
    }
}

// Layer norms of rows of the fp32 stream x [M][d], one warp per row, the row
// in registers:
// FINAL = false: y = bf16(LN_1(x)) (a module's input);
// FINAL = true:  x = LN_1(x) in place (a block's closing norm), then, with
//                g2 != nullptr, y = bf16(LN_2(x)) (the next block's first
//                module input, from the same registers), else y = bf16(x)
//                when y != nullptr (the encoder's output).
template <bool FINAL, int kMaxQ>  // d <= 128 kMaxQ
__global__ void __launch_bounds__(256) k_ln(float* x, uint16_t* y, int M, int d, const float* g, const float* b,
                                            const float* g2, const float* b2) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r = blockIdx.x * 8 + warp;
  if (r >= M) return;
  float* xr = x + (size_t)r * d;
  const int nq = d / 128;  // float4 groups per lane
  float4 v[kMaxQ];
#pragma unroll
  for (int i = 0; i < kMaxQ; ++i)
    if (i < nq) v[i] = *reinterpret_cast<const float4*>(xr + 128 * i + 4 * lane);
  ln_regs<kMaxQ>(v, nq, d, lane, g, b);
  if (FINAL) {
#pragma unroll
    for (int i = 0; i < kMaxQ; ++i)
      if (i < nq) *reinterpret_cast<float4*>(xr + 128 * i + 4 * lane) = v[i];
    if (g2) ln_regs<kMaxQ>(v, nq, d, lane, g2, b2);
  }
  if (y) store_bf16<kMaxQ>(y + (size_t)r * d, v, nq, lane);
}

struct AttnArgs {
  const uint16_t* qkv;      // [M][3d] bf16: q, k, v of the chunk's frames
  uint16_t* out;            // [M][d] bf16
  const uint16_t* pos_tab;  // [n_off][d] bf16: this block's W_pos r(delta), row delta + cmax - 1
  const float* pu;          // [d] content bias u
  const float* pv;          // [d] position bias v
  uint16_t* kc;             // k cache: [slot][layer][head][left][dh]
  uint16_t* vc;
  const int32_t* seen;      // frames seen per slot (before this chunk)
  const int32_t* slots;     // [n]
  int d, heads, left, layers, layer, C, cmax;
  float scale;              // 1 / sqrt(dh)
};

__host__ __device__ constexpr int round16(int x) { return (x + 15) / 16 * 16; }

// Shared memory of k_attn for a chunk of C frames (worst case nv = left):
// q + u and q + v, k, v and the table rows as bf16 rows padded by 8 elements
// (16-byte aligned, conflict-free ldmatrix), then one 16-row block's scores,
// position scores (fp32) and probabilities (bf16).
__host__ __device__ constexpr size_t attn_smem(int dh, int left, int C) {
  return (size_t)2 * round16(C) * (dh + 8) * 2 + (size_t)2 * round16(left + C) * (dh + 8) * 2 +
         (size_t)round16(left + 2 * C - 1) * (dh + 8) * 2 + (size_t)16 * (round16(left + C) + 4) * 4 +
         (size_t)16 * (round16(left + 2 * C - 1) + 4) * 4 + (size_t)16 * (round16(left + C) + 8) * 2;
}

__device__ __forceinline__ void ldsm_x4(const void* p, uint32_t* r) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"((uint32_t)__cvta_generic_to_shared(p)));
}
__device__ __forceinline__ void ldsm_x2(const void* p, uint32_t* r) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x2.shared.b16 {%0, %1}, [%2];"
               : "=r"(r[0]), "=r"(r[1])
               : "r"((uint32_t)__cvta_generic_to_shared(p)));
}
__device__ __forceinline__ void ldsm_x2_trans(const void* p, uint32_t* r) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x2.trans.shared.b16 {%0, %1}, [%2];"
               : "=r"(r[0]), "=r"(r[1])
               : "r"((uint32_t)__cvta_generic_to_shared(p)));
}
// 16-byte global -> shared copy that completes asynchronously (waited for
// with cp.async.wait_group); both addresses 16-byte aligned.
__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"((uint32_t)__cvta_generic_to_shared(dst)), "l"(src)
               : "memory");
}
// D (16x8 fp32) += A (16x16 bf16, row-major) . B (16x8 bf16, column-major)
__device__ __forceinline__ void mma16816(float* c, const uint32_t* a, const uint32_t* b) {
  asm volatile("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
               "{%0, %1, %2, %3};"
               : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
               : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b[0]), "r"(b[1]));
}

// One (stream, head) per CTA, 16 warps: chunked, limited-context attention
// with the relative-position term over the window [cached frames, chunk
// frames].  The three products -- (q + u) against the keys, (q + v)
// against the position-table rows, the probabilities against the values --
// run on the tensor cores as 16 x 8 x 16 bf16 MMAs with fp32 accumulation
// (a chunk has 13 query rows: one 16-row tile).  Then the chunk's k and v go
// into the ring cache.
constexpr int kAttnThreads = 512;

template <int DH>
__global__ void __launch_bounds__(kAttnThreads) k_attn(AttnArgs a) {
  extern __shared__ __align__(16) unsigned char sm[];
  constexpr int RS = DH + 8;  // bf16 row stride
  constexpr int E8 = DH / 8;  // 16-byte groups per row
  const int b = blockIdx.x, h = blockIdx.y, tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int C = a.C, d = a.d;
  const int slot = a.slots[b];
  const int sn = a.seen[slot];
  const int nv = min(sn, a.left);
  const int W = nv + C;
  const int nrel = nv + 2 * C - 1;  // offsets -(C-1) .. nv+C-1
  const int CR = round16(C), Wp = round16(a.left + C), Np = round16(a.left + 2 * C - 1);
  const int Wa = round16(W), Na = round16(nrel);  // this stream's padded extents
  const int SS = Wp + 4, SPS = Np + 4, PRS = Wp + 8;
  uint16_t* Qu = reinterpret_cast<uint16_t*>(sm);
  uint16_t* Qv = Qu + CR * RS;
  uint16_t* Kb = Qv + CR * RS;
  uint16_t* Vb = Kb + Wp * RS;
  uint16_t* Pb = Vb + Wp * RS;
  float* S = reinterpret_cast<float*>(Pb + Np * RS);  // [16][SS]
  float* Sp = S + 16 * SS;                             // [16][SPS]
  uint16_t* Pr = reinterpret_cast<uint16_t*>(Sp + 16 * SPS);  // [16][PRS]

  const size_t cb = (((size_t)slot * a.layers + a.layer) * a.heads + h) * (size_t)a.left * DH;
  const uint4 zero = make_uint4(0u, 0u, 0u, 0u);
  // keys, values and table rows go global -> shared with asynchronous 16-byte
  // copies (all of a thread's copies in flight at once); padding rows are
  // zeroed with plain stores
  for (int idx = tid; idx < Wa * E8; idx += blockDim.x) {
    const int jj = idx / E8, e8 = idx - jj * E8;
    uint16_t* kd = Kb + jj * RS + 8 * e8;
    uint16_t* vd = Vb + jj * RS + 8 * e8;
    if (jj < nv) {
      const int ring = (sn - nv + jj) % a.left;
      cp_async16(kd, a.kc + cb + (size_t)ring * DH + 8 * e8);
      cp_async16(vd, a.vc + cb + (size_t)ring * DH + 8 * e8);
    } else if (jj < W) {
      const uint16_t* row = a.qkv + (size_t)(b * C + jj - nv) * 3 * d + h * DH + 8 * e8;
      cp_async16(kd, row + d);
      cp_async16(vd, row + 2 * d);
    } else {
      *reinterpret_cast<uint4*>(kd) = zero;
      *reinterpret_cast<uint4*>(vd) = zero;
    }
  }
  for (int idx = tid; idx < Na * E8; idx += blockDim.x) {
    const int t = idx / E8, e8 = idx - t * E8;
    uint16_t* pd = Pb + t * RS + 8 * e8;
    if (t < nrel) cp_async16(pd, a.pos_tab + (size_t)(t + a.cmax - C) * d + h * DH + 8 * e8);
    else *reinterpret_cast<uint4*>(pd) = zero;
  }
  asm volatile("cp.async.commit_group;" ::: "memory");
  for (int idx = tid; idx < CR * E8; idx += blockDim.x) {
    const int i = idx / E8, e8 = idx - i * E8;
    uint4 qu = zero, qv = zero;
    if (i < C) {
      const uint4 qw = reinterpret_cast<const uint4*>(a.qkv + (size_t)(b * C + i) * 3 * d + h * DH)[e8];
      const uint32_t* qp = reinterpret_cast<const uint32_t*>(&qw);
      const float* u = a.pu + h * DH + 8 * e8;
      const float* v = a.pv + h * DH + 8 * e8;
      uint32_t* up = reinterpret_cast<uint32_t*>(&qu);
      uint32_t* vp = reinterpret_cast<uint32_t*>(&qv);
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const float q0 = __uint_as_float(qp[k] << 16), q1 = __uint_as_float(qp[k] & 0xffff0000u);
        up[k] = (uint32_t)f2bf(q0 + u[2 * k]) | ((uint32_t)f2bf(q1 + u[2 * k + 1]) << 16);
        vp[k] = (uint32_t)f2bf(q0 + v[2 * k]) | ((uint32_t)f2bf(q1 + v[2 * k + 1]) << 16);
      }
    }
    *reinterpret_cast<uint4*>(Qu + i * RS + 8 * e8) = qu;
    *reinterpret_cast<uint4*>(Qv + i * RS + 8 * e8) = qv;
  }
  asm volatile("cp.async.wait_group 0;" ::: "memory");
  __syncthreads();
  // the cache was read above: the chunk's k and v (window rows nv .. W-1 in
  // shared memory) replace the oldest frames
  if (a.left > 0) {
    for (int idx = tid; idx < C * E8; idx += blockDim.x) {
      const int i = idx / E8, e8 = idx - i * E8;
      if (i < C - a.left) continue;
      const int ring = (sn + i) % a.left;
      reinterpret_cast<uint4*>(a.kc + cb + (size_t)ring * DH)[e8] =
          *reinterpret_cast<const uint4*>(Kb + (nv + i) * RS + 8 * e8);
      reinterpret_cast<uint4*>(a.vc + cb + (size_t)ring * DH)[e8] =
          *reinterpret_cast<const uint4*>(Vb + (nv + i) * RS + 8 * e8);
    }
  }
  const int fr = lane >> 2, fc = (lane & 3) * 2;  // this lane's place in a 16 x 8 result
  for (int rb = 0; rb < CR; rb += 16) {
    // content scores S = (q + u) k^T and position scores Sp = (q + v) p^T,
    // one 16 x 8 tile per warp at a time
    const int nts = Wa / 8, ntp = Na / 8;
    for (int nt = warp; nt < nts + ntp; nt += kAttnThreads / 32) {
      const bool pos = nt >= nts;
      const int n0 = (pos ? nt - nts : nt) * 8;
      const uint16_t* A = (pos ? Qv : Qu) + (rb + (lane & 15)) * RS + (lane >> 4) * 8;
      const uint16_t* B = (pos ? Pb : Kb) + (n0 + (lane & 7)) * RS + ((lane >> 3) & 1) * 8;
      float c[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int kk = 0; kk < DH / 16; ++kk) {
        uint32_t af[4], bf[2];
        ldsm_x4(A + kk * 16, af);
        ldsm_x2(B + kk * 16, bf);
        mma16816(c, af, bf);
      }
      float* o = pos ? Sp : S;
      const int os = pos ? SPS : SS;
      *reinterpret_cast<float2*>(o + fr * os + n0 + fc) = make_float2(c[0], c[1]);
      *reinterpret_cast<float2*>(o + (fr + 8) * os + n0 + fc) = make_float2(c[2], c[3]);
    }
    __syncthreads();
    {
      // scores, softmax and bf16 probabilities: 16 threads per query row
      constexpr int G = kAttnThreads / 16;
      const int r = tid / G, l8 = tid % G, i = rb + r;
      float m = -INFINITY;
      if (i < C)
        for (int jj = l8; jj < W; jj += G) {
          const float v = (S[r * SS + jj] + Sp[r * SPS + (i - jj + nv + C - 1)]) * a.scale;
          S[r * SS + jj] = v;
          m = fmaxf(m, v);
        }
#pragma unroll
      for (int o = G / 2; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
      float z = 0.f;
      if (i < C)
        for (int jj = l8; jj < W; jj += G) {
          const float e = expf(S[r * SS + jj] - m);
          S[r * SS + jj] = e;
          z += e;
        }
#pragma unroll
      for (int o = G / 2; o > 0; o >>= 1) z += __shfl_xor_sync(0xffffffffu, z, o);
      const float inv = i < C ? 1.f / z : 0.f;
      for (int jj = l8; jj < Wa; jj += G) Pr[r * PRS + jj] = (i < C && jj < W) ? f2bf(S[r * SS + jj] * inv) : 0;
    }
    __syncthreads();
    // out = probabilities . v, one 16 x 8 tile of head columns per warp at a time
    for (int nt = warp; nt < DH / 8; nt += kAttnThreads / 32) {
      float c[4] = {0.f, 0.f, 0.f, 0.f};
      for (int kk = 0; kk < Wa / 16; ++kk) {
        uint32_t af[4], bf[2];
        ldsm_x4(Pr + (lane & 15) * PRS + kk * 16 + (lane >> 4) * 8, af);
        ldsm_x2_trans(Vb + (kk * 16 + (lane & 15)) * RS + nt * 8, bf);
        mma16816(c, af, bf);
      }
      const int i0 = rb + fr, i1 = rb + fr + 8, col = h * DH + nt * 8 + fc;
      if (i0 < C)
        *reinterpret_cast<uint32_t*>(a.out + (size_t)(b * C + i0) * d + col) =
            (uint32_t)f2bf(c[0]) | ((uint32_t)f2bf(c[1]) << 16);
      if (i1 < C)
        *reinterpret_cast<uint32_t*>(a.out + (size_t)(b * C + i1) * d + col) =
            (uint32_t)f2bf(c[2]) | ((uint32_t)f2bf(c[3]) << 16);
    }
    __syncthreads();
  }
}

struct ConvArgs {
  const uint16_t* glu;  // [M][d]
  uint16_t* z;          // [M][d]
  uint16_t* cache;      // [slot][layer][K-1][d]
  const float *w, *bias, *sc, *sh;
  const int32_t* slots;
  int d, K, C, layers, layer;
};

// Causal depthwise convolution over [cached K-1 frames, chunk frames], the
// batch-norm affine map and Swish; thread = channel.  The last K-1 frames of
// the window become the cache.  KT > 0: the kernel width as a constant, so
// the taps stay in registers.
template <int KT>
__global__ void __launch_bounds__(128) k_dwconv(ConvArgs a) {
  extern __shared__ float seq[];  // [K-1+C][128]
  const int b = blockIdx.x, c = blockIdx.y * 128 + threadIdx.x, tid = threadIdx.x;
  const int K = KT > 0 ? KT : a.K;
  const int K1 = K - 1, C = a.C, d = a.d;
  const int slot = a.slots[b];
  uint16_t* cc = a.cache + ((size_t)slot * a.layers + a.layer) * (size_t)K1 * d;
#pragma unroll 4
  for (int t = 0; t < K1; ++t) seq[t * 128 + tid] = bf2f(cc[(size_t)t * d + c]);
#pragma unroll 4
  for (int t = 0; t < C; ++t) seq[(K1 + t) * 128 + tid] = bf2f(a.glu[(size_t)(b * C + t) * d + c]);
  const float* w = a.w + (size_t)c * K;
  const float bias = a.bias[c], sc = a.sc[c], sh = a.sh[c];
  float wk[KT > 0 ? KT : 1];
  if (KT > 0) {
#pragma unroll
    for (int k = 0; k < KT; ++k) wk[k] = w[k];
  }
  for (int t = 0; t < C; ++t) {
    float acc = 0.f;
    if (KT > 0) {
#pragma unroll
      for (int k = 0; k < KT; ++k) acc = fmaf(wk[k], seq[(t + k) * 128 + tid], acc);
    } else {
      for (int k = 0; k < K; ++k) acc = fmaf(w[k], seq[(t + k) * 128 + tid], acc);
    }
    const float yv = (acc + bias) * sc + sh;
    a.z[(size_t)(b * C + t) * d + c] = f2bf(yv / (1.f + expf(-yv)));
  }
  for (int t = 0; t < K1; ++t) cc[(size_t)t * d + c] = f2bf(seq[(C + t) * 128 + tid]);
}

// P[row][c] = bf16(sum_k W_pos[c][k] r_k(delta)), delta = row - (cmax - 1), r
// the sinusoidal code (sin at 2j, cos at 2j+1 of delta / 10000^(2j/d));
// computed in double once at create and rounded once to bf16 (it is an MMA
// operand).
__global__ void k_pos_table(const uint16_t* pos_w, uint16_t* tab, int d, int cmax) {
  extern __shared__ double r[];
  const double delta = (double)((int)blockIdx.x - (cmax - 1));
  for (int k = threadIdx.x; k < d; k += blockDim.x) {
    const double w = pow(10000.0, -2.0 * (double)(k / 2) / (double)d);
    r[k] = (k & 1) ? cos(delta * w) : sin(delta * w);
  }
  __syncthreads();
  for (int c = threadIdx.x; c < d; c += blockDim.x) {
    const uint16_t* wr = pos_w + (size_t)c * d;
    double acc = 0.0;
    for (int k = 0; k < d; ++k) acc += (double)bf2f(wr[k]) * r[k];
    const __nv_bfloat16 v = __double2bfloat16(acc);
    tab[(size_t)blockIdx.x * d + c] = *reinterpret_cast<const uint16_t*>(&v);
  }
}

// W_pw1 [2d][d] -> rows interleaved in groups of 32: output group p's value
// rows, then its gate rows (the GLU epilogue finds both in one tile).
__global__ void k_glu_repack(const uint16_t* src, const float* bsrc, uint16_t* dst, float* bdst, int d) {
  const int r = blockIdx.x;  // destination row
  const int p = r / 64, w = r % 64;
  const int s = w < 32 ? 32 * p + w : d + 32 * p + (w - 32);
  for (int k = threadIdx.x; k < d; k += blockDim.x) dst[(size_t)r * d + k] = src[(size_t)s * d + k];
  if (threadIdx.x == 0) bdst[r] = bsrc[s];
}

__global__ void k_advance(int32_t* seen, const int32_t* slots, int n, int C) {
  for (int b = threadIdx.x; b < n; b += blockDim.x) seen[slots[b]] += C;
}

tsd_status set_device(tsd_encoder* e) {
  int cur = -1;
  TSD_CUDA(cudaGetDevice(&cur));
  if (cur != e->device) TSD_CUDA(cudaSetDevice(e->device));
  return TSD_OK;
}

int n_marks(const tsd_encoder* e) { return 2 + 14 * e->cfg.layers + 1 + 1; }

void launch_attn(const tsd_encoder* e, const AttnArgs& a, int n, cudaStream_t s) {
  const size_t sm = attn_smem(e->cfg.d / e->cfg.heads, e->cfg.left, a.C);
  dim3 grid(n, e->cfg.heads);
  if (e->cfg.d / e->cfg.heads == 64) k_attn<64><<<grid, kAttnThreads, sm, s>>>(a);
  else k_attn<128><<<grid, kAttnThreads, sm, s>>>(a);
}

template <bool FINAL>
void ln_launch(dim3 grid, cudaStream_t s, float* x, uint16_t* y, int M, int d, const float* g, const float* b,
               const float* g2 = nullptr, const float* b2 = nullptr) {
  if (d <= 512) k_ln<FINAL, 4><<<grid, 256, 0, s>>>(x, y, M, d, g, b, g2, b2);
  else if (d <= 1024) k_ln<FINAL, 8><<<grid, 256, 0, s>>>(x, y, M, d, g, b, g2, b2);
  else k_ln<FINAL, 16><<<grid, 256, 0, s>>>(x, y, M, d, g, b, g2, b2);
}

// The block sequence for streams [off, off + n) of the call (their rows
// off*C .. (off+n)*C - 1 of every work buffer), on stream s.  With events,
// each kernel's start is marked and classed (0 GEMM, 1 attention, 2 other).
void enqueue_rows(tsd_encoder* e, int off, int n, int C, cudaStream_t s, const std::vector<cudaEvent_t>* ev,
                  std::vector<int8_t>* cls, int& mk) {
  const tsd_encoder_cfg& c = e->cfg;
  const int M = n * C, d = c.d, r0 = off * C;
  auto mark = [&](int k) {
    if (!ev) return;
    cudaEventRecordWithFlags((*ev)[(size_t)mk], s, cudaEventRecordExternal);
    if (cls) (*cls)[(size_t)mk] = (int8_t)k;
    ++mk;
  };
  const dim3 ln_grid((M + 7) / 8);
  auto gemm = [&](int epi, const CUtensorMap& A, const CUtensorMap& B, int N, int K, const float* bias, void* out,
                  int ld, float alpha) {
    mark(0);
    EGemm g{M, N, K, bias, out, ld, alpha, e->err, r0};
    launch_egemm(epi, g, A, B, s);
  };
  float* x = e->x + (size_t)r0 * d;
  uint16_t* nrm = e->nrm + (size_t)r0 * d;
  const int32_t* slots = e->slots_dev + off;
  gemm(kEInit, e->m_feat, e->m_sub, d, c.stack * c.feat, e->sub_b, e->x, d, 1.f);
  mark(2);
  ln_launch<false>(ln_grid, s, x, nrm, M, d, e->L[0].ln_ff1_g, e->L[0].ln_ff1_b);
  for (int l = 0; l < c.layers; ++l) {
    EncLayerDev& L = e->L[(size_t)l];
    // the first module's norm of this block ran with the previous block's closing norm
    gemm(kESwish, e->m_nrm, L.m_ff1_w1, c.ff, d, L.ff1_b1, e->hid, c.ff, 1.f);
    gemm(kEResid, e->m_hid, L.m_ff1_w2, d, c.ff, L.ff1_b2, e->x, d, 0.5f);
    mark(2);
    ln_launch<false>(ln_grid, s, x, nrm, M, d, L.ln_att_g, L.ln_att_b);
    gemm(kEPlain, e->m_nrm, L.m_qkv, 3 * d, d, L.qkv_b, e->qkv, 3 * d, 1.f);
    mark(1);
    AttnArgs aa{e->qkv + (size_t)r0 * 3 * d, e->att + (size_t)r0 * d, L.pos_tab, L.pos_u, L.pos_v, e->kc, e->vc,
                e->seen, slots, d, c.heads, c.left, c.layers, l, C, c.max_chunk, 1.f / sqrtf((float)(d / c.heads))};
    launch_attn(e, aa, n, s);
    gemm(kEResid, e->m_att, L.m_out, d, d, L.out_b, e->x, d, 1.f);
    mark(2);
    ln_launch<false>(ln_grid, s, x, nrm, M, d, L.ln_conv_g, L.ln_conv_b);
    gemm(kEGlu, e->m_nrm, L.m_pw1, 2 * d, d, L.pw1_b, e->glu, d, 1.f);
    mark(2);
    ConvArgs ca{e->glu + (size_t)r0 * d, e->convz + (size_t)r0 * d, e->cc, L.dw_w, L.dw_b, L.bn_scale, L.bn_shift,
                slots, d, c.kernel, C, c.layers, l};
    const size_t conv_smem = (size_t)(c.kernel - 1 + C) * 128 * sizeof(float);
    if (c.kernel == 9) k_dwconv<9><<<dim3(n, d / 128), 128, conv_smem, s>>>(ca);
    else k_dwconv<0><<<dim3(n, d / 128), 128, conv_smem, s>>>(ca);
    gemm(kEResid, e->m_convz, L.m_pw2, d, d, L.pw2_b, e->x, d, 1.f);
    mark(2);
    ln_launch<false>(ln_grid, s, x, nrm, M, d, L.ln_ff2_g, L.ln_ff2_b);
    gemm(kESwish, e->m_nrm, L.m_ff2_w1, c.ff, d, L.ff2_b1, e->hid, c.ff, 1.f);
    gemm(kEResid, e->m_hid, L.m_ff2_w2, d, c.ff, L.ff2_b2, e->x, d, 0.5f);
    mark(2);
    if (l + 1 < c.layers)
      ln_launch<true>(ln_grid, s, x, nrm, M, d, L.ln_out_g, L.ln_out_b, e->L[(size_t)l + 1].ln_ff1_g,
                      e->L[(size_t)l + 1].ln_ff1_b);
    else
      ln_launch<true>(ln_grid, s, x, e->outb + (size_t)r0 * d, M, d, L.ln_out_g, L.ln_out_b);
  }
}

// How the call's streams split into parallel branches of the graph (rows of
// different streams never meet until the output, so one branch's attention,
// layer norms and convolution fill the SMs while another's GEMMs run):
// branch i takes streams at[i] .. at[i+1]-1.  Up to kEncBranches branches
// of at least 256 rows each; a boundary moves up to a multiple of the
// 128-row tile where one lies within its share.  Returns the branch count.
int branch_points(int n, int C, int* at) {
  int P = std::min(kEncBranches, n * C / 256);
  P = std::min(P, n);
  at[0] = 0;
  if (P < 2) {
    at[1] = n;
    return 1;
  }
  for (int i = 1; i < P; ++i) {
    const int lo = i * n / P, hi = (i + 1) * n / P;
    int k = lo;
    while (k < hi && k * C % 128) ++k;
    at[i] = k < hi ? k : lo;
  }
  at[P] = n;
  return P;
}

// The whole chunk step on stream s.  With events (the instrumented pass) the
// kernels run in one sequence so that every kernel boundary is marked;
// otherwise the call's streams run as parallel branches.
void enqueue(tsd_encoder* e, int n, int C, cudaStream_t s, const std::vector<cudaEvent_t>* ev,
             std::vector<int8_t>* cls) {
  int mk = 0;
  int at[kEncBranches + 1];
  const int P = ev ? 1 : branch_points(n, C, at);
  if (P == 1) {
    enqueue_rows(e, 0, n, C, s, ev, cls, mk);
  } else {
    cudaEventRecord(e->fork_ev, s);
    for (int i = 1; i < P; ++i) cudaStreamWaitEvent(e->branch[i - 1], e->fork_ev, 0);
    for (int i = 0; i < P; ++i)
      enqueue_rows(e, at[i], at[i + 1] - at[i], C, i ? e->branch[i - 1] : s, nullptr, nullptr, mk);
    for (int i = 1; i < P; ++i) {
      cudaEventRecord(e->join_ev[i - 1], e->branch[i - 1]);
      cudaStreamWaitEvent(s, e->join_ev[i - 1], 0);
    }
  }
  if (ev) {
    cudaEventRecordWithFlags((*ev)[(size_t)mk], s, cudaEventRecordExternal);
    if (cls) (*cls)[(size_t)mk] = 2;
    ++mk;
  }
  k_advance<<<1, 256, 0, s>>>(e->seen, e->slots_dev, n, C);
  if (ev) {
    cudaEventRecordWithFlags((*ev)[(size_t)mk], s, cudaEventRecordExternal);
    if (cls) (*cls)[(size_t)mk] = -1;
  }
}

void harvest(tsd_encoder* e, tsd_encoder::Graph& g) {
  if (!g.pending) return;
  cudaEventSynchronize(g.ev.back());
  for (size_t i = 0; i + 1 < g.ev.size(); ++i) {
    float ms = 0.f;
    const int k = g.cls[i];
    if (k >= 0 && k < 3 && cudaEventElapsedTime(&ms, g.ev[i], g.ev[i + 1]) == cudaSuccess) {
      e->ms[k] += ms;
      e->launches[k] += 1;
    }
  }
  cudaGetLastError();
  g.pending = false;
}

tsd_status copy_dev(tsd::DevArena& A, uint16_t** dst, const void* src, size_t n, cudaStream_t s) {
  tsd_status st = A.alloc(dst, n);
  if (st) return st;
  TSD_CUDA(cudaMemcpyAsync(*dst, src, n * 2, cudaMemcpyDeviceToDevice, s));
  return TSD_OK;
}

tsd_status copy_dev(tsd::DevArena& A, float** dst, const float* src, size_t n, cudaStream_t s) {
  tsd_status st = A.alloc(dst, n);
  if (st) return st;
  TSD_CUDA(cudaMemcpyAsync(*dst, src, n * 4, cudaMemcpyDeviceToDevice, s));
  return TSD_OK;
}

size_t round_up(size_t x, size_t m) { return (x + m - 1) / m * m; }

}  // namespace

}  // namespace tsd

using namespace tsd;

extern "C" tsd_status tsd_encoder_create(const tsd_encoder_cfg* cfg, const void* sub_w, const float* sub_b,
                                         const tsd_encoder_layer* layers, void* cuda_stream, tsd_encoder** out) {
  clear_error();
  if (!cfg || !sub_w || !sub_b || !layers || !out) return fail(TSD_EINVAL, "tsd_encoder_create: NULL argument");
  const tsd_encoder_cfg c = *cfg;
  if (c.d < 128 || c.d > 2048 || c.d % 128) return fail(TSD_EINVAL, "tsd_encoder_create: d=%d", c.d);
  if (c.heads < 1 || c.d % c.heads || (c.d / c.heads != 64 && c.d / c.heads != 128))
    return fail(TSD_EINVAL, "tsd_encoder_create: d/heads must be 64 or 128 (d=%d heads=%d)", c.d, c.heads);
  if (c.ff < 128 || c.ff > 8192 || c.ff % 128) return fail(TSD_EINVAL, "tsd_encoder_create: ff=%d", c.ff);
  if (c.layers < 1 || c.layers > 64) return fail(TSD_EINVAL, "tsd_encoder_create: layers=%d", c.layers);
  if (c.kernel < 1 || c.kernel > 32) return fail(TSD_EINVAL, "tsd_encoder_create: kernel=%d", c.kernel);
  if (c.left < 0 || c.left > 128) return fail(TSD_EINVAL, "tsd_encoder_create: left=%d", c.left);
  if (c.max_chunk < 1 || c.max_chunk > 32) return fail(TSD_EINVAL, "tsd_encoder_create: max_chunk=%d", c.max_chunk);
  if (c.feat < 1 || c.stack < 1 || (c.stack * c.feat) % 64 || c.stack * c.feat > 8192)
    return fail(TSD_EINVAL, "tsd_encoder_create: stack*feat=%d must be a multiple of 64, <= 8192", c.stack * c.feat);
  if (c.max_streams < 1 || c.max_streams > 4096)
    return fail(TSD_EINVAL, "tsd_encoder_create: max_streams=%d", c.max_streams);
  for (int l = 0; l < c.layers; ++l) {
    const tsd_encoder_layer& L = layers[l];
    const void* ptrs[] = {L.ln_ff1_g, L.ln_ff1_b, L.ff1_w1, L.ff1_b1, L.ff1_w2, L.ff1_b2, L.ln_att_g, L.ln_att_b,
                          L.qkv_w, L.qkv_b, L.pos_w, L.pos_u, L.pos_v, L.out_w, L.out_b, L.ln_conv_g, L.ln_conv_b,
                          L.pw1_w, L.pw1_b, L.dw_w, L.dw_b, L.bn_scale, L.bn_shift, L.pw2_w, L.pw2_b, L.ln_ff2_g,
                          L.ln_ff2_b, L.ff2_w1, L.ff2_b1, L.ff2_w2, L.ff2_b2, L.ln_out_g, L.ln_out_b};
    for (const void* p : ptrs)
      if (!p) return fail(TSD_EINVAL, "tsd_encoder_create: layer %d has a NULL weight", l);
  }
  struct Guard {  // on a failed create, let queued copies finish before the memory is released
    std::unique_ptr<tsd_encoder> p;
    cudaStream_t s;
    ~Guard() {
      if (p) cudaStreamSynchronize(s);
    }
  } guard{std::unique_ptr<tsd_encoder>(new tsd_encoder()), static_cast<cudaStream_t>(cuda_stream)};
  tsd_encoder* const e = guard.p.get();
  e->cfg = c;
  TSD_CUDA(cudaGetDevice(&e->device));
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  e->last_stream = s;
  TSD_CUDA(egemm_prepare());
  const int d = c.d, ff = c.ff, K1 = c.kernel - 1, dh = d / c.heads;
  const size_t asm_ = attn_smem(dh, c.left, c.max_chunk);
  if (asm_ > 227 * 1024) return fail(TSD_EINVAL, "tsd_encoder_create: attention window too large");
  if (dh == 64) TSD_CUDA(cudaFuncSetAttribute(k_attn<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)asm_));
  else TSD_CUDA(cudaFuncSetAttribute(k_attn<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)asm_));
  e->n_off = c.left + 2 * c.max_chunk - 1;
  e->M_pad = (int)round_up((size_t)c.max_streams * c.max_chunk, 128);
  DevArena& A = e->arena;
  tsd_status st;
  if ((st = copy_dev(A, &e->sub_w, sub_w, (size_t)d * c.stack * c.feat, s)) || (st = copy_dev(A, &e->sub_b, sub_b, d, s)))
    return st;
  e->L.resize((size_t)c.layers);
  for (int l = 0; l < c.layers; ++l) {
    const tsd_encoder_layer& W = layers[l];
    EncLayerDev& L = e->L[(size_t)l];
    float *g[10];
    const float* gs[10] = {W.ln_ff1_g, W.ln_ff1_b, W.ln_att_g, W.ln_att_b, W.ln_conv_g,
                           W.ln_conv_b, W.ln_ff2_g, W.ln_ff2_b, W.ln_out_g, W.ln_out_b};
    for (int i = 0; i < 10; ++i)
      if ((st = copy_dev(A, &g[i], gs[i], d, s))) return st;
    L.ln_ff1_g = g[0], L.ln_ff1_b = g[1], L.ln_att_g = g[2], L.ln_att_b = g[3], L.ln_conv_g = g[4];
    L.ln_conv_b = g[5], L.ln_ff2_g = g[6], L.ln_ff2_b = g[7], L.ln_out_g = g[8], L.ln_out_b = g[9];
    if ((st = copy_dev(A, &L.ff1_w1, W.ff1_w1, (size_t)ff * d, s)) || (st = copy_dev(A, &L.ff1_b1, W.ff1_b1, ff, s)) ||
        (st = copy_dev(A, &L.ff1_w2, W.ff1_w2, (size_t)d * ff, s)) || (st = copy_dev(A, &L.ff1_b2, W.ff1_b2, d, s)) ||
        (st = copy_dev(A, &L.qkv_w, W.qkv_w, (size_t)3 * d * d, s)) || (st = copy_dev(A, &L.qkv_b, W.qkv_b, 3 * d, s)) ||
        (st = copy_dev(A, &L.pos_w, W.pos_w, (size_t)d * d, s)) || (st = copy_dev(A, &L.pos_u, W.pos_u, d, s)) ||
        (st = copy_dev(A, &L.pos_v, W.pos_v, d, s)) || (st = copy_dev(A, &L.out_w, W.out_w, (size_t)d * d, s)) ||
        (st = copy_dev(A, &L.out_b, W.out_b, d, s)) || (st = A.alloc(&L.pw1_w, (size_t)2 * d * d)) ||
        (st = A.alloc(&L.pw1_b, (size_t)2 * d)) || (st = copy_dev(A, &L.dw_w, W.dw_w, (size_t)d * c.kernel, s)) ||
        (st = copy_dev(A, &L.dw_b, W.dw_b, d, s)) || (st = copy_dev(A, &L.bn_scale, W.bn_scale, d, s)) ||
        (st = copy_dev(A, &L.bn_shift, W.bn_shift, d, s)) || (st = copy_dev(A, &L.pw2_w, W.pw2_w, (size_t)d * d, s)) ||
        (st = copy_dev(A, &L.pw2_b, W.pw2_b, d, s)) || (st = copy_dev(A, &L.ff2_w1, W.ff2_w1, (size_t)ff * d, s)) ||
        (st = copy_dev(A, &L.ff2_b1, W.ff2_b1, ff, s)) || (st = copy_dev(A, &L.ff2_w2, W.ff2_w2, (size_t)d * ff, s)) ||
        (st = copy_dev(A, &L.ff2_b2, W.ff2_b2, d, s)) || (st = A.alloc(&L.pos_tab, (size_t)e->n_off * d)))
      return st;
    k_glu_repack<<<2 * d, 128, 0, s>>>(static_cast<const uint16_t*>(W.pw1_w), W.pw1_b, L.pw1_w, L.pw1_b, d);
    k_pos_table<<<e->n_off, 256, (size_t)d * sizeof(double), s>>>(L.pos_w, L.pos_tab, d, c.max_chunk);
    TSD_CUDA(cudaGetLastError());
    if (!egemm_map_b(&L.m_ff1_w1, L.ff1_w1, ff, d) || !egemm_map_b(&L.m_ff1_w2, L.ff1_w2, d, ff) ||
        !egemm_map_b(&L.m_qkv, L.qkv_w, 3 * d, d) || !egemm_map_b(&L.m_out, L.out_w, d, d) ||
        !egemm_map_b(&L.m_pw1, L.pw1_w, 2 * d, d) || !egemm_map_b(&L.m_pw2, L.pw2_w, d, d) ||
        !egemm_map_b(&L.m_ff2_w1, L.ff2_w1, ff, d) || !egemm_map_b(&L.m_ff2_w2, L.ff2_w2, d, ff))
      return fail(TSD_ECUDA, "tsd_encoder_create: tensor map encoding failed");
  }
  const size_t Mp = (size_t)e->M_pad, SF = (size_t)c.stack * c.feat;
  if ((st = A.alloc(&e->feat, Mp * SF)) || (st = A.alloc(&e->x, Mp * d)) || (st = A.alloc(&e->nrm, Mp * d)) ||
      (st = A.alloc(&e->hid, Mp * ff)) || (st = A.alloc(&e->qkv, Mp * 3 * d)) || (st = A.alloc(&e->att, Mp * d)) ||
      (st = A.alloc(&e->glu, Mp * d)) || (st = A.alloc(&e->convz, Mp * d)) || (st = A.alloc(&e->outb, Mp * d)))
    return st;
  const size_t kv = (size_t)c.max_streams * c.layers * c.left * d;
  const size_t cv = (size_t)c.max_streams * c.layers * std::max(K1, 1) * d;
  if ((st = A.alloc(&e->kc, std::max<size_t>(kv, 1))) || (st = A.alloc(&e->vc, std::max<size_t>(kv, 1))) ||
      (st = A.alloc(&e->cc, cv)) || (st = A.alloc(&e->seen, (size_t)c.max_streams)) ||
      (st = A.alloc(&e->slots_dev, (size_t)c.max_streams)) || (st = A.alloc(&e->err, 1)))
    return st;
  TSD_CUDA(cudaMemsetAsync(e->kc, 0, std::max<size_t>(kv, 1) * 2, s));
  TSD_CUDA(cudaMemsetAsync(e->vc, 0, std::max<size_t>(kv, 1) * 2, s));
  TSD_CUDA(cudaMemsetAsync(e->cc, 0, cv * 2, s));
  TSD_CUDA(cudaMemsetAsync(e->seen, 0, (size_t)c.max_streams * 4, s));
  TSD_CUDA(cudaMemsetAsync(e->err, 0, 4, s));
  TSD_CUDA(cudaMemsetAsync(e->feat, 0, Mp * SF * 2, s));
  TSD_CUDA(cudaMemsetAsync(e->nrm, 0, Mp * d * 2, s));
  TSD_CUDA(cudaMemsetAsync(e->hid, 0, Mp * ff * 2, s));
  TSD_CUDA(cudaMemsetAsync(e->att, 0, Mp * d * 2, s));
  TSD_CUDA(cudaMemsetAsync(e->convz, 0, Mp * d * 2, s));
  if (!egemm_map_a(&e->m_feat, e->feat, e->M_pad, (int)SF) || !egemm_map_a(&e->m_nrm, e->nrm, e->M_pad, d) ||
      !egemm_map_a(&e->m_hid, e->hid, e->M_pad, ff) || !egemm_map_a(&e->m_att, e->att, e->M_pad, d) ||
      !egemm_map_a(&e->m_convz, e->convz, e->M_pad, d) || !egemm_map_b(&e->m_sub, e->sub_w, d, (int)SF))
    return fail(TSD_ECUDA, "tsd_encoder_create: tensor map encoding failed");
  TSD_CUDA(cudaMallocHost(&e->slots_host, sizeof(int32_t) * (size_t)c.max_streams));
  TSD_CUDA(cudaEventCreateWithFlags(&e->slots_ev, cudaEventDisableTiming));
  TSD_CUDA(cudaStreamCreateWithFlags(&e->cap_stream, cudaStreamNonBlocking));
  TSD_CUDA(cudaEventCreateWithFlags(&e->fork_ev, cudaEventDisableTiming));
  for (int i = 0; i < kEncBranches - 1; ++i) {
    TSD_CUDA(cudaStreamCreateWithFlags(&e->branch[i], cudaStreamNonBlocking));
    TSD_CUDA(cudaEventCreateWithFlags(&e->join_ev[i], cudaEventDisableTiming));
  }
  TSD_CUDA(cudaStreamSynchronize(s));
  TSD_CUDA(cudaGetLastError());
  e->slot_open.assign((size_t)c.max_streams, 0);
  *out = guard.p.release();
  return TSD_OK;
}

extern "C" void tsd_encoder_free(tsd_encoder* e) {
  if (!e) return;
  set_device(e);
  cudaDeviceSynchronize();
  delete e;  // the destructor releases graphs, events, the stream and device memory
}

extern "C" tsd_status tsd_encoder_open(tsd_encoder* e, int32_t* slot_out) {
  clear_error();
  if (!e || !slot_out) return fail(TSD_EINVAL, "tsd_encoder_open: NULL argument");
  auto it = std::find(e->slot_open.begin(), e->slot_open.end(), 0);
  if (it == e->slot_open.end()) return fail(TSD_ESTATE, "tsd_encoder_open: all %d slots are open", e->cfg.max_streams);
  tsd_status st = set_device(e);
  if (st) return st;
  const int slot = (int)(it - e->slot_open.begin());
  const tsd_encoder_cfg& c = e->cfg;
  const size_t kv = (size_t)c.layers * c.left * c.d, cv = (size_t)c.layers * (c.kernel - 1) * c.d;
  cudaStream_t s = e->last_stream;
  if (kv) {
    TSD_CUDA(cudaMemsetAsync(e->kc + (size_t)slot * kv, 0, kv * 2, s));
    TSD_CUDA(cudaMemsetAsync(e->vc + (size_t)slot * kv, 0, kv * 2, s));
  }
  if (cv) TSD_CUDA(cudaMemsetAsync(e->cc + (size_t)slot * cv, 0, cv * 2, s));
  TSD_CUDA(cudaMemsetAsync(e->seen + slot, 0, 4, s));
  *it = 1;
  *slot_out = slot;
  return TSD_OK;
}

extern "C" tsd_status tsd_encoder_close(tsd_encoder* e, int32_t slot) {
  clear_error();
  if (!e) return fail(TSD_EINVAL, "tsd_encoder_close: NULL encoder");
  if (slot < 0 || slot >= e->cfg.max_streams || !e->slot_open[(size_t)slot])
    return fail(TSD_ESTATE, "tsd_encoder_close: slot %d is not open", slot);
  e->slot_open[(size_t)slot] = 0;
  return TSD_OK;
}

extern "C" tsd_status tsd_encode_chunk(tsd_encoder* e, int32_t n, const int32_t* slots, const void* feats_bf16,
                                       int32_t C, void* out_bf16, void* cuda_stream) {
  clear_error();
  NvtxRange nvtx("tsd_encode_chunk");
  if (!e || !slots || !feats_bf16 || !out_bf16) return fail(TSD_EINVAL, "tsd_encode_chunk: NULL argument");
  const tsd_encoder_cfg& c = e->cfg;
  if (n < 1 || n > c.max_streams) return fail(TSD_EINVAL, "tsd_encode_chunk: n=%d out of [1, %d]", n, c.max_streams);
  if (C < 1 || C > c.max_chunk) return fail(TSD_EINVAL, "tsd_encode_chunk: C=%d out of [1, %d]", C, c.max_chunk);
  {
    std::vector<uint8_t> seen((size_t)c.max_streams, 0);
    for (int i = 0; i < n; ++i) {
      const int s = slots[i];
      if (s < 0 || s >= c.max_streams || !e->slot_open[(size_t)s])
        return fail(TSD_ESTATE, "tsd_encode_chunk: slot %d is not open", s);
      if (seen[(size_t)s]) return fail(TSD_EINVAL, "tsd_encode_chunk: slot %d listed twice", s);
      seen[(size_t)s] = 1;
    }
  }
  tsd_status st = set_device(e);
  if (st) return st;
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  e->last_stream = s;
  TSD_CUDA(cudaEventSynchronize(e->slots_ev));
  std::memcpy(e->slots_host, slots, sizeof(int32_t) * (size_t)n);
  TSD_CUDA(cudaMemcpyAsync(e->slots_dev, e->slots_host, sizeof(int32_t) * (size_t)n, cudaMemcpyHostToDevice, s));
  TSD_CUDA(cudaEventRecord(e->slots_ev, s));
  const size_t M = (size_t)n * C;
  TSD_CUDA(cudaMemcpyAsync(e->feat, feats_bf16, M * c.stack * c.feat * 2, cudaMemcpyDeviceToDevice, s));
  auto key = std::make_pair(std::make_pair(n, C), e->timing);
  tsd_encoder::Graph& g = e->graphs[key];
  if (e->timing) {
    harvest(e, g);
    if (g.ev.empty()) {
      g.ev.resize((size_t)n_marks(e));
      g.cls.assign(g.ev.size(), -1);
      for (auto& ev : g.ev) TSD_CUDA(cudaEventCreate(&ev));
    }
  }
  if (!g.exec) {
    cudaGraph_t gr = nullptr;
    TSD_CUDA(cudaStreamBeginCapture(e->cap_stream, cudaStreamCaptureModeThreadLocal));
    enqueue(e, n, C, e->cap_stream, e->timing ? &g.ev : nullptr, e->timing ? &g.cls : nullptr);
    cudaError_t ce = cudaStreamEndCapture(e->cap_stream, &gr);
    if (ce != cudaSuccess) return cuda_fail(ce, "tsd_encode_chunk: graph capture");
    ce = cudaGraphInstantiate(&g.exec, gr, 0);
    cudaGraphDestroy(gr);
    if (ce != cudaSuccess) {
      g.exec = nullptr;
      return cuda_fail(ce, "tsd_encode_chunk: graph instantiate");
    }
  }
  TSD_CUDA(cudaGraphLaunch(g.exec, s));
  if (e->timing) g.pending = true;
  TSD_CUDA(cudaMemcpyAsync(out_bf16, e->outb, M * c.d * 2, cudaMemcpyDeviceToDevice, s));
  return TSD_OK;
}

extern "C" tsd_status tsd_encoder_check(tsd_encoder* e) {
  clear_error();
  if (!e) return fail(TSD_EINVAL, "tsd_encoder_check: NULL encoder");
  tsd_status st = set_device(e);
  if (st) return st;
  TSD_CUDA(cudaStreamSynchronize(e->last_stream));
  unsigned int v = 0;
  TSD_CUDA(cudaMemcpy(&v, e->err, 4, cudaMemcpyDeviceToHost));
  if (v) {
    TSD_CUDA(cudaMemset(e->err, 0, 4));
    return fail(TSD_EDEVICE, "tsd_encoder_check: a bounded wait expired in the encoder GEMM (code %u)", v);
  }
  return TSD_OK;
}

extern "C" tsd_status tsd_encoder_set_timing(tsd_encoder* e, int32_t enable) {
  clear_error();
  if (!e) return fail(TSD_EINVAL, "tsd_encoder_set_timing: NULL encoder");
  e->timing = enable ? 1 : 0;
  return TSD_OK;
}

extern "C" tsd_status tsd_encoder_timing(tsd_encoder* e, double* ms, int64_t* launches, int32_t n_classes,
                                         int32_t reset) {
  clear_error();
  if (!e) return fail(TSD_EINVAL, "tsd_encoder_timing: NULL encoder");
  tsd_status st = set_device(e);
  if (st) return st;
  for (auto& kv : e->graphs) harvest(e, kv.second);
  for (int i = 0; i < n_classes && i < 3; ++i) {
    if (ms) ms[i] = e->ms[i];
    if (launches) launches[i] = e->launches[i];
  }
  if (reset)
    for (int i = 0; i < 3; ++i) {
      e->ms[i] = 0;
      e->launches[i] = 0;
    }
  return TSD_OK;
}

extern "C" tsd_status tsd_encoder_gemm_flops(const tsd_encoder* e, int32_t n, int32_t C, double* flops) {
  clear_error();
  if (!e || !flops) return fail(TSD_EINVAL, "tsd_encoder_gemm_flops: NULL argument");
  const tsd_encoder_cfg& c = e->cfg;
  const double M = (double)n * C, d = c.d, ff = c.ff;
  // subsampling; per block q/k/v (3d^2), output (d^2), GLU pointwise (2d^2), pointwise (d^2), two
  // feed-forward halves (2 x 2 ff d)
  *flops = 2.0 * M * d * c.stack * c.feat + c.layers * 2.0 * M * (7.0 * d * d + 4.0 * ff * d);
  return TSD_OK;
}

extern "C" tsd_status tsd_encoder_launches_per_chunk(const tsd_encoder* e, int32_t n, int32_t C, int64_t* launches) {
  clear_error();
  if (!e || !launches) return fail(TSD_EINVAL, "tsd_encoder_launches_per_chunk: NULL argument");
  if (n < 1 || n > e->cfg.max_streams || C < 1 || C > e->cfg.max_chunk)
    return fail(TSD_EINVAL, "tsd_encoder_launches_per_chunk: n=%d C=%d out of range", n, C);
  int at[kEncBranches + 1];
  const int P = branch_points(n, C, at);
  *launches = (int64_t)P * (2 + 14 * e->cfg.layers) + 1;
  return TSD_OK;
}
