// Tensor-core GEMMs of the stateful Transducer form (prediction network and
// joint projections), out[r][j] = sum_k A[r][k] * B[j][k] with A and B bf16
// and K-major, 128 x 128 output tiles on tcgen05 (accumulator in TMEM, TMA
// loads into 128-byte-swizzled stages), each with its own epilogue:
//   kEncProj:   P_enc = enc W_enc + b_enc, stored fp32 (once per chunk);
//   kLstm:      the LSTM cell on the gate pre-activations (columns 4u+q are
//               gate q of unit u): for rows that emitted a label (or start a
//               sequence) c' = s(f) c + s(i) tanh(g), h' = s(o) tanh(c') into
//               the stream's state; every row's h goes on to the projection;
//   kJointIn:   the joint input A = bf16(ReLU(P_enc[t] + h W_pred + b_pred))
//               for the row's current frame t.
// Warp roles (192 threads): warp 0 TMA producer, warp 1 TMEM allocator and
// MMA issuer, warps 2-5 epilogue (thread = row).  Every mbarrier wait is
// bounded in time; on expiry the kernel records an error and returns.
#include <cuda.h>

#include "decoder.h"
#include "gemm_tc.h"
#include "tc_common.cuh"

namespace tsd {

namespace {

using namespace tc;

// Output-tile width per epilogue.  The per-step GEMMs have few rows (one
// 128-row tile per 128 streams), so narrower tiles put more SMs on the
// weights, and deeper pipelines keep more of each CTA's k-blocks in flight.
template <int EPI>
struct Shape {
  static constexpr int BN = EPI == kEncProj ? 128 : (EPI == kLstm ? 64 : 32);
  static constexpr int ABytes = kBM * kBK * 2;
  static constexpr int BBytes = BN * kBK * 2;
  static constexpr int StageBytes = ABytes + BBytes;
  static constexpr int Stages = (200 * 1024) / StageBytes;  // 6 / 8 / 10
  static constexpr int Smem = Stages * StageBytes + 1024 /*align*/ + 256 /*barriers*/ + BN * 4 /*bias*/;
  static_assert((2 * Stages + 1) * 8 + 4 <= 256, "barrier area");
};
constexpr int kGThreads = 192;
constexpr int kGBar = 256;  // mbarriers and the TMEM address

__device__ __forceinline__ float sigm(float x) { return 1.f / (1.f + expf(-x)); }

__device__ __forceinline__ uint16_t bf16_bits(float v) {
  const __nv_bfloat16 b = __float2bfloat16_rn(v);
  return *reinterpret_cast<const uint16_t*>(&b);
}

template <int EPI>
__global__ void __launch_bounds__(kGThreads, 1)
    k_gemm_tc(DecView d, GemmArgs g, const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB) {
  constexpr int kGN = Shape<EPI>::BN;
  constexpr int kGStages = Shape<EPI>::Stages;
  constexpr int kGABytes = Shape<EPI>::ABytes;
  constexpr int kGStageBytes = Shape<EPI>::StageBytes;
  static_assert(kGN % 32 == 0 && kGStageBytes % 1024 == 0, "tile shape");
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + kGStages * kGStageBytes);
  uint64_t* empty = full + kGStages;
  uint64_t* accum = empty + kGStages;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(accum + 1);
  float* s_bias = reinterpret_cast<float*>(smem + kGStages * kGStageBytes + kGBar);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n0 = blockIdx.x * kGN, m0 = blockIdx.y * kBM;
  const int KB = g.K / kBK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kGStages; ++s) {
      mbar_init(full + s, 1);
      mbar_init(empty + s, 1);
    }
    mbar_init(accum, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(kGN)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  if (warp >= 2) {
    // the tile's bias (a constant weight) to shared memory
    const int j = threadIdx.x - 64;
    if (j < kGN) s_bias[j] = n0 + j < g.N ? g.bias[n0 + j] : 0.f;
  }
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem = *tmem_slot;
  bool ok = true;
  // the weights are constant: the first stages' B tiles go out before the
  // dependency wait
  const int pre = min(KB, kGStages);
  if (warp == 0 && lane == 0) {
    for (int kb = 0; kb < pre; ++kb) {
      mbar_expect_tx(full + kb, kGStageBytes);
      tma_load_2d(smem + kb * kGStageBytes + kGABytes, &tmB, full + kb, kb * kBK, n0);
    }
  }
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  if (warp == 0) {
    if (lane == 0) {
      int issued = 0;
      for (int kb = 0; kb < KB; ++kb) {
        const int s = kb % kGStages;
        const uint32_t ph = (uint32_t)(kb / kGStages) & 1u;
        unsigned char* sa = smem + s * kGStageBytes;
        if (kb < pre) {
          tma_load_2d(sa, &tmA, full + s, kb * kBK, m0);
          ++issued;
          continue;
        }
        if (!mbar_wait(empty + s, ph ^ 1u)) { ok = false; break; }
        mbar_expect_tx(full + s, kGStageBytes);
        tma_load_2d(sa, &tmA, full + s, kb * kBK, m0);
        tma_load_2d(sa + kGABytes, &tmB, full + s, kb * kBK, n0);
        ++issued;
      }
      if (!ok) {
        for (int kb = max(0, issued - kGStages); kb < issued; ++kb)
          mbar_wait(full + kb % kGStages, (uint32_t)(kb / kGStages) & 1u);
        atomicOr(d.err, 64);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16(kBM, kGN);
      for (int kb = 0; kb < KB; ++kb) {
        const int s = kb % kGStages;
        const uint32_t ph = (uint32_t)(kb / kGStages) & 1u;
        if (!mbar_wait(full + s, ph)) { ok = false; break; }
        fence_after();
        const uint32_t sa = smem_u32(smem + s * kGStageBytes);
        const uint64_t ad = sw128_desc(sa), bd = sw128_desc(sa + kGABytes);
#pragma unroll
        for (int k = 0; k < kBK / 16; ++k)
          mma_bf16(tmem, ad + (uint64_t)(2 * k), bd + (uint64_t)(2 * k), idesc, (kb | k) ? 1u : 0u);
        mma_commit(empty + s);
      }
      mma_commit(accum);
      if (!ok) atomicOr(d.err, 128);
    }
    __syncwarp();
  } else {
    const int q = warp & 3;
    const int row = q * 32 + lane;
    const int gr = m0 + row;
    // Per-row operands the epilogue combines with the accumulator are loaded
    // into registers before the accumulator is ready: with the stores that
    // follow (possibly aliasing, to the compiler) they would otherwise each
    // cost a dependent round trip to memory.
    const Params* P = d.params;
    const bool live = gr < g.M;
    int slot = 0, flag = 0, t = 0, T = 1;
    float4 pre4[EPI == kLstm ? kGN / 16 : (EPI == kJointIn ? kGN / 4 : 1)];
    uint4 h4[EPI == kLstm ? kGN / 32 : 1];
    const int D = d.pred_D;
    const int u0 = n0 / 4;  // kLstm: the tile's first LSTM unit
    if (EPI == kLstm && live) {
      slot = P->slots[gr];
      flag = d.pflag[gr];
      if (flag) {
        const float4* cp = reinterpret_cast<const float4*>(d.pred_c + (size_t)slot * D + u0);
#pragma unroll
        for (int i = 0; i < kGN / 16; ++i) pre4[i] = cp[i];
      } else {
        const uint4* hp = reinterpret_cast<const uint4*>(d.pred_h + (size_t)slot * D + u0);
#pragma unroll
        for (int i = 0; i < kGN / 32; ++i) h4[i] = hp[i];
      }
    }
    if (EPI == kJointIn && live) {
      t = d.r_t[gr];
      T = P->T;
      if (t < T) {
        const float4* pe = reinterpret_cast<const float4*>(d.pred_penc + ((size_t)gr * T + t) * g.ld + n0);
#pragma unroll
        for (int i = 0; i < kGN / 4; ++i)
          if (n0 + 4 * i < g.N) pre4[i] = pe[i];  // N is a multiple of 32: whole chunks
      }
    }
    ok = __all_sync(0xffffffffu, mbar_wait(accum, 0));
    if (!ok && lane == 0) atomicOr(d.err, 256);
    fence_after();
    if (ok) {
      const uint32_t tbase = tmem + ((uint32_t)(q * 32) << 16);
#pragma unroll
      for (int c = 0; c < kGN / 32; ++c) {
        __syncwarp();
        float v[32];
        tmem_ld32(tbase + (uint32_t)(c * 32), v);
        const int c0 = n0 + c * 32;
        if (!live || c0 >= g.N) continue;
        const float* bb = s_bias + c * 32;
        if (EPI == kEncProj) {
          float* out = g.out + (size_t)gr * g.ld + c0;
#pragma unroll
          for (int i = 0; i < 32; i += 4)
            *reinterpret_cast<float4*>(out + i) =
                make_float4(v[i] + bb[i], v[i + 1] + bb[i + 1], v[i + 2] + bb[i + 2], v[i + 3] + bb[i + 3]);
        } else if (EPI == kLstm) {
          // columns 4u+q of this chunk: gates (i, f, g, o) of units u0+8c .. u0+8c+7
          const size_t base = (size_t)slot * D + u0 + 8 * c;
          uint4 hv;
          if (flag) {
            float cn[8];
            const float* cprev = reinterpret_cast<const float*>(&pre4[2 * c]);
            uint16_t* hb = reinterpret_cast<uint16_t*>(&hv);
#pragma unroll
            for (int j = 0; j < 8; ++j) {
              const float gi = sigm(v[4 * j] + bb[4 * j]);
              const float gf = sigm(v[4 * j + 1] + bb[4 * j + 1]);
              const float gg = tanhf(v[4 * j + 2] + bb[4 * j + 2]);
              const float go = sigm(v[4 * j + 3] + bb[4 * j + 3]);
              cn[j] = gf * cprev[j] + gi * gg;
              hb[j] = bf16_bits(go * tanhf(cn[j]));
            }
            float4* cw = reinterpret_cast<float4*>(d.pred_c + base);
            cw[0] = make_float4(cn[0], cn[1], cn[2], cn[3]);
            cw[1] = make_float4(cn[4], cn[5], cn[6], cn[7]);
            *reinterpret_cast<uint4*>(d.pred_h + base) = hv;
          } else {
            hv = h4[c];
          }
          *reinterpret_cast<uint4*>(d.pred_hin + (size_t)gr * D + u0 + 8 * c) = hv;
        } else {  // kJointIn
          if (t < T) {
            const float* pe = reinterpret_cast<const float*>(&pre4[8 * c]);
            uint16_t* a = d.A + (size_t)gr * d.H + c0;
#pragma unroll
            for (int i = 0; i < 32; i += 8) {
              uint4 o;
              uint16_t* ob = reinterpret_cast<uint16_t*>(&o);
#pragma unroll
              for (int k = 0; k < 8; ++k) ob[k] = bf16_bits(fmaxf(pe[i + k] + (v[i + k] + bb[i + k]), 0.f));
              *reinterpret_cast<uint4*>(a + i) = o;
            }
          }
        }
      }
    }
  }
  fence_before();
  __syncthreads();
  if (warp == 1) {
    fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kGN) : "memory");
  }
}

}  // namespace

bool gemm_tc_map_a(CUtensorMap* m, const uint16_t* A, int rows, int K) {
  return make_map(m, A, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, K, rows, kBK, kBM);
}

bool gemm_tc_map_b(CUtensorMap* m, int epi, const uint16_t* B, int rows, int K) {
  const int bn = epi == kEncProj ? Shape<kEncProj>::BN : (epi == kLstm ? Shape<kLstm>::BN : Shape<kJointIn>::BN);
  return make_map(m, B, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, K, rows, kBK, bn);
}

cudaError_t gemm_tc_prepare() {
  cudaError_t e = cudaFuncSetAttribute(k_gemm_tc<kEncProj>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       Shape<kEncProj>::Smem);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(k_gemm_tc<kLstm>, cudaFuncAttributeMaxDynamicSharedMemorySize, Shape<kLstm>::Smem);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(k_gemm_tc<kJointIn>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             Shape<kJointIn>::Smem);
  return e;
}

namespace {
template <int EPI>
void launch_one(const DecView& d, const GemmArgs& g, const CUtensorMap& a, const CUtensorMap& b, cudaStream_t s,
                bool pdl) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((g.N + Shape<EPI>::BN - 1) / Shape<EPI>::BN, (g.M + kBM - 1) / kBM);
  cfg.blockDim = dim3(kGThreads);
  cfg.dynamicSmemBytes = Shape<EPI>::Smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  cudaLaunchKernelEx(&cfg, k_gemm_tc<EPI>, d, g, a, b);
}
}  // namespace

void launch_gemm_tc(int epi, const DecView& d, const GemmArgs& g, const CUtensorMap& a, const CUtensorMap& b,
                    cudaStream_t s, bool pdl) {
  if (epi == kEncProj) launch_one<kEncProj>(d, g, a, b, s, pdl);
  else if (epi == kLstm) launch_one<kLstm>(d, g, a, b, s, pdl);
  else launch_one<kJointIn>(d, g, a, b, s, pdl);
}

}  // namespace tsd
