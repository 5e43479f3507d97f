// Tensor-core GEMM of the cache-aware encoder: out = A . B^T with A [M][K]
// and B [N][K] bf16 K-major (B = a weight stored [out][in]), fp32 accumulate
// in TMEM, 128 x 128 output tiles.  Persistent: one CTA per SM walks the
// tile list (tiles of one weight column block are adjacent, so concurrent
// CTAs share B in L2).  Warp 0 streams A and B k-blocks by TMA into a
// 6-stage ring of 128-byte-swizzled stages that continues across tiles;
// warp 1 allocates two 128-column TMEM accumulators and issues the MMAs of
// tile i into accumulator i mod 2; warps 2-9 run the epilogue of tile i
// (thread = output row; warp w reads TMEM lanes 32 (w mod 4) .., the two
// warps of a lane quadrant alternate 32-column chunks) while the MMAs of
// tile i+1 run, then hand the accumulator back.  The epilogue
// applies the bias and one of: the residual update of the fp32 stream
// (x = acc + b, or x += alpha (acc + b)), Swish to bf16, plain bf16, or GLU
// to bf16.  Every mbarrier wait is bounded in time; on expiry the kernel
// records an error bit and the other roles run out their own bounded waits.
#include <cuda.h>
#include <cuda_bf16.h>

#include "encoder.h"
#include "tc_common.cuh"

namespace tsd {

namespace {

using namespace tc;

constexpr int kBN = kEgBN;
constexpr int kStages = 6;
constexpr int kThreads = 320;  // warp 0 TMA, warp 1 MMA, warps 2-9 epilogue
constexpr int kEpiWarps = 8;
constexpr int kABytes = kBM * kBK * 2;
constexpr int kBBytes = kBN * kBK * 2;
constexpr int kStageBytes = kABytes + kBBytes;
constexpr int kBarBytes = 256;
constexpr int kSmem = kStages * kStageBytes + 1024 /*align*/ + kBarBytes + kEpiWarps * 2 * kBN * 4 /*bias: per warp, per accumulator*/;
static_assert((2 * kStages + 4) * 8 + 4 <= kBarBytes, "barrier area");
int g_sms = 148;

__device__ __forceinline__ float sigm(float x) { return 1.f / (1.f + expf(-x)); }

__device__ __forceinline__ uint32_t pack_bf16(float a, float b) {
  const __nv_bfloat16 x = __float2bfloat16_rn(a), y = __float2bfloat16_rn(b);
  return (uint32_t)(*reinterpret_cast<const uint16_t*>(&x)) | ((uint32_t)(*reinterpret_cast<const uint16_t*>(&y)) << 16);
}

template <int EPI>
__global__ void __launch_bounds__(kThreads, 1)
    k_egemm(EGemm g, const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB) {
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + kStages * kStageBytes);
  uint64_t* empty = full + kStages;
  uint64_t* accf = empty + kStages;  // [2] accumulator holds a finished tile
  uint64_t* acce = accf + 2;         // [2] accumulator read out by the epilogue
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(acce + 2);
  float* s_bias = reinterpret_cast<float*>(smem + kStages * kStageBytes + kBarBytes);  // [8 warps][2][kBN]

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int KB = g.K / kBK;
  const int Mt = (g.M + kBM - 1) / kBM, Nt = (g.N + kBN - 1) / kBN;
  const int tiles = Mt * Nt;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(full + s, 1);
      mbar_init(empty + s, 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(accf + b, 1);
      mbar_init(acce + b, kEpiWarps);  // one arrival per epilogue warp
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(2 * kBN)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      int it = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x) {
        const int m0 = g.m0 + (t % Mt) * kBM, n0 = (t / Mt) * kBN;
        for (int kb = 0; kb < KB; ++kb, ++it) {
          const int s = it % kStages;
          const uint32_t ph = (uint32_t)(it / kStages) & 1u;
          if (it >= kStages && !mbar_wait(empty + s, ph ^ 1u)) { ok = false; break; }
          unsigned char* sa = smem + s * kStageBytes;
          mbar_expect_tx(full + s, kStageBytes);
          tma_load_2d(sa, &tmA, full + s, kb * kBK, m0);
          tma_load_2d(sa + kABytes, &tmB, full + s, kb * kBK, n0);
        }
      }
      if (!ok) {
        // drain this CTA's copies still in flight
        for (int j = max(0, it - kStages); j < it; ++j) mbar_wait(full + j % kStages, (uint32_t)(j / kStages) & 1u);
        atomicOr(g.err, 1u);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16(kBM, kBN);
      int it = 0, tl = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x, ++tl) {
        const int buf = tl & 1, use = tl >> 1;
        if (tl >= 2 && !mbar_wait(acce + buf, (uint32_t)(use - 1) & 1u)) { ok = false; break; }
        fence_after();
        const uint32_t acc = tmem + (uint32_t)(buf * kBN);
        for (int kb = 0; kb < KB; ++kb, ++it) {
          const int s = it % kStages;
          const uint32_t ph = (uint32_t)(it / kStages) & 1u;
          if (!mbar_wait(full + s, ph)) { ok = false; break; }
          fence_after();
          const uint32_t sa = smem_u32(smem + s * kStageBytes);
          const uint64_t ad = sw128_desc(sa), bd = sw128_desc(sa + kABytes);
#pragma unroll
          for (int k = 0; k < kBK / 16; ++k)
            mma_bf16(acc, ad + (uint64_t)(2 * k), bd + (uint64_t)(2 * k), idesc, (kb | k) ? 1u : 0u);
          mma_commit(empty + s);
        }
        mma_commit(accf + buf);  // also after a timeout: nothing is left in flight
      }
      if (!ok) atomicOr(g.err, 2u);
    }
    __syncwarp();
  } else {
    const int q = warp & 3;             // TMEM lane quadrant this warp may access
    const int half = (warp - 2) >> 2;   // the quadrant's two warps take alternate chunks
    int tl = 0;
    bool ok = true;
    for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x, ++tl) {
      const int buf = tl & 1, use = tl >> 1;
      const int m0 = g.m0 + (t % Mt) * kBM, n0 = (t / Mt) * kBN;
      const int gr = m0 + q * 32 + lane;
      const bool live = gr < g.m0 + g.M;
      // each epilogue warp keeps its own copy of the tile's bias (no
      // cross-warp barrier: a warp that gives up cannot stall the others)
      float* bias = s_bias + ((warp - 2) * 2 + buf) * kBN;
      {
        const int c = 4 * lane;
        const float4 bv = n0 + c < g.N ? *reinterpret_cast<const float4*>(g.bias + n0 + c) : make_float4(0.f, 0.f, 0.f, 0.f);
        *reinterpret_cast<float4*>(bias + c) = bv;
      }
      // this warp's chunks of the residual row segment are read while the MMAs run
      float4 xr[EPI == kEResid ? kBN / 8 : 1];
      if (EPI == kEResid && live) {
        const float4* xp = reinterpret_cast<const float4*>(static_cast<float*>(g.out) + (size_t)gr * g.ld + n0);
#pragma unroll
        for (int c2 = 0; c2 < kBN / 64; ++c2) {
          const int c = 2 * c2 + half;
#pragma unroll
          for (int i = 0; i < 8; ++i)
            if (n0 + 32 * c + 4 * i < g.N) xr[c2 * 8 + i] = xp[c * 8 + i];
        }
      }
      __syncwarp();  // the warp's bias copy is in place
      ok = __all_sync(0xffffffffu, mbar_wait(accf + buf, (uint32_t)use & 1u));
      if (!ok) {
        if (lane == 0) atomicOr(g.err, 4u);
        break;
      }
      fence_after();
      const uint32_t tbase = tmem + (uint32_t)(buf * kBN) + ((uint32_t)(q * 32) << 16);
      if (EPI == kEGlu) {
        // tile columns [64 p, 64 p + 32) are values, [64 p + 32, 64 p + 64) their gates;
        // group p = half of this warp
#pragma unroll
        for (int p = half; p < kBN / 64; p += 2) {
          __syncwarp();
          float a[32], b[32];
          tmem_ld32(tbase + (uint32_t)(64 * p), a);
          tmem_ld32(tbase + (uint32_t)(64 * p + 32), b);
          if (!live || n0 + 64 * p >= g.N) continue;
          const float* ba = bias + 64 * p;
          const float* bg = ba + 32;
          uint4* o = reinterpret_cast<uint4*>(static_cast<uint16_t*>(g.out) + (size_t)gr * g.ld + (n0 + 64 * p) / 2);
#pragma unroll
          for (int i = 0; i < 32; i += 8) {
            uint4 w;
            w.x = pack_bf16((a[i] + ba[i]) * sigm(b[i] + bg[i]), (a[i + 1] + ba[i + 1]) * sigm(b[i + 1] + bg[i + 1]));
            w.y = pack_bf16((a[i + 2] + ba[i + 2]) * sigm(b[i + 2] + bg[i + 2]),
                            (a[i + 3] + ba[i + 3]) * sigm(b[i + 3] + bg[i + 3]));
            w.z = pack_bf16((a[i + 4] + ba[i + 4]) * sigm(b[i + 4] + bg[i + 4]),
                            (a[i + 5] + ba[i + 5]) * sigm(b[i + 5] + bg[i + 5]));
            w.w = pack_bf16((a[i + 6] + ba[i + 6]) * sigm(b[i + 6] + bg[i + 6]),
                            (a[i + 7] + ba[i + 7]) * sigm(b[i + 7] + bg[i + 7]));
            o[i / 8] = w;
          }
        }
      } else {
#pragma unroll
        for (int c2 = 0; c2 < kBN / 64; ++c2) {
          const int c = 2 * c2 + half;
          __syncwarp();
          float v[32];
          tmem_ld32(tbase + (uint32_t)(c * 32), v);
          const int c0 = n0 + c * 32;
          if (!live || c0 >= g.N) continue;
          const float* bb = bias + c * 32;
#pragma unroll
          for (int i = 0; i < 32; ++i) v[i] += bb[i];
          if (EPI == kEInit || EPI == kEResid) {
            float4* xp = reinterpret_cast<float4*>(static_cast<float*>(g.out) + (size_t)gr * g.ld + c0);
#pragma unroll
            for (int i = 0; i < 32; i += 4) {
              float4 r = make_float4(v[i], v[i + 1], v[i + 2], v[i + 3]);
              if (EPI == kEResid) {
                const float4 o = xr[c2 * 8 + i / 4];
                r = make_float4(o.x + g.alpha * r.x, o.y + g.alpha * r.y, o.z + g.alpha * r.z, o.w + g.alpha * r.w);
              }
              xp[i / 4] = r;
            }
          } else {
            if (EPI == kESwish) {
#pragma unroll
              for (int i = 0; i < 32; ++i) v[i] = v[i] * sigm(v[i]);
            }
            uint4* o = reinterpret_cast<uint4*>(static_cast<uint16_t*>(g.out) + (size_t)gr * g.ld + c0);
#pragma unroll
            for (int i = 0; i < 32; i += 8)
              o[i / 8] = make_uint4(pack_bf16(v[i], v[i + 1]), pack_bf16(v[i + 2], v[i + 3]),
                                    pack_bf16(v[i + 4], v[i + 5]), pack_bf16(v[i + 6], v[i + 7]));
          }
        }
      }
      // this warp's reads of the accumulator are done: hand it back
      fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(acce + buf);
    }
  }
  fence_before();
  __syncthreads();
  if (warp == 1) {
    fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(2 * kBN) : "memory");
  }
}

template <int EPI>
void launch_one(const EGemm& g, const CUtensorMap& a, const CUtensorMap& b, cudaStream_t s) {
  const int tiles = ((g.M + kBM - 1) / kBM) * ((g.N + kBN - 1) / kBN);
  k_egemm<EPI><<<tiles < g_sms ? tiles : g_sms, kThreads, kSmem, s>>>(g, a, b);
}

}  // namespace

bool egemm_map_a(CUtensorMap* m, const uint16_t* A, int rows, int K) {
  return tc::make_map(m, A, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, K, rows, tc::kBK, tc::kBM);
}

bool egemm_map_b(CUtensorMap* m, const uint16_t* B, int rows, int K) {
  return tc::make_map(m, B, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, K, rows, tc::kBK, kBN);
}

cudaError_t egemm_prepare() {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&g_sms, cudaDevAttrMultiProcessorCount, dev);
  auto set = [&](const void* f) {
    if (e == cudaSuccess) e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmem);
  };
  set((const void*)k_egemm<kEInit>);
  set((const void*)k_egemm<kEResid>);
  set((const void*)k_egemm<kESwish>);
  set((const void*)k_egemm<kEPlain>);
  set((const void*)k_egemm<kEGlu>);
  return e;
}

void launch_egemm(int epi, const EGemm& g, const CUtensorMap& a, const CUtensorMap& b, cudaStream_t s) {
  switch (epi) {
    case kEInit: launch_one<kEInit>(g, a, b, s); break;
    case kEResid: launch_one<kEResid>(g, a, b, s); break;
    case kESwish: launch_one<kESwish>(g, a, b, s); break;
    case kEPlain: launch_one<kEPlain>(g, a, b, s); break;
    default: launch_one<kEGlu>(g, a, b, s); break;
  }
}

}  // namespace tsd
