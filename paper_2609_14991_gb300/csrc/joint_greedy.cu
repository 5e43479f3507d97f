// Joint GEMM on the tcgen05 tensor cores for greedy decoding with at most
// one n-gram LM, with one of two epilogues (the decoder option fusion_path).
//
// DENSE (fusion_path 1): per row r and label v of a 128 x BN tile the
// epilogue evaluates Eq. 1 up to the row's constant c_r (see row_fused.cu):
//   F0[v] = logit[v] + D[v] + lambda * dense0[u_r][v]
// with D the call's defaults (d.dvec) and u_r the dense LM row of the row's
// unigram state (d.c_info), and reduces the tile to one partial per row:
// softmax max and sum of the raw logits, and the best F0 over the labels not
// on the row's correction list (d.c_mask), ties to the lowest label.  The
// listed labels' raw logits are stored (d.logits) for the row pass.  The
// row's segment of its dense LM row is requested into L2 while the MMAs run
// and copied into the drained operand stages by one bulk copy per row once
// they have completed; the softmax pass runs while the copies land.
//
// Streaming (fusion_path 0): the epilogue writes logit + D[v] for every
// label (d.logits, through per-warp swizzled staging buffers and TMA
// stores) and the softmax partial; the row pass after it (row_stream.cu)
// adds the row's LM and trie terms and takes the argmax.
//
// Warp roles (320 threads): warp 0 TMA producer (A tile 128 x 64 and W_out
// tile BN x 64 per stage, 128-byte swizzle), warp 1 TMEM
// allocator and MMA issuer, warps 2-9 epilogue (thread = row; the two warps
// of a TMEM lane quadrant take alternate 32-column chunks).  Every wait on an
// mbarrier is bounded; on expiry the kernel records an error in the
// decoder's status word, drains its own copies and MMAs and returns.
#include <cuda.h>

#include "decoder.h"
#include "joint_tc.h"
#include "tc_common.cuh"

namespace tsd {

namespace {

using namespace tc;
constexpr int kEW = 4;                 // epilogue warps per TMEM lane quadrant
constexpr int kDEpi = 128 * kEW;       // epilogue threads: warps 2 .. 2 + 4 kEW - 1
constexpr int kDThreads = 64 + kDEpi;  // and the producer and MMA warps
constexpr float kNegInf = -__builtin_huge_valf();

// Shared memory: [operand stages][defaults D][barriers].  After the
// mainloop the stages hold the epilogue warps' exchange and, past it, either the
// rows' dense LM segments (rows 16 bytes apart beyond their BN floats, so
// that the 16-byte reads of eight consecutive rows fall in different bank
// groups) or the streaming epilogue's staging buffers (two 32 x 32 fp32
// boxes per warp).
template <int BN>
struct DSmem {
  static constexpr int kABytes = kBM * kBK * 2;
  static constexpr int kBBytes = BN * kBK * 2;
  static constexpr int kStageBytes = kABytes + kBBytes;
  static constexpr int kStages = BN == 256 ? 4 : (BN == 128 ? 5 : 8);
  static constexpr int kRowStride = BN * 4 + 16;
  static constexpr int kDenseOff = 10240;  // past the epilogue warps' exchange
  static constexpr int kCW = 32;            // columns per TMEM load in the epilogue
  static constexpr int kStageOff = 16384;   // streaming: staging buffers, two 32 x 32 boxes per warp
  static constexpr int kStageWarp = 2 * (kCW / 32) * 4096;
  static constexpr int kDOff = kStages * kStageBytes;
  static constexpr int kBarOff = kDOff + BN * 4;
  static constexpr int kBytes = kBarOff + 256 + 1024 /*align*/;
  static_assert(kBM * 4 * (kEW - 1) * 4 + 4 * 4 * kEW <= kDenseOff, "the exchange stays clear of the dense rows");
  static_assert(kDenseOff + kBM * kRowStride <= kStages * kStageBytes, "the dense rows fit the drained stages");
  static_assert(kStageOff + 4 * kEW * kStageWarp <= kStages * kStageBytes, "the staging buffers fit the drained stages");
  static_assert(kBytes <= 227 * 1024, "shared memory per CTA");
};

// Sum over a block of 2^(l[i] * log2 e - s2) in four independent accumulators.
template <int W>
__device__ __forceinline__ float sum_exp2_block(const float* l, float s2) {
  float a[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
  for (int i = 0; i < W; ++i) a[i & 3] += ex2_approx(fmaf(l[i], kLog2e, -s2));
  return (a[0] + a[1]) + (a[2] + a[3]);
}

// The maximum of a block by a tree (the block is left unchanged).
template <int W>
__device__ __forceinline__ float block_max(const float* v) {
  float t[W / 2];
#pragma unroll
  for (int i = 0; i < W / 2; ++i) t[i] = fmaxf(v[i], v[i + W / 2]);
#pragma unroll
  for (int w = W / 4; w > 0; w >>= 1)
#pragma unroll
    for (int i = 0; i < w; ++i) t[i] = fmaxf(t[i], t[i + w]);
  return t[0];
}

template <int N>
__device__ __forceinline__ uint32_t pick(const uint32_t (&a)[N], int k) {
  uint32_t v = a[0];
#pragma unroll
  for (int i = 1; i < N; ++i) v = (k == i) ? a[i] : v;
  return v;
}

template <int BN, bool DENSE>
__global__ void __launch_bounds__(kDThreads, 1)
    k_joint_greedy(DecView d, int step, const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const __grid_constant__ CUtensorMap tmLogits) {
  using S = DSmem<BN>;
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  float* sD = reinterpret_cast<float*>(smem + S::kDOff);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + S::kBarOff);
  uint64_t* empty = full + S::kStages;
  uint64_t* accum = empty + S::kStages;  // every MMA has completed
  uint64_t* dbar = accum + 1;            // the rows' dense segments have landed
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(dbar + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n0 = blockIdx.x * BN, m0 = blockIdx.y * kBM;
  const int M = d.params->n * d.K;
  const int KB = d.H / kBK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S::kStages; ++s) {
      mbar_init(full + s, 1);
      mbar_init(empty + s, 1);
    }
    mbar_init(accum, 1);
    mbar_init(dbar, kBM);  // one arrival per row
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(BN)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem = *tmem_slot;
  // W_out is constant: the first stages' tiles are requested before the
  // dependency wait (each stage's barrier expects its A tile as well)
  const int pre = min(KB, S::kStages);
  if (warp == 0 && lane == 0) {
    for (int kb = 0; kb < pre; ++kb) {
      mbar_expect_tx(full + kb, S::kStageBytes);
      tma_load_2d(smem + kb * S::kStageBytes + S::kABytes, &tmB, full + kb, kb * kBK, n0);
    }
  }
  // Programmatic dependent launch: the set-up above overlaps the row pass;
  // its outputs (joint input, correction list) are read after the wait.
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  if (warp == 0) {
    if (lane == 0) {
      bool ok = true;
      int issued = 0;
      for (int kb = 0; kb < KB; ++kb) {
        const int s = kb % S::kStages;
        const uint32_t ph = (uint32_t)(kb / S::kStages) & 1u;
        unsigned char* sa = smem + s * S::kStageBytes;
        if (kb < pre) {  // first use of the stage: W_out already requested
          tma_load_2d(sa, &tmA, full + s, kb * kBK, m0);
          ++issued;
          continue;
        }
        if (!mbar_wait(empty + s, ph ^ 1u, d.wait_ns)) { ok = false; break; }
        mbar_expect_tx(full + s, S::kStageBytes);
        tma_load_2d(sa, &tmA, full + s, kb * kBK, m0);
        tma_load_2d(sa + S::kABytes, &tmB, full + s, kb * kBK, n0);
        ++issued;
      }
      // never exit with copies in flight (the long limit)
      for (int kb = max(0, issued - S::kStages); kb < issued; ++kb)
        mbar_wait(full + kb % S::kStages, (uint32_t)(kb / S::kStages) & 1u);
      if (!ok) atomicOr(d.err, 1);
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      bool ok = true;
      const uint32_t idesc = idesc_bf16(kBM, BN);
      for (int kb = 0; kb < KB; ++kb) {
        const int s = kb % S::kStages;
        const uint32_t ph = (uint32_t)(kb / S::kStages) & 1u;
        if (!mbar_wait(full + s, ph, d.wait_ns)) { ok = false; break; }
        fence_after();
        const uint32_t sa = smem_u32(smem + s * S::kStageBytes);
        const uint64_t ad = sw128_desc(sa), bd = sw128_desc(sa + S::kABytes);
#pragma unroll
        for (int k = 0; k < kBK / 16; ++k)
          mma_bf16(tmem, ad + (uint64_t)(2 * k), bd + (uint64_t)(2 * k), idesc, (kb | k) ? 1u : 0u);
        mma_commit(empty + s);
      }
      // signals the epilogue once every issued MMA has completed (also after
      // a timeout, so nothing is in flight when TMEM is released)
      mma_commit(accum);
      if (!ok) atomicOr(d.err, 2);
    }
    __syncwarp();
  } else {
    // epilogue: thread = row of the tile; the kEW warps of a TMEM lane
    // quadrant take blocks of kCW columns in turn (one TMEM load each)
    constexpr int kCW = S::kCW;
    constexpr int kNB = BN / kCW;              // blocks per tile
    constexpr int kMyB = (kNB + kEW - 1) / kEW;  // blocks per warp, at most
    constexpr int kWB = kCW / 32;          // mask words and 32 x 32 store boxes per block
    const int q = warp & 3;  // TMEM lane quadrant this warp may access
    const int ehalf = (warp - 2) >> 2;  // this warp's turn among its quadrant's warps
    const int row = q * 32 + lane;
    const int gr = m0 + row;
    const bool live = gr < M;
    const int N = d.N, V4 = d.V4;
    float mx = kNegInf, se = 0.f, bv = kNegInf;
    int bi = INT_MAX;
    // while the MMAs run: the call's defaults of the tile's labels, lambda,
    // the row's dense LM row and mask words (written by the row pass before
    // this grid's wait)
    for (int i = (int)threadIdx.x - 64; i < BN; i += kDEpi) sD[i] = __ldcg(d.dvec + n0 + i);
    const float lam = d.params->lambda;
    uint32_t mw[kMyB * kWB];  // [block of this warp][word]
#pragma unroll
    for (int k = 0; k < kMyB * kWB; ++k) mw[k] = 0u;
    int uoff = -1;
    if (DENSE && live) {
      const int u = __ldcg(&d.c_info[gr].x);
      if (u >= 0 && u < d.lm.n_dense) uoff = u * V4;
      const uint32_t* mrow = d.c_mask + (size_t)gr * d.mask_words + n0 / 32;
#pragma unroll
      for (int k = 0; k < kMyB; ++k)
#pragma unroll
        for (int j = 0; j < kWB; ++j)
          if (ehalf + kEW * k < kNB) mw[k * kWB + j] = __ldcg(mrow + (ehalf + kEW * k) * kWB + j);
    }
    unsigned char* drow = smem + S::kDenseOff + row * S::kRowStride;
    const int seg = min(BN, V4 - n0);  // labels of the tile inside the dense rows
    if (DENSE && ehalf == 0 && uoff >= 0 && seg > 0) {  // the row's segment into L2 while the MMAs run
      asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(d.lm.dense0 + uoff + n0), "r"((uint32_t)seg * 4u)
                   : "memory");
    }
    asm volatile("bar.sync 2, %0;" ::"n"(kDEpi) : "memory");  // sD complete
    bool ok = __all_sync(0xffffffffu, mbar_wait(accum, 0, d.wait_ns));  // tcgen05.ld wants the warp whole
    if (!ok && lane == 0) atomicOr(d.err, 4);
    fence_after();
    // the row's segment into the drained stages (every MMA has completed) by
    // one bulk copy, and the row's arrival on dbar (with the copy's bytes)
    if (DENSE && ehalf == 0) {
      if (ok && uoff >= 0 && seg > 0) {
        mbar_expect_tx(dbar, (uint32_t)seg * 4u);
        bulk_g2s(drow, d.lm.dense0 + uoff + n0, (uint32_t)seg * 4u, dbar);
      } else {
        mbar_arrive(dbar);
      }
    }
    const uint32_t tbase = tmem + ((uint32_t)(q * 32) << 16);
    if (ok) {
      // pass 1 (DENSE: while the copies land): the softmax partial of the
      // raw logits; DENSE: the listed labels' logits go out for the row
      // pass; streaming: logit + D of every label goes out
#pragma unroll 1
      for (int k = 0; k < kMyB; ++k) {
        const int b = ehalf + kEW * k;
        if (b >= kNB) break;
        __syncwarp();
        const int c0 = n0 + b * kCW;
        float l[kCW];
        tmem_ld<kCW>(tbase + (uint32_t)(b * kCW), l);
        if (c0 + kCW > N) {
#pragma unroll
          for (int i = 0; i < kCW; ++i)
            if (c0 + i >= N) l[i] = kNegInf;
        }
        const float cm = block_max<kCW>(l);
        if (cm != kNegInf) {
          const float m2 = fmaxf(mx, cm);
          const float s2 = m2 * kLog2e;
          float acc = (mx == kNegInf) ? 0.f : se * ex2_approx(mx * kLog2e - s2);
          acc += sum_exp2_block<kCW>(l, s2);
          se = acc;
          mx = m2;
        }
        if (d.cap_logits && step < d.cap_steps && live) {
          float* cl = d.cap_logits + ((size_t)step * M + gr) * N;
#pragma unroll
          for (int i = 0; i < kCW; ++i)
            if (c0 + i < N) cl[c0 + i] = l[i];
        }
        if constexpr (DENSE) {
#pragma unroll
          for (int j = 0; j < kWB; ++j) {
            const uint32_t mk = pick(mw, k * kWB + j);
            if (mk) {
              float* lo = d.logits + (size_t)gr * d.N_pad + c0 + 32 * j;
#pragma unroll
              for (int i = 0; i < 32; ++i)
                if ((mk >> i) & 1u) lo[i] = l[32 * j + i];
            }
          }
        } else {
          // the warp's 32-row boxes of logit + D by TMA stores from staging
          // buffers in the drained stages (two sets per warp, alternating by
          // block; the 128-byte swizzle keeps the row-per-thread writes
          // conflict-free)
          const float4* dv4 = reinterpret_cast<const float4*>(sD + b * kCW);
#pragma unroll
          for (int j = 0; j < kCW / 4; ++j) {
            const float4 dq = dv4[j];
            l[4 * j] += dq.x; l[4 * j + 1] += dq.y; l[4 * j + 2] += dq.z; l[4 * j + 3] += dq.w;
          }
          unsigned char* stg = smem + S::kStageOff + (warp - 2) * S::kStageWarp + (k & 1) * kWB * 4096;
          if (lane == 0) tma_store_wait_read<kWB>();  // the stores of two blocks ago have read this set
          __syncwarp();
#pragma unroll
          for (int j = 0; j < kWB; ++j)
#pragma unroll
            for (int e = 0; e < 8; ++e)
              *reinterpret_cast<float4*>(stg + j * 4096 + lane * 128 + ((e ^ (lane & 7)) << 4)) =
                  make_float4(l[32 * j + 4 * e], l[32 * j + 4 * e + 1], l[32 * j + 4 * e + 2], l[32 * j + 4 * e + 3]);
          fence_async_smem();
          __syncwarp();
          if (lane == 0) {
#pragma unroll
            for (int j = 0; j < kWB; ++j) {
              tma_store_2d(&tmLogits, stg + j * 4096, c0 + 32 * j, m0 + q * 32);
              tma_store_commit();
            }
          }
        }
      }
      if (DENSE) {
        ok = __all_sync(0xffffffffu, mbar_wait(dbar, 0, d.wait_ns));
        if (!ok && lane == 0) atomicOr(d.err, 64);
      }
    }
    if (DENSE && ok) {
      // pass 2: F0 = logit + D + lambda * dense0[u] of the unlisted labels and
      // the tile's best of them
#pragma unroll 1
      for (int k = 0; k < kMyB; ++k) {
        const int b = ehalf + kEW * k;
        if (b >= kNB) break;
        __syncwarp();
        const int c0 = n0 + b * kCW;
        float l[kCW];
        tmem_ld<kCW>(tbase + (uint32_t)(b * kCW), l);
        if (c0 + kCW > N) {
#pragma unroll
          for (int i = 0; i < kCW; ++i)
            if (c0 + i >= N) l[i] = kNegInf;
        }
        const float4* dv4 = reinterpret_cast<const float4*>(sD + b * kCW);
#pragma unroll
        for (int j = 0; j < kCW / 4; ++j) {
          const float4 dq = dv4[j];
          float4 xq = make_float4(0.f, 0.f, 0.f, 0.f);
          if (uoff >= 0 && b * kCW + 4 * j < seg) xq = *reinterpret_cast<const float4*>(drow + (b * kCW + 4 * j) * 4);
          l[4 * j] += fmaf(lam, xq.x, dq.x);
          l[4 * j + 1] += fmaf(lam, xq.y, dq.y);
          l[4 * j + 2] += fmaf(lam, xq.z, dq.z);
          l[4 * j + 3] += fmaf(lam, xq.w, dq.w);
        }
#pragma unroll
        for (int j = 0; j < kWB; ++j) {
          const uint32_t mk = pick(mw, k * kWB + j);
          if (mk) {
#pragma unroll
            for (int i = 0; i < 32; ++i)
              if ((mk >> i) & 1u) l[32 * j + i] = kNegInf;
          }
        }
        const float fm = block_max<kCW>(l);
        if (fm > bv) {
          int jx = kCW - 1;
#pragma unroll
          for (int i = kCW - 1; i >= 0; --i)
            if (l[i] == fm) jx = i;
          bv = fm;
          bi = c0 + jx;
        }
      }
    }
    // never leave with MMAs still writing the accumulator or row copies still
    // landing (the long limit whatever wait_ns is)
    if (warp == 2 && lane == 0) {
      mbar_wait(accum, 0);
      if (DENSE) mbar_wait(dbar, 0);
    }
    // the staging buffers must have been read before the CTA's shared memory
    // goes; the stores' writes complete with the grid (the row pass reads
    // them after its dependency wait)
    if (!DENSE && lane == 0) tma_store_wait_read<0>();
    __syncwarp();
    // merge the quadrant's warps' partials of each row: warps 1..kEW-1 of the
    // quadrant leave theirs in the drained stages, warp 0 combines and stores
    float* xbase = reinterpret_cast<float*>(smem);
    int* xok = reinterpret_cast<int*>(xbase + kBM * 4 * (kEW - 1));  // [quadrant][warp 1..]
    if (ehalf > 0) {
      float* xch = xbase + (row * (kEW - 1) + ehalf - 1) * 4;
      if (ok) {
        xch[0] = mx;
        xch[1] = se;
        xch[2] = bv;
        xch[3] = __int_as_float(bi);
      }
      if (lane == 0) xok[q * (kEW - 1) + ehalf - 1] = ok ? 1 : 0;
    }
    asm volatile("bar.sync 1, %0;" ::"n"(kDEpi) : "memory");
    if (ehalf == 0 && ok && live) {
      bool all = true;
#pragma unroll
      for (int e = 1; e < kEW; ++e) {
        if (!xok[q * (kEW - 1) + e - 1]) {
          all = false;
          continue;
        }
        const float* xch = xbase + (row * (kEW - 1) + e - 1) * 4;
        const float m1 = xch[0], s1 = xch[1];
        if (m1 != kNegInf) {
          if (mx == kNegInf) {
            mx = m1;
            se = s1;
          } else {
            const float m2 = fmaxf(mx, m1);
            se = se * ex2_approx((mx - m2) * kLog2e) + s1 * ex2_approx((m1 - m2) * kLog2e);
            mx = m2;
          }
        }
        const float v1 = xch[2];
        const int i1 = __float_as_int(xch[3]);
        if (v1 > bv || (v1 == bv && i1 < bi)) { bv = v1; bi = i1; }
      }
      if (all) d.part[(size_t)gr * d.n_ptiles + blockIdx.x] = make_float4(mx, se, bv, __int_as_float(bi));
    }
  }
  fence_before();
  __syncthreads();
  if (warp == 1) {
    fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(BN) : "memory");
  }
}

}  // namespace

cudaError_t joint_greedy_prepare(int bn) {
  const auto attr = cudaFuncAttributeMaxDynamicSharedMemorySize;
  cudaError_t e = cudaSuccess;
  if (bn == 256) {
    e = cudaFuncSetAttribute(k_joint_greedy<256, true>, attr, DSmem<256>::kBytes);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_joint_greedy<256, false>, attr, DSmem<256>::kBytes);
  } else if (bn == 128) {
    e = cudaFuncSetAttribute(k_joint_greedy<128, true>, attr, DSmem<128>::kBytes);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_joint_greedy<128, false>, attr, DSmem<128>::kBytes);
  } else {
    e = cudaFuncSetAttribute(k_joint_greedy<64, true>, attr, DSmem<64>::kBytes);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_joint_greedy<64, false>, attr, DSmem<64>::kBytes);
  }
  return e;
}

namespace {
template <int BN>
void launch_greedy_bn(cudaLaunchConfig_t& cfg, const JointTc& jt, const DecView& d, int step) {
  cfg.dynamicSmemBytes = DSmem<BN>::kBytes;
  if (d.fz_dense) cudaLaunchKernelEx(&cfg, k_joint_greedy<BN, true>, d, step, jt.mapA, jt.mapB, jt.mapLogits);
  else cudaLaunchKernelEx(&cfg, k_joint_greedy<BN, false>, d, step, jt.mapA, jt.mapB, jt.mapLogits);
}
}  // namespace

void launch_joint_greedy(const JointTc& jt, const DecView& d, int M, int step, cudaStream_t s, bool pdl) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(d.N_pad / jt.bn, (M + kBM - 1) / kBM);
  cfg.blockDim = dim3(kDThreads);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  if (jt.bn == 256) launch_greedy_bn<256>(cfg, jt, d, step);
  else if (jt.bn == 128) launch_greedy_bn<128>(cfg, jt, d, step);
  else launch_greedy_bn<64>(cfg, jt, d, step);
}

}  // namespace tsd
