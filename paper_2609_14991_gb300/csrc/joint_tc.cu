// Joint GEMM on the 5th-generation tensor cores (tcgen05) with the fused
// selection epilogue.
//
// logits[r][v] = sum_k A[r][k] * Wt[v][k]: A (joint input, bf16 [M][H]) and
// Wt (W_out label-major, bf16 [N_pad][H]) are both K-major, loaded by TMA
// into 128-byte-swizzled shared-memory stages; one elected thread issues
// tcgen05.mma (kind::f16, bf16 x bf16 -> fp32) into a 128 x BN accumulator in
// tensor memory.  Eight epilogue warps read the accumulator back with
// tcgen05.ld (thread = row; two warps per 32-lane quadrant take alternate
// 32-column chunks) and reduce it on chip to the row's selection partial for
// this tile: softmax max and sum over the real labels, and the best fused
// value logit + bias (the dense fusion bias row of several LMs), ties to the
// lowest label, or (BEAM) the tile's top K.  Greedy decoding with at most one
// LM runs joint_greedy.cu instead.  Logits never leave the SM.
//
// Warp roles (320 threads): warp 0 TMA producer, warp 1 TMEM allocator and
// MMA issuer, warps 2-9 epilogue.  Every wait on an mbarrier is bounded in
// time; on expiry the kernel records an error in the decoder's status word,
// drains its own copies and returns.
#include <cuda.h>

#include "decoder.h"
#include "joint_tc.h"
#include "tc_common.cuh"

namespace tsd {

namespace {

using namespace tc;  // kBM, kBK and the tcgen05 / TMA helpers
constexpr int kThreads = 320;
constexpr int kEpiThreads = 256;  // warps 2-9
constexpr float kNegInf = -__builtin_huge_valf();
// Shared memory: [operand stages][bias boxes][barriers].  With a fusion
// bias (several LMs), the bias of the tile (128 rows x BN fp32) arrives by
// TMA in 128 x 32 boxes with the 128-byte swizzle while the mainloop runs;
// at BN = 256 only the first half has its own buffer and the second half
// lands in the drained stages.
template <int BN>
struct Smem {
  static constexpr int kStages = (BN == 256) ? 3 : (BN == 128 ? 4 : 8);
  static constexpr int kABytes = kBM * kBK * 2;
  static constexpr int kBBytes = BN * kBK * 2;
  static constexpr int kStageBytes = kABytes + kBBytes;
  static constexpr int kBoxBytes = kBM * 32 * 4;
  static constexpr int kBoxes = BN / 32;
  static constexpr int kEarly = (BN == 256) ? 4 : kBoxes;
  static constexpr int kBiasBytes = kEarly * kBoxBytes;
  static constexpr int kBytes = kStages * kStageBytes + kBiasBytes + 1024 /*align*/ + 256 /*barriers*/;
  static_assert((kBoxes - kEarly) * kBoxBytes <= kStages * kStageBytes, "late bias boxes fit the stages");
  // the epilogue halves' exchange (per row 18 floats, 4 flags) after the late boxes
  static_assert((kBoxes - kEarly) * kBoxBytes + kBM * 18 * 4 + 16 <= kStages * kStageBytes, "exchange fits");
};

// Sum over a chunk of 2^(l[i] * log2 e - s2) in four independent
// accumulators (a single running sum would chain 32 dependent adds).
__device__ __forceinline__ float sum_exp2_32(const float* l, float s2) {
  float a[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
  for (int i = 0; i < 32; ++i) a[i & 3] += ex2_approx(fmaf(l[i], kLog2e, -s2));
  return (a[0] + a[1]) + (a[2] + a[3]);
}

// BEAM: instead of the single best fused label, each row keeps the top-K
// (K = d.topk <= 8: the beam width, or the pruned-fusion candidate count)
// values of the tile, ties to the lower label.  With pruned fusion (d.prune)
// the values are the plain logits: no bias tile is loaded.
template <int BN, bool BEAM>
__global__ void __launch_bounds__(kThreads, 1)
    k_joint_tc(DecView d, int step, const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
               const __grid_constant__ CUtensorMap tmBias) {
  using S = Smem<BN>;
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  unsigned char* bias_early = smem + S::kStages * S::kStageBytes;
  uint64_t* full = reinterpret_cast<uint64_t*>(bias_early + S::kBiasBytes);
  uint64_t* empty = full + S::kStages;
  uint64_t* accum = empty + S::kStages;
  uint64_t* biasbar = accum + 1;  // [0] early boxes, [1] late boxes
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(biasbar + 2);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n0 = blockIdx.x * BN, m0 = blockIdx.y * kBM;
  const bool use_bias = !(BEAM && d.prune);
  const int M = d.params->n * d.K;
  const int KB = d.H / kBK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S::kStages; ++s) {
      mbar_init(full + s, 1);
      mbar_init(empty + s, 1);
    }
    mbar_init(accum, 1);
    mbar_init(biasbar, 1);
    mbar_init(biasbar + 1, 1);
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
  bool ok = true;
  // W_out is constant, so the first stages' W_out tiles are requested before
  // the dependency wait (each stage's barrier expects its A tile as well).
  const int pre = min(KB, S::kStages);
  if (warp == 0 && lane == 0) {
    for (int kb = 0; kb < pre; ++kb) {
      mbar_expect_tx(full + kb, S::kStageBytes);
      tma_load_2d(smem + kb * S::kStageBytes + S::kABytes, &tmB, full + kb, kb * kBK, n0);
    }
  }
  // Programmatic dependent launch: the set-up above overlaps the row pass;
  // its outputs (joint input, bias) are read only after the wait.  The next
  // row pass may launch once every CTA is past this point.
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  if (warp == 0) {
    if (lane == 0) {
      // the bias tile first: the epilogue needs it as soon as the MMAs end
      if (use_bias) {
        mbar_expect_tx(biasbar, S::kEarly * S::kBoxBytes);
        for (int c = 0; c < S::kEarly; ++c)
          tma_load_2d(bias_early + c * S::kBoxBytes, &tmBias, biasbar, n0 + 32 * c, m0);
      }
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
      // Never exit with copies in flight: wait for the last use of every
      // stage (its final phase; complete already when the MMAs consumed it,
      // as they do unless a wait expired), with the long limit.
      for (int kb = max(0, issued - S::kStages); kb < issued; ++kb)
        mbar_wait(full + kb % S::kStages, (uint32_t)(kb / S::kStages) & 1u);
      if (!ok) atomicOr(d.err, 1);
    }
    __syncwarp();  // reconverge before the CTA barrier below (bar.sync is warp-aligned)
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16(kBM, BN);
      for (int kb = 0; kb < KB; ++kb) {
        const int s = kb % S::kStages;
        const uint32_t ph = (uint32_t)(kb / S::kStages) & 1u;
        if (!mbar_wait(full + s, ph, d.wait_ns)) { ok = false; break; }
        fence_after();
        const uint32_t sa = smem_u32(smem + s * S::kStageBytes);
        const uint64_t ad = sw128_desc(sa), bd = sw128_desc(sa + S::kABytes);
#pragma unroll
        for (int k = 0; k < kBK / 16; ++k)  // K = 16 per instruction: +32 bytes in the swizzle atom
          mma_bf16(tmem, ad + (uint64_t)(2 * k), bd + (uint64_t)(2 * k), idesc, (kb | k) ? 1u : 0u);
        mma_commit(empty + s);
      }
      // signals the epilogue once every issued MMA has completed (also after a
      // timeout, so nothing is in flight when TMEM is released)
      mma_commit(accum);
      if (!ok) atomicOr(d.err, 2);
    }
    __syncwarp();
  } else {
    // epilogue: warps 2..9, thread = row of the tile; the two warps of a
    // TMEM lane quadrant take alternate 32-column chunks
    const int q = warp & 3;  // TMEM lane quadrant this warp may access
    const int half = (warp - 2) >> 2;
    const int row = q * 32 + lane;
    const int gr = m0 + row;
    const bool live = gr < M;
    const int N = d.N;
    float mx = kNegInf, se = 0.f, bv = kNegInf;
    int bi = INT_MAX;
    const int K = d.topk;
    float tv[8];
    int ti[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) { tv[j] = kNegInf; ti[j] = INT_MAX; }
    float tmin = kNegInf;  // tv[K-1]
    ok = __all_sync(0xffffffffu, mbar_wait(accum, 0, d.wait_ns));  // warp-uniform: tcgen05.ld is .sync.aligned
    if (!ok && lane == 0) atomicOr(d.err, 4);
    fence_after();
    // the second half of a 256-wide bias tile goes into the drained stages
    // (every MMA has completed, so nothing reads them any more)
    const bool late = ok && use_bias && S::kEarly < S::kBoxes;
    if (late && warp == 2 && lane == 0) {
      mbar_expect_tx(biasbar + 1, (S::kBoxes - S::kEarly) * S::kBoxBytes);
      for (int c = S::kEarly; c < S::kBoxes; ++c)
        tma_load_2d(smem + (c - S::kEarly) * S::kBoxBytes, &tmBias, biasbar + 1, n0 + 32 * c, m0);
    }
    const bool have_early = use_bias ? __all_sync(0xffffffffu, mbar_wait(biasbar, 0, d.wait_ns)) : true;
    if (!have_early) {
      ok = false;
      if (lane == 0) atomicOr(d.err, 16);
    }
    bool late_done = !late;
    if (ok) {
      const uint32_t tbase = tmem + ((uint32_t)(q * 32) << 16);
      const int sw = row & 7;  // 128-byte swizzle: 16-byte chunk j of a row sits at j ^ (row % 8)
#pragma unroll 1
      for (int c = half; c < BN / 32; c += 2) {
        __syncwarp();  // the per-chunk selection branches; tcgen05.ld wants the warp whole
        if (use_bias && c >= S::kEarly && !late_done) {
          late_done = true;
          if (!__all_sync(0xffffffffu, mbar_wait(biasbar + 1, 0, d.wait_ns))) {
            if (lane == 0) atomicOr(d.err, 32);
            break;
          }
        }
        const unsigned char* box = (c < S::kEarly) ? bias_early + c * S::kBoxBytes : smem + (c - S::kEarly) * S::kBoxBytes;
        float b[32];
        if (use_bias) {
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            const float4 v = *reinterpret_cast<const float4*>(box + row * 128 + ((j ^ sw) << 4));
            b[4 * j] = v.x; b[4 * j + 1] = v.y; b[4 * j + 2] = v.z; b[4 * j + 3] = v.w;
          }
        } else {
#pragma unroll
          for (int j = 0; j < 32; ++j) b[j] = 0.f;
        }
        float l[32];
        tmem_ld32(tbase + (uint32_t)(c * 32), l);
        const int c0 = n0 + c * 32;
        // Labels at or past V+1 (padding of the last tile) take no part:
        // their logit becomes -inf.  Blank (label V) has bias 0 in the row.
        if (c0 + 32 > N) {
#pragma unroll
          for (int i = 0; i < 32; ++i)
            if (c0 + i >= N) l[i] = kNegInf;
        }
        // fused values f = logit + bias (reuse b), chunk maxima by trees
        float t[16], u[16];
#pragma unroll
        for (int i = 0; i < 32; ++i) b[i] += l[i];
#pragma unroll
        for (int i = 0; i < 16; ++i) { t[i] = fmaxf(l[i], l[i + 16]); u[i] = fmaxf(b[i], b[i + 16]); }
#pragma unroll
        for (int w = 8; w > 0; w >>= 1)
#pragma unroll
          for (int i = 0; i < w; ++i) { t[i] = fmaxf(t[i], t[i + w]); u[i] = fmaxf(u[i], u[i + w]); }
        const float cm = t[0], fm = u[0];
        if (!BEAM) {
          // the first label of the chunk holding the chunk's best fused value
          if (fm > bv) {
            int j = 31;
#pragma unroll
            for (int i = 31; i >= 0; --i)
              if (b[i] == fm) j = i;
            bv = fm;
            bi = c0 + j;
          }
        } else if (fm > tmin) {
          // Take the chunk's values in decreasing order while they beat the
          // K-th kept value: at most K rounds, usually none after the first
          // chunks.  Each round finds the first (lowest-label) position of the
          // chunk maximum, bubbles it into the sorted list (an equal value
          // already kept stays ahead: it has the lower label), masks it out
          // and takes the next maximum.
          float cmx = fm;
#pragma unroll 1
          for (int it = 0; it < K && cmx > tmin; ++it) {
            int jx = 31;
#pragma unroll
            for (int i = 31; i >= 0; --i)
              if (b[i] == cmx) jx = i;
            float cv = cmx;
            int ci = c0 + jx;
#pragma unroll
            for (int j = 0; j < 8; ++j) {
              if (j < K && cv > tv[j]) {
                const float tf = tv[j]; tv[j] = cv; cv = tf;
                const int tk = ti[j]; ti[j] = ci; ci = tk;
              }
            }
#pragma unroll
            for (int j = 0; j < 8; ++j)
              if (j == K - 1) tmin = tv[j];
#pragma unroll
            for (int i = 0; i < 32; ++i)
              if (i == jx) b[i] = kNegInf;
#pragma unroll
            for (int i = 0; i < 16; ++i) u[i] = fmaxf(b[i], b[i + 16]);
#pragma unroll
            for (int w = 8; w > 0; w >>= 1)
#pragma unroll
              for (int i = 0; i < w; ++i) u[i] = fmaxf(u[i], u[i + w]);
            cmx = u[0];
          }
        }
        if (cm != kNegInf) {
          // online softmax partial: sum of 2^((logit - max) * log2 e)
          const float m2 = fmaxf(mx, cm);
          const float s2 = m2 * kLog2e;
          float acc = (mx == kNegInf) ? 0.f : se * ex2_approx(mx * kLog2e - s2);
          acc += sum_exp2_32(l, s2);
          se = acc;
          mx = m2;
        }
        if (d.cap_logits && step < d.cap_steps && live) {
          float* cl = d.cap_logits + ((size_t)step * M + gr) * N;
#pragma unroll
          for (int i = 0; i < 32; ++i)
            if (c0 + i < N) cl[c0 + i] = l[i];
        }
      }
    }
    // never leave with bias boxes still landing in shared memory or MMAs
    // still writing the accumulator (these drains keep the long limit
    // whatever wait_ns is)
    if (!late_done && warp == 2 && lane == 0) mbar_wait(biasbar + 1, 0);
    if (!have_early && warp == 2 && lane == 0) mbar_wait(biasbar, 0);
    if (warp == 2 && lane == 0) mbar_wait(accum, 0);
    __syncwarp();
    // Merge the two halves' partials of each row: the second half leaves its
    // partial in shared memory past the late bias boxes (the stages are
    // drained: every MMA has completed), the first half combines and stores.
    float* xbase = reinterpret_cast<float*>(smem + (S::kBoxes - S::kEarly) * S::kBoxBytes);
    float* xch = xbase + row * 18;  // (max, sum, then best or top-8 (value, label))
    int* xok = reinterpret_cast<int*>(xbase + kBM * 18);  // per quadrant: the second half finished
    if (half == 1) {
      if (ok) {
        xch[0] = mx;
        xch[1] = se;
        if (!BEAM) {
          xch[2] = bv;
          xch[3] = __int_as_float(bi);
        } else {
#pragma unroll
          for (int j = 0; j < 8; ++j) { xch[2 + 2 * j] = tv[j]; xch[3 + 2 * j] = __int_as_float(ti[j]); }
        }
      }
      if (lane == 0) xok[q] = ok ? 1 : 0;
    }
    asm volatile("bar.sync 1, %0;" ::"n"(kEpiThreads) : "memory");
    if (half == 0 && ok && xok[q] && live) {
      const float m1 = xch[0], s1 = xch[1];
      if (m1 != kNegInf) {
        if (mx == kNegInf) { mx = m1; se = s1; }
        else {
          const float m2 = fmaxf(mx, m1);
          se = se * ex2_approx((mx - m2) * kLog2e) + s1 * ex2_approx((m1 - m2) * kLog2e);
          mx = m2;
        }
      }
      if (!BEAM) {
        const float v1 = xch[2];
        const int i1 = __float_as_int(xch[3]);
        if (v1 > bv || (v1 == bv && i1 < bi)) { bv = v1; bi = i1; }
        d.part[(size_t)gr * d.n_ptiles + blockIdx.x] = make_float4(mx, se, bv, __int_as_float(bi));
      } else {
        // merge two lists sorted by (value desc, label asc): an entry's
        // place is its index plus the other list's entries ordered before it
        // (unfilled entries (-inf, INT_MAX) of both lists land on the same
        // trailing places with the same contents)
        float2* bp = d.bpart + ((size_t)gr * d.n_ptiles + blockIdx.x) * (1 + K);
        bp[0] = make_float2(mx, se);
        float ov[8];
        int oi[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) { ov[j] = xch[2 + 2 * j]; oi[j] = __float_as_int(xch[3 + 2 * j]); }
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          if (i < K) {
            int pa = i, pb = i;
#pragma unroll
            for (int j = 0; j < 8; ++j) {
              if (j < K) {
                pa += (ov[j] > tv[i] || (ov[j] == tv[i] && oi[j] < ti[i])) ? 1 : 0;
                pb += (tv[j] > ov[i] || (tv[j] == ov[i] && ti[j] < oi[i])) ? 1 : 0;
              }
            }
            if (pa < K) bp[1 + pa] = make_float2(tv[i], __int_as_float(ti[i]));
            if (pb < K) bp[1 + pb] = make_float2(ov[i], __int_as_float(oi[i]));
          }
        }
      }
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

unsigned long long tc_wait_ns_default() { return kWaitNs; }

int joint_tc_pick_bn(int M_max, int N_pad, int sms) {
  // wider tiles re-read fewer operands; take the widest whose tiles still
  // cover ~80% of the SMs (measured: 256 at 1024 x 4352, 64 at 256 x 1280)
  const int mt = (M_max + kBM - 1) / kBM;
  if (mt * (N_pad / 256) * 5 >= sms * 4) return 256;
  if (mt * (N_pad / 128) * 5 >= sms * 4) return 128;
  return 64;
}

cudaError_t joint_tc_prepare(JointTc* jt, const uint16_t* A, int M_pad, const uint16_t* Wt, int N_pad, int H, int bn,
                             const float* bias, const float* logits) {
  jt->bn = bn;
  if (!make_map(&jt->mapA, A, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, H, M_pad, kBK, kBM)) return cudaErrorInvalidValue;
  if (!make_map(&jt->mapB, Wt, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, H, N_pad, kBK, bn)) return cudaErrorInvalidValue;
  if (!make_map(&jt->mapBias, bias, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, N_pad, M_pad, 32, kBM))
    return cudaErrorInvalidValue;
  if (!make_map(&jt->mapLogits, logits ? logits : bias, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, N_pad, M_pad, 32, 32))
    return cudaErrorInvalidValue;
  const auto attr = cudaFuncAttributeMaxDynamicSharedMemorySize;
  cudaError_t e = cudaSuccess;
  if (bn == 256) {
    e = cudaFuncSetAttribute(k_joint_tc<256, false>, attr, Smem<256>::kBytes);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_joint_tc<256, true>, attr, Smem<256>::kBytes);
  } else if (bn == 128) {
    e = cudaFuncSetAttribute(k_joint_tc<128, false>, attr, Smem<128>::kBytes);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_joint_tc<128, true>, attr, Smem<128>::kBytes);
  } else {
    e = cudaFuncSetAttribute(k_joint_tc<64, false>, attr, Smem<64>::kBytes);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_joint_tc<64, true>, attr, Smem<64>::kBytes);
  }
  if (e == cudaSuccess) e = joint_greedy_prepare(bn);
  return e;
}

namespace {
template <int BN>
void launch_bn(cudaLaunchConfig_t& cfg, const JointTc& jt, const DecView& d, int step) {
  const bool beam = d.topk > 1 || d.prune > 0;  // the top-K epilogue
  cfg.dynamicSmemBytes = Smem<BN>::kBytes;
  if (beam) cudaLaunchKernelEx(&cfg, k_joint_tc<BN, true>, d, step, jt.mapA, jt.mapB, jt.mapBias);
  else cudaLaunchKernelEx(&cfg, k_joint_tc<BN, false>, d, step, jt.mapA, jt.mapB, jt.mapBias);
}
}  // namespace

void launch_joint_tc(const JointTc& jt, const DecView& d, int M, int step, cudaStream_t s, bool pdl) {
  if (d.fused) {
    launch_joint_greedy(jt, d, M, step, s, pdl);
    return;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(d.N_pad / jt.bn, (M + kBM - 1) / kBM);
  cfg.blockDim = dim3(kThreads);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  if (jt.bn == 256) launch_bn<256>(cfg, jt, d, step);
  else if (jt.bn == 128) launch_bn<128>(cfg, jt, d, step);
  else launch_bn<64>(cfg, jt, d, step);
}

}  // namespace tsd
