// Arbitration at draft/target mismatches (Sec. 3.3 of the paper).
//
// One warp per sequence; lane i-1 owns draft position i (K <= 31).
// Delta_i = 1[y_hat_i = y_tilde_i] (Eq. 3).  Matches are forced accepted
// (z_tilde = +inf, Eq. 13-14).  At a mismatch the policy probability is
// sigma(z_i) with z_i from a one-hidden-layer feature MLP standing in for the
// head g_phi of Eq. 11, or 0 / 1 for the forced "always target" / "always
// draft" policies, and the action is 1[p > lambda] (Eq. 17).  All z_i of a
// round are independent of the round's actions (the arbitrator input of Eq. 9
// holds none), so they are evaluated in parallel: for each position the
// warp's lanes split the hidden units and sum with shuffles.
#include <math.h>

#include "cospec_device.cuh"
#include "cospec_internal.h"

namespace cospec {

namespace {

constexpr int WARPS = 4;
constexpr int NF = 8;

__global__ void __launch_bounds__(WARPS * 32)
    arbitrate_kernel(int B, int K, const int32_t* __restrict__ draft,
                     const int32_t* __restrict__ argmax, const float* __restrict__ stats, int H,
                     const float* __restrict__ w1, const float* __restrict__ b1,
                     const float* __restrict__ w2, float b2, float lambda, int mode,
                     float* __restrict__ p_out, uint8_t* __restrict__ accept) {
  extern __shared__ float sm[];            // w1 [H][8], b1 [H], w2 [H] when mode == 0
  __shared__ float feat[WARPS][32][NF];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // The MLP weights do not come from the previous kernel: stage them while
  // it finishes, then wait for its statistics.
  if (mode == 0) {
    // unrolled so that several loads of a thread are in flight at once
#pragma unroll 8
    for (int e = threadIdx.x; e < H * NF; e += blockDim.x) sm[e] = __ldg(w1 + e);
#pragma unroll 4
    for (int e = threadIdx.x; e < H; e += blockDim.x) {
      sm[H * NF + e] = __ldg(b1 + e);
      sm[H * NF + H + e] = __ldg(w2 + e);
    }
  }
  griddep_wait();
  griddep_launch_dependents();
  if (mode == 0) __syncthreads();
  const int b = blockIdx.x * WARPS + warp;
  if (b >= B) return;

  const int R = K + 1;
  const bool act = lane < K;
  const int dft = act ? draft[(size_t)b * K + lane] : -1;
  const int tgt = act ? argmax[(size_t)b * R + lane] : -2;
  const bool match = act && (dft == tgt);
  const unsigned mball = __ballot_sync(0xffffffffu, match);
  const unsigned actmask = (K >= 32) ? 0xffffffffu : ((1u << K) - 1u);
  const unsigned mismatches = actmask & ~mball;

  float p = 1.f;
  if (mode == 0 && mismatches != 0u) {
    if (act) {
      const float* sr = stats + ((size_t)b * R + lane) * 5;       // row i-1
      const float* sn = sr + 5;                                    // row i
      const float invK = 1.f / (float)K;
      float* f = feat[warp][lane];
      f[0] = sr[4] - sr[2];
      f[1] = sr[0] - sr[2];
      f[2] = sr[0] - sr[1];
      f[3] = sr[3];
      f[4] = sn[0] - sn[2];
      f[5] = (lane + 1 < K) ? (sn[4] - sn[2]) : 0.f;
      f[6] = (float)(lane + 1) * invK;
      f[7] = (float)__popc(mball & ((1u << lane) - 1u)) * invK;
    }
    __syncwarp();
    const float* sw1 = sm;
    const float* sb1 = sm + H * NF;
    const float* sw2 = sm + H * NF + H;
    float z_mine = 0.f;
    for (int i = 0; i < K; ++i) {
      if (!((mismatches >> i) & 1u)) continue;                    // warp-uniform
      float fi[NF];
#pragma unroll
      for (int k = 0; k < NF; ++k) fi[k] = feat[warp][i][k];
      float zp = 0.f;
      for (int h = lane; h < H; h += 32) {
        float a = sb1[h];
#pragma unroll
        for (int k = 0; k < NF; ++k) a = fmaf(sw1[h * NF + k], fi[k], a);
        zp = fmaf(sw2[h], fmaxf(a, 0.f), zp);
      }
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) zp += __shfl_xor_sync(0xffffffffu, zp, off);
      if (lane == i) z_mine = zp + b2;
    }
    p = 1.f / (1.f + __expf(-z_mine));
  } else if (mode == 1) {
    p = 0.f;
  } else if (mode == 2) {
    p = 1.f;
  }
  if (act) {
    const bool a = match || (p > lambda);
    p_out[(size_t)b * K + lane] = match ? 1.f : p;
    accept[(size_t)b * K + lane] = a ? 1 : 0;
  }
}

}  // namespace

cudaError_t launch_arbitrate(int B, int K, const int32_t* draft, const int32_t* argmax,
                             const float* stats, int H, const float* w1, const float* b1,
                             const float* w2, float b2, float lambda, int mode, float* p_out,
                             uint8_t* accept, cudaStream_t stream) {
  if (B == 0 || K == 0) return cudaSuccess;
  const size_t smem = (mode == 0) ? (size_t)H * (NF + 2) * sizeof(float) : 0;
  if (smem > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(arbitrate_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
  }
  const int grid = (B + WARPS - 1) / WARPS;
  return launch_pdl(arbitrate_kernel, dim3(grid), dim3(WARPS * 32), smem, stream, B, K, draft,
                    argmax, stats, H, w1, b1, w2, b2, lambda, mode, p_out, accept);
}

}  // namespace cospec
