// Speculative-sampling acceptance of the exact-match baseline at temperature
// T (Sec. 3.1 "Stochastic decoding", App. C.3: the distribution-preserving
// baselines use standard speculative sampling with acceptance-ratio
// correction; the algorithm is that of Leviathan et al., ICML 2023, and Chen
// et al., 2023).
//
// Inputs are the LM head's scaled logits x / T of every block row with their
// statistics (cospec_lmhead_logits_features), the draft tokens and the
// draft's distributions q.  For draft position i (block row i - 1):
//   p_i(y) = exp(x_{i-1}[y] - lse_{i-1}),  ratio_i = min(1, p_i(y_hat_i) / q_i(y_hat_i)),
//   y_hat_i is accepted iff u_i * q_i(y_hat_i) < p_i(y_hat_i);
// the first rejected position i* draws its token from the residual
// max(0, p_{i*} - q_{i*}) (renormalised), or, with no rejection, the bonus row
// K draws from p_{K+1}.  Both draws are Gumbel-max over the vocabulary:
// argmax_v (log w(v) + g_{m,v}) with w the residual (where positive) or p,
// g the Gumbel noise of block row m = b (K + 1) + row -- the noise the
// temperature sampling of the LM head uses -- and ties to the lowest id.
//
// Randomness is Philox4x32-10 keyed by the 64-bit seed: the acceptance
// uniform of (sequence b, position i) is output word 0 at counter
// (i - 1, b, 1, 0), u = (floor(r / 2^9) + 0.5) / 2^23; the noise of row m at
// id v is output m mod 4 at counter (v, floor(m / 4), 0, 0).
//
// Two kernels: the first (CTAs = vocabulary slices x sequences) takes every
// sequence's accept/reject decisions (each CTA of a sequence takes the same
// ones, from the same bits) and the best residual and plain keys of its
// vocabulary slice; the second (a warp per sequence) merges the slices.  The
// outputs plug into cospec_accept_commit as (argmax, accept): accepted
// positions carry their draft token, the stop row the drawn token.
#include <math.h>

#include "cospec_device.cuh"
#include "cospec_internal.h"

namespace cospec {

namespace {

constexpr int SPS_THREADS = 256;

struct SpsParams {
  int B, K, V, ns;
  const int32_t* draft;       // [B][K]
  const float* stats;         // [B*(K+1)][5], of x / T
  const float* logits;        // [B*(K+1)][V], x / T
  const float* q;             // [B][K][V]
  const unsigned long long* seed;
  int32_t* target;            // [B][K+1]
  uint8_t* accept;            // [B][K]
  float* ratio;               // [B][K]
  float4* part;               // [B][ns]: (residual key, its id, plain key, its id)
  int* row_of;                // [B]: the sampled block row
  int* err;
};

struct KeyId {
  float k;
  int i;
};

CS_DEV KeyId better(KeyId a, KeyId b) {
  return (b.k > a.k || (b.k == a.k && b.i < a.i)) ? b : a;
}

CS_DEV KeyId warp_best(KeyId a) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    KeyId o;
    o.k = __shfl_xor_sync(0xffffffffu, a.k, off);
    o.i = __shfl_xor_sync(0xffffffffu, a.i, off);
    a = better(a, o);
  }
  return a;
}

__global__ void __launch_bounds__(SPS_THREADS) sps_sample_kernel(const SpsParams p) {
  __shared__ int s_row;
  __shared__ KeyId s_best[2][SPS_THREADS / 32];
  const int b = blockIdx.y, x = blockIdx.x;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int R = p.K + 1;
  griddep_wait();                         // stats and logits come from the LM head
  const unsigned long long sd = *p.seed;
  const uint32_t k0 = (uint32_t)sd, k1 = (uint32_t)(sd >> 32);
  if (warp == 0) {
    // lane i decides draft position i + 1 (block row i)
    bool rej = false;
    int y = 0;
    if (lane < p.K) {
      y = p.draft[(size_t)b * p.K + lane];
      const bool bad = y < 0 || y >= p.V;
      if (bad && x == 0) set_err(p.err, ERR_TOKEN);
      const int m = b * R + lane;
      const float* st = p.stats + (size_t)m * 5;
      const float pv = bad ? 0.f : __expf(st[4] - st[2]);
      const float qv = bad ? 1.f : p.q[((size_t)b * p.K + lane) * p.V + y];
      const uint4 r = philox4x32_10(make_uint4((uint32_t)lane, (uint32_t)b, 1u, 0u), k0, k1);
      const float u = ((float)(r.x >> 9) + 0.5f) * 1.1920928955078125e-7f;
      rej = !(u * qv < pv);
      if (x == 0) p.ratio[(size_t)b * p.K + lane] = qv > 0.f ? fminf(1.f, pv / qv) : 1.f;
    }
    const unsigned rmask = __ballot_sync(0xffffffffu, rej);
    const int row = rmask ? __ffs(rmask) - 1 : p.K;     // the first rejected position's row
    if (x == 0) {
      if (lane < p.K) {
        p.accept[(size_t)b * p.K + lane] = lane < row ? 1 : 0;
        p.target[(size_t)b * R + lane] = lane < row ? y : -1;   // the row itself: the merge
      }
      if (lane == 0) {
        if (row < p.K) p.target[(size_t)b * R + p.K] = -1;
        p.row_of[b] = row;
      }
    }
    if (lane == 0) s_row = row;
  }
  __syncthreads();
  const int row = s_row;
  const bool residual = row < p.K;
  const int m = b * R + row;
  const float lse = p.stats[(size_t)m * 5 + 2];
  const float* xr = p.logits + (size_t)m * p.V;
  const float* qr = p.q + ((size_t)b * p.K + (residual ? row : 0)) * p.V;
  const int v0 = (int)(((long long)p.V * x) / p.ns);
  const int v1 = (int)(((long long)p.V * (x + 1)) / p.ns);
  KeyId best_r{-INFINITY, 0x7fffffff}, best_p{-INFINITY, 0x7fffffff};
  for (int v = v0 + tid; v < v1; v += SPS_THREADS) {
    const float xv = xr[v];
    const uint4 r = philox4x32_10(make_uint4((uint32_t)v, (uint32_t)(m >> 2), 0u, 0u), k0, k1);
    const uint32_t word = (m & 3) == 0 ? r.x : (m & 3) == 1 ? r.y : (m & 3) == 2 ? r.z : r.w;
    const float g = gumbel_of(word);
    const float kp = xv + g;                       // log p(v) + g up to the constant lse
    if (kp > best_p.k) best_p = KeyId{kp, v};      // ids rise along a thread: ties keep the first
    if (residual) {
      const float w = __expf(xv - lse) - qr[v];
      if (w > 0.f) {
        const float kr = __logf(w) + g;
        if (kr > best_r.k) best_r = KeyId{kr, v};
      }
    }
  }
  best_r = warp_best(best_r);
  best_p = warp_best(best_p);
  if (lane == 0) {
    s_best[0][warp] = best_r;
    s_best[1][warp] = best_p;
  }
  __syncthreads();
  if (tid == 0) {
    KeyId r = s_best[0][0], q = s_best[1][0];
#pragma unroll
    for (int w = 1; w < SPS_THREADS / 32; ++w) {
      r = better(r, s_best[0][w]);
      q = better(q, s_best[1][w]);
    }
    p.part[(size_t)b * p.ns + x] = make_float4(r.k, __int_as_float(r.i), q.k, __int_as_float(q.i));
  }
  griddep_launch_dependents();
}

// One warp per sequence: merge the vocabulary slices.  The residual draw
// wins when any slice found a positive residual entry; otherwise (the bonus
// row, or a residual emptied by rounding) the plain draw from p.
__global__ void __launch_bounds__(128) sps_merge_kernel(const SpsParams p) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int b = blockIdx.x * 4 + warp;
  griddep_wait();
  griddep_launch_dependents();
  if (b >= p.B) return;
  KeyId r{-INFINITY, 0x7fffffff}, q{-INFINITY, 0x7fffffff};
  for (int x = lane; x < p.ns; x += 32) {
    const float4 v = p.part[(size_t)b * p.ns + x];
    r = better(r, KeyId{v.x, __float_as_int(v.y)});
    q = better(q, KeyId{v.z, __float_as_int(v.w)});
  }
  r = warp_best(r);
  q = warp_best(q);
  if (lane == 0) {
    const int row = p.row_of[b];
    const int tok = (r.i != 0x7fffffff) ? r.i : q.i;
    p.target[(size_t)b * (p.K + 1) + row] = tok;
  }
}

}  // namespace

int sps_slices(int B, int V, int num_sms) {
  int ns = (2 * num_sms + B - 1) / (B > 0 ? B : 1);
  const int by_v = (V + 1023) / 1024;            // at least ~1k ids per slice
  if (ns > by_v) ns = by_v;
  if (ns > SPS_MAX_SLICES) ns = SPS_MAX_SLICES;
  return ns < 1 ? 1 : ns;
}

cudaError_t launch_sps(const SpsArgs& a, int num_sms, int* err, cudaStream_t stream) {
  SpsParams p{};
  p.B = a.B;
  p.K = a.K;
  p.V = a.V;
  p.ns = sps_slices(a.B, a.V, num_sms);
  p.draft = a.draft;
  p.stats = a.stats;
  p.logits = a.logits;
  p.q = a.q;
  p.seed = a.seed;
  p.target = a.target;
  p.accept = a.accept;
  p.ratio = a.ratio;
  uint8_t* ws = static_cast<uint8_t*>(a.ws);
  p.part = reinterpret_cast<float4*>(ws);
  p.row_of = reinterpret_cast<int*>(ws + (size_t)a.B * SPS_MAX_SLICES * sizeof(float4));
  p.err = err;
  cudaError_t e = launch_pdl(sps_sample_kernel, dim3(p.ns, a.B), dim3(SPS_THREADS), 0, stream, p);
  if (e != cudaSuccess) return e;
  return launch_pdl(sps_merge_kernel, dim3((a.B + 3) / 4), dim3(128), 0, stream, p);
}

}  // namespace cospec
