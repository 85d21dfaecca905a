// Accepted length, emitted tokens (Sec. 3.3 Eq. 15; App. F, Inference
// Procedure) and the commit of the accepted rows' K/V into the paged cache.
//
// scan:   one warp per sequence.  A rejected mismatch is Delta_i = 0 and
//         a_i = 0; s = position of the first one (ballot + ffs), else K+1.
//         Emits y_hat_1..y_hat_{s-1}, y_tilde_s and advances ctx_len by s.
// commit: runs first; one CTA per (layer, sequence) finds s the same way and
//         copies block rows 0..s-1 of the staging K and V into cache
//         positions C..C+s-1 (C = ctx_len before the round) with 16-byte
//         vector loads/stores.  The scan, launched after it on the same
//         stream, is the only writer of ctx_len.
#include "cospec_device.cuh"
#include "cospec_internal.h"

namespace cospec {

namespace {

__global__ void __launch_bounds__(128)
    accept_scan_kernel(int B, int K, const int32_t* __restrict__ draft,
                       const int32_t* __restrict__ argmax, const uint8_t* __restrict__ accept,
                       int32_t* __restrict__ ctx_len, int32_t* __restrict__ accept_len,
                       int32_t* __restrict__ emitted, int capacity, int* err) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int b = blockIdx.x * 4 + warp;
  griddep_wait();
  griddep_launch_dependents();
  if (b >= B) return;
  const int R = K + 1;
  const bool act = lane < K;
  const int dft = act ? draft[(size_t)b * K + lane] : 0;
  const int tgt = act ? argmax[(size_t)b * R + lane] : 0;
  const bool rejected = act && (dft != tgt) && (accept[(size_t)b * K + lane] == 0);
  const unsigned rej = __ballot_sync(0xffffffffu, rejected);
  const int s = rej ? __ffs(rej) : R;      // 1-based position of the first rejection
  if (lane < R) {
    int tok = -1;
    if (lane < s - 1) tok = dft;
    else if (lane == s - 1) tok = argmax[(size_t)b * R + lane];
    emitted[(size_t)b * R + lane] = tok;
  }
  if (lane == 0) {
    const int C = ctx_len[b];
    accept_len[b] = s;
    if (C < 0 || C + s > capacity) {
      set_err(err, ERR_CTX);
    } else {
      ctx_len[b] = C + s;
    }
  }
}

__global__ void __launch_bounds__(128)
    commit_kernel(const CommitArgs a, int capacity, int* err) {
  __shared__ int s_len;
  const int l = blockIdx.x, b = blockIdx.y;
  const int R = a.K + 1;
  griddep_wait();
  griddep_launch_dependents();
  if (threadIdx.x < 32) {
    const int lane = threadIdx.x;
    const bool act = lane < a.K;
    const bool rejected = act && (a.draft[(size_t)b * a.K + lane] != a.argmax[(size_t)b * R + lane]) &&
                          (a.accept[(size_t)b * a.K + lane] == 0);
    const unsigned rej = __ballot_sync(0xffffffffu, rejected);
    if (lane == 0) s_len = rej ? __ffs(rej) : R;
  }
  __syncthreads();
  const int s = s_len;
  const int C = a.ctx_len[b];
  if (C < 0 || C + s > capacity) return;   // flagged by the scan
  const int chunks = a.D / 8;              // 16-byte chunks per (row, head)
  const int per_row = a.Hkv * chunks;
  const int total = s * per_row;
  const int* ptab = a.page_table + (size_t)b * a.max_pages;
  for (int e = threadIdx.x; e < total; e += blockDim.x) {
    const int t = e / per_row;
    const int rem = e % per_row;
    const int h = rem / chunks, c = rem % chunks;
    const int pos = C + t;
    const int page = ptab[pos / a.P];
    if ((unsigned)page >= (unsigned)a.num_pages) {
      if (c == 0) set_err(err, ERR_PAGE);
      continue;
    }
    const size_t src = ((((size_t)l * a.B + b) * R + t) * a.Hkv + h) * a.D + (size_t)c * 8;
    const size_t dst = (size_t)l * a.pool_layer_stride +
                       (((size_t)page * a.Hkv + h) * a.P + (pos % a.P)) * a.D + (size_t)c * 8;
    *reinterpret_cast<uint4*>(a.k_pages + dst) = __ldg(reinterpret_cast<const uint4*>(a.k_blk + src));
    *reinterpret_cast<uint4*>(a.v_pages + dst) = __ldg(reinterpret_cast<const uint4*>(a.v_blk + src));
  }
}

}  // namespace

cudaError_t launch_accept_commit(const CommitArgs& a, int* err, cudaStream_t stream) {
  if (a.B == 0) return cudaSuccess;
  const int capacity = a.max_pages * a.P;
  if (a.L > 0) {
    cudaError_t e = launch_pdl(commit_kernel, dim3(a.L, a.B), dim3(128), 0, stream, a, capacity, err);
    if (e != cudaSuccess) return e;
  }
  return launch_pdl(accept_scan_kernel, dim3((a.B + 3) / 4), dim3(128), 0, stream, a.B, a.K,
                    a.draft, a.argmax, a.accept, a.ctx_len, a.accept_len, a.emitted, capacity, err);
}

}  // namespace cospec
