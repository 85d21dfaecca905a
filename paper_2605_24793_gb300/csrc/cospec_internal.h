// Internal host-side interface between the C-ABI layer (api.cu) and the
// kernel translation units.  Not part of the public ABI.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <atomic>
#include <functional>
#include <stddef.h>
#include <stdint.h>

namespace cospec {

// Launch with programmatic stream serialization: the kernel may start while
// the previous kernel of the stream finishes; it must call griddep_wait()
// before reading anything an earlier kernel wrote.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t stream, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, args...);
}

int device_num_sms();
int* device_error_word();  // device address of the error word of the current device

// Per-device record of the limits already set on one kernel.
constexpr int KL_MAX_DEV = 64;
struct KernelLimits {
  std::atomic<size_t> smem[KL_MAX_DEV];   // dynamic shared-memory limit set so far
  std::atomic<bool> cluster[KL_MAX_DEV];  // non-portable cluster sizes allowed
};
// Raise `kern`'s dynamic shared-memory limit on the current device to at
// least `smem_bytes` (never lowering it, so graphs captured earlier stay
// launchable) and, with `cluster`, allow non-portable cluster sizes.  Calls
// from several host threads are serialised; later calls that need nothing
// new only read `lim`.
// Records e as the calling thread's last CUDA error (cospec_last_cuda_error)
// and returns COSPEC_ERR_CUDA, or COSPEC_OK for cudaSuccess.
int cuda_status(cudaError_t e);
// The same for a failed lookup that returned no cudaError_t: records the
// runtime's pending error (cudaErrorUnknown if there is none).
int cuda_lookup_failed();

cudaError_t ensure_kernel_limits(const void* kern, KernelLimits& lim, size_t smem_bytes,
                                 bool cluster);

// cuTensorMapEncodeTiled for a bf16 tensor (rank 1..5, innermost first),
// 128-byte swizzle, zero fill out of bounds.  dims/box in elements, strides
// in bytes for dimensions 1..rank-1.
bool encode_tensor_map_bf16(void* map, const void* base, int rank, const uint64_t* dims,
                            const uint64_t* strides, const uint32_t* box);

// ---------------------------------------------------------------- attention
struct AttnArgs {
  const __nv_bfloat16* q;
  const __nv_bfloat16* k_blk;
  const __nv_bfloat16* v_blk;
  const __nv_bfloat16* k_pages;
  const __nv_bfloat16* v_pages;
  const int32_t* page_table;
  const int32_t* ctx_len;
  __nv_bfloat16* out;
  int B, R, Hq, Hkv, D, P, max_pages, num_pages;
  float scale;
  int max_ctx;
  int kv_stable;   // cache-side reads may start before the previous kernel finishes
  int block_full;  // block rows attend to every block row
};
struct AttnPlan {
  int kind;               // 0: mma.sync kernel, 1: tcgen05 kernel (query rows as MMA M)
  int mt, wk, nrp;        // mma.sync: row tiles, key groups, padded rows
  int nt, jb, jbq, rg;    // tcgen05: row capacity (128), block rows per row group,
                          // block rows of the query box, row groups
  int cluster;            // CTAs per (sequence, KV head, row group): the KV split
  long long units;        // (sequence, KV head, row group) units, one cluster each
  int one_wave;           // small batch: take the largest split whose clusters are
                          // all resident at once (latency-bound)
};
// Clusters of `S` CTAs of the plan's kernel variant resident at once on the
// device (0: not schedulable).
using ResidentFn = std::function<long long(const AttnPlan&, int S)>;
AttnPlan plan_verify_attn(int B, int R, int Hq, int Hkv, int D, int max_ctx, int num_sms,
                          bool kv_stable, const ResidentFn& resident);
int attn_max_active_clusters(int D, int mt, int wk, int S, int Hkv, int B, int kbr);
cudaError_t launch_verify_attn(const AttnArgs& a, const AttnPlan& plan, int* err,
                               cudaStream_t stream);
bool tcq_attn_supported(int D, int G);
int attn_tcq_max_active_clusters(int D, int S, int Hkv, int B, int RG);
cudaError_t launch_verify_attn_tcq(const AttnArgs& a, const AttnPlan& plan, int* err,
                                   cudaStream_t stream);

// ---------------------------------------------------------------- LM head
struct LmheadPlan {
  int n_mma;       // MMA N (padded rows per pass), multiple of 16, <= 256
  int passes;      // ceil(M / 256)
  int num_tiles;   // ceil(V / 128)
  int grid;        // persistent CTAs
  int stages;
  size_t smem_bytes;
  size_t ws_bytes;
};
LmheadPlan plan_lmhead(int M, int d, int V, int num_sms);
cudaError_t launch_lmhead(int M, int d, int V, const __nv_bfloat16* hidden,
                          const __nv_bfloat16* w, const int32_t* draft_for_row, int32_t* argmax,
                          float* stats, void* ws, const LmheadPlan& plan, int* err,
                          cudaStream_t stream, const unsigned long long* seed = nullptr,
                          float inv_temp = 1.f, float* logits = nullptr);

// ---------------------------------------------------------------- speculative sampling
constexpr int SPS_MAX_SLICES = 64;   // vocabulary slices (CTAs) per sequence
struct SpsArgs {
  int B, K, V;
  const int32_t* draft;
  const float* stats;
  const float* logits;
  const float* q;
  const unsigned long long* seed;
  int32_t* target;
  uint8_t* accept;
  float* ratio;
  void* ws;
};
int sps_slices(int B, int V, int num_sms);
cudaError_t launch_sps(const SpsArgs& a, int num_sms, int* err, cudaStream_t stream);

// ---------------------------------------------------------------- arbitration
cudaError_t launch_arbitrate(int B, int K, const int32_t* draft, const int32_t* argmax,
                             const float* stats, int H, const float* w1, const float* b1,
                             const float* w2, float b2, float lambda, int mode, float* p_out,
                             uint8_t* accept, cudaStream_t stream);

// ---------------------------------------------------------------- accept + commit
struct CommitArgs {
  int B, K, L, Hkv, D, P, max_pages, num_pages;
  long long pool_layer_stride;
  const int32_t* draft;
  const int32_t* argmax;
  const uint8_t* accept;
  const __nv_bfloat16* k_blk;
  const __nv_bfloat16* v_blk;
  __nv_bfloat16* k_pages;
  __nv_bfloat16* v_pages;
  const int32_t* page_table;
  int32_t* ctx_len;
  int32_t* accept_len;
  int32_t* emitted;
};
cudaError_t launch_accept_commit(const CommitArgs& a, int* err, cudaStream_t stream);

}  // namespace cospec
