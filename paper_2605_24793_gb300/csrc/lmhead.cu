// LM head fused with argmax and log-prob statistics (Sec. 3.1 Eq. 2: the
// target prediction y_tilde is the argmax of each block row's logits;
// Eq. 23: l_i = x[y_hat_i] - lse).  The M x V logits never reach memory.
//
// tcgen05 swap-AB GEMM: the vocabulary is the MMA M dimension (128 rows of W
// per tile) and the verify rows are N (padded to a multiple of 16, <= 256 per
// pass), so a handful of rows still fills the tensor core and W -- the only
// large operand -- is streamed from HBM exactly once.  Persistent CTAs (one
// per SM) walk vocabulary tiles; warp 0 issues the TMA loads of W (128B
// swizzle, evict-first) and warp 10 those of the hidden rows (evict-last) into
// a ring of stages (one warp's bulk copies are processed one after another,
// so two warps keep the ring full when the hidden rows are a large share of
// each stage), warp 1 issues tcgen05.mma into one of two TMEM accumulators, warps 2-9 read
// the finished accumulator with tcgen05.ld and fold it into per-row running
// statistics while the next tile is multiplied.  A warp may only read the
// TMEM lane quarter (warp id mod 4), so two epilogue warps share each quarter
// (128 vocabulary rows / 4) and take alternate 16-column chunks; two warps per
// SM sub-partition hide each other's shuffle and MUFU latency.  A second small kernel
// merges the per-CTA partials.
//
// Statistics are kept as a tuple (m, i, sec, s, t): max logit, its lowest
// id, second largest logit, s = sum e^(x-m), t = sum e^(x-m) (x-m); then
// lse = m + log s and entropy = log s - t/s.
//
// Stochastic decoding (Sec. 3.1, App. C.3: candidates drawn at temperature
// T = 1) uses the same kernel with KEYED = true: the target candidate is a
// sample of softmax(x / T) taken by the Gumbel-max rule, argmax_v of
// k_v = x_v / T + g_v with g_v = -log(-log u_v).  u comes from Philox4x32-10
// (Salmon et al., SC 2011) keyed by a 64-bit seed read from device memory, at
// counter (v, m / 4, 0, 0), output m % 4, so a thread that owns vocab id v and
// four consecutive rows makes one generator call.  The tuple then carries the
// best key k and i becomes its id; m, sec, s, t stay statistics of the logits.
//
// Speculative sampling (the distribution-preserving baseline at temperature
// T, Sec. 3.1) needs the target's whole distribution at the row where a draft
// token is rejected, so a third mode (MODE_LOGITS) scales the logits by 1 / T,
// writes them out ([M, V] fp32) and keeps the statistics of the scaled logits.
#include <cuda.h>
#include <math.h>

#include <atomic>

#include "../../include/cospec.h"
#include "cospec_device.cuh"
#include "cospec_internal.h"

namespace cospec {

namespace {

constexpr int BM = 128;                 // vocab rows per tile (MMA M)
constexpr int BK = 64;                  // K elements per stage (one 128-byte swizzle row)
constexpr int A_BYTES = BM * BK * 2;    // 16 KB
constexpr int EPI_WARPS = 8;            // two per TMEM lane quarter
constexpr int EPI_THREADS = 32 * EPI_WARPS;
constexpr int H_WARP = 2 + EPI_WARPS;   // producer of the hidden-row boxes
constexpr int NUM_THREADS = 64 + EPI_THREADS + 32;   // W producer, MMA, epilogue, hidden producer
constexpr int MAX_ROWS = 256;           // rows per pass
constexpr uint64_t WAIT_NS = 2000000000ull;

struct Stat {
  float m;
  int i;
  float sec;
  float s;
  float t;
  float k;    // KEYED only: largest perturbed key, whose id is i
};

CS_DEV Stat stat_identity() { return Stat{-INFINITY, 0x7fffffff, -INFINITY, 0.f, 0.f, -INFINITY}; }

template <bool KEYED>
CS_DEV Stat stat_merge(const Stat& a, const Stat& b) {
  Stat r;
  bool a_hi;
  if (KEYED) {
    const bool a_key = (a.k > b.k) || (a.k == b.k && a.i < b.i);
    r.k = a_key ? a.k : b.k;
    r.i = a_key ? a.i : b.i;
    a_hi = a.m >= b.m;
  } else {
    a_hi = (a.m > b.m) || (a.m == b.m && a.i < b.i);
    r.i = a_hi ? a.i : b.i;
    r.k = 0.f;
  }
  const Stat& hi = a_hi ? a : b;
  const Stat& lo = a_hi ? b : a;
  r.m = hi.m;
  r.sec = fmaxf(fmaxf(hi.sec, lo.sec), lo.m);
  if (lo.s > 0.f) {
    const float dm = lo.m - hi.m;
    const float e = __expf(dm);
    r.s = hi.s + lo.s * e;
    r.t = hi.t + e * (lo.t + lo.s * dm);
  } else {
    r.s = hi.s;
    r.t = hi.t;
  }
  return r;
}

template <bool KEYED>
CS_DEV Stat stat_shfl_xor(const Stat& a, int off) {
  Stat r;
  r.m = __shfl_xor_sync(0xffffffffu, a.m, off);
  r.i = __shfl_xor_sync(0xffffffffu, a.i, off);
  r.sec = __shfl_xor_sync(0xffffffffu, a.sec, off);
  r.s = __shfl_xor_sync(0xffffffffu, a.s, off);
  r.t = __shfl_xor_sync(0xffffffffu, a.t, off);
  r.k = KEYED ? __shfl_xor_sync(0xffffffffu, a.k, off) : 0.f;
  return r;
}

CS_DEV Stat stat_of(float x, float k, int v) {
  return Stat{x, v, -INFINITY, (x == -INFINITY) ? 0.f : 1.f, 0.f, k};
}

// Reduce 16 columns held by every lane of a warp (lane l holds vocab id
// base + l) so that lanes 2c and 2c+1 end with column c reduced over all 32
// lanes.  Each butterfly level exchanges half of the remaining columns, so a
// column costs about one merge per lane instead of five.
template <bool KEYED>
CS_DEV Stat warp_reduce16(const float (&x)[16], const float (&key)[16], int lane, int vid) {
  Stat a[8];
  {
    const bool up = (lane & 16) != 0;
    const int pv = vid ^ 16;
#pragma unroll
    for (int c = 0; c < 8; ++c) {
      const float send = up ? x[c] : x[c + 8];
      const float keep = up ? x[c + 8] : x[c];
      const float recv = __shfl_xor_sync(0xffffffffu, send, 16);
      float keep_k = 0.f, recv_k = 0.f;
      if (KEYED) {
        const float send_k = up ? key[c] : key[c + 8];
        keep_k = up ? key[c + 8] : key[c];
        recv_k = __shfl_xor_sync(0xffffffffu, send_k, 16);
      }
      a[c] = stat_merge<KEYED>(stat_of(keep, keep_k, vid), stat_of(recv, recv_k, pv));
    }
  }
  Stat b4[4];
  {
    const bool up = (lane & 8) != 0;
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const Stat send = up ? a[c] : a[c + 4];
      const Stat keep = up ? a[c + 4] : a[c];
      b4[c] = stat_merge<KEYED>(keep, stat_shfl_xor<KEYED>(send, 8));
    }
  }
  Stat c2[2];
  {
    const bool up = (lane & 4) != 0;
#pragma unroll
    for (int c = 0; c < 2; ++c) {
      const Stat send = up ? b4[c] : b4[c + 2];
      const Stat keep = up ? b4[c + 2] : b4[c];
      c2[c] = stat_merge<KEYED>(keep, stat_shfl_xor<KEYED>(send, 4));
    }
  }
  Stat d1;
  {
    const bool up = (lane & 2) != 0;
    const Stat send = up ? c2[0] : c2[1];
    const Stat keep = up ? c2[1] : c2[0];
    d1 = stat_merge<KEYED>(keep, stat_shfl_xor<KEYED>(send, 2));
  }
  return stat_merge<KEYED>(d1, stat_shfl_xor<KEYED>(d1, 1));
}

struct LmParams {
  const int32_t* draft_for_row;  // [M]
  float* stats;                  // [M][5]
  float4* part;                  // [gridDim.x][n_rows]: (m, sec, s, t)
  int* part_idx;                 // [gridDim.x][n_rows]
  float* part_k;                 // [gridDim.x][n_rows], KEYED only
  const unsigned long long* seed;  // KEYED only: Philox key (low word, high word)
  float inv_temp;                // KEYED and LOGITS: 1 / T
  float* logits;                 // LOGITS only: [M][V] x / T
  int row0, n_rows, n_mma;
  int d, V, num_tiles, stages;
  uint32_t tmem_cols;
  int* err;
};

struct SmemLayout {
  uint32_t a_off, b_off, bar_off, epi_off, key_off, total;
};

// The KEYED tuples (per-warp keys [4][n_mma], running keys [n_mma]) go after
// everything else, so the greedy layout is the same with or without them.
__host__ __device__ inline SmemLayout lm_layout(int stages, int n_mma, bool keyed) {
  SmemLayout L;
  L.a_off = 0;
  L.b_off = (uint32_t)stages * A_BYTES;
  L.bar_off = L.b_off + (uint32_t)stages * n_mma * 128;
  const uint32_t bar_bytes = (uint32_t)(2 * stages + 5) * 8 + 16;
  L.epi_off = (L.bar_off + bar_bytes + 15) / 16 * 16;
  // epilogue: per-warp tuples [4][n_mma] (float4 + int), running [n_mma] (float4 + int), draft ids
  const uint32_t epi = 4u * n_mma * 20u + (uint32_t)n_mma * 20u + (uint32_t)n_mma * 4u +
                       4u * EPI_WARPS;
  L.key_off = L.epi_off + epi;
  L.total = L.key_off + (keyed ? 5u * (uint32_t)n_mma * 4u : 0u);
  return L;
}

enum : int { MODE_GREEDY = 0, MODE_KEYED = 1, MODE_LOGITS = 2 };

template <int MODE>
__global__ void __launch_bounds__(NUM_THREADS, 1)
    lmhead_kernel(const __grid_constant__ CUtensorMap tmap_w,
                  const __grid_constant__ CUtensorMap tmap_h, const LmParams p) {
  constexpr bool KEYED = MODE == MODE_KEYED;
  constexpr bool LOGITS = MODE == MODE_LOGITS;
  extern __shared__ uint8_t smem_raw[];
  // TMA with 128B swizzle and the UMMA descriptors need 1024-byte alignment.
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const SmemLayout L = lm_layout(p.stages, p.n_mma, KEYED);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + L.bar_off);
  uint64_t* empty = full + p.stages;
  uint64_t* tfull = empty + p.stages;    // [2]
  uint64_t* tempty = tfull + 2;          // [2]
  uint64_t* mma_done = tempty + 2;       // [1]
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(mma_done + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);
  float4* s_wt = reinterpret_cast<float4*>(smem + L.epi_off);      // [4][n_mma]
  int* s_wti = reinterpret_cast<int*>(s_wt + 4 * p.n_mma);         // [4][n_mma]
  float4* s_run = reinterpret_cast<float4*>(s_wti + 4 * p.n_mma);  // [n_mma]
  int* s_runi = reinterpret_cast<int*>(s_run + p.n_mma);           // [n_mma]
  int* s_draft = s_runi + p.n_mma;                                 // [n_mma]
  volatile int* s_fail = reinterpret_cast<volatile int*>(s_draft + p.n_mma);  // [EPI_WARPS]
  float* s_wk = reinterpret_cast<float*>(smem + L.key_off);         // [4][n_mma], KEYED
  float* s_runk = s_wk + 4 * p.n_mma;                               // [n_mma], KEYED

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int kblocks = p.d / BK;
  const uint32_t b_bytes = (uint32_t)p.n_mma * 128u;

  if (tid == 0) {
    for (int s = 0; s < p.stages; ++s) {
      mbar_init(&full[s], 2);               // the W and the hidden-row producer
      mbar_init(&empty[s], 1);
    }
    mbar_init(&tfull[0], 1);
    mbar_init(&tfull[1], 1);
    mbar_init(&tempty[0], EPI_THREADS);
    mbar_init(&tempty[1], EPI_THREADS);
    mbar_init(mma_done, 1);
    *abort_flag = 0;
    fence_barrier_init();
    tma_prefetch_desc(&tmap_w);
    tma_prefetch_desc(&tmap_h);
  }
  if (warp == 1) {
    tmem_alloc(tmem_holder, p.tmem_cols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_holder;
  // The hidden rows may come from the previous kernel; the W producer
  // (warp 0) reads nothing that does and starts streaming at once.
  if (warp != 0) griddep_wait();
  uint32_t seed_lo = 0, seed_hi = 0;
  if (warp >= 2 && warp < H_WARP) {      // epilogue warps
    if (KEYED) {
      const unsigned long long sd = *p.seed;
      seed_lo = (uint32_t)sd;
      seed_hi = (uint32_t)(sd >> 32);
    }
    for (int c = tid - 64; c < p.n_mma; c += EPI_THREADS) {
      s_run[c] = make_float4(-INFINITY, -INFINITY, 0.f, 0.f);
      s_runi[c] = 0x7fffffff;
      if (KEYED) s_runk[c] = -INFINITY;
      s_draft[c] = (c < p.n_rows) ? p.draft_for_row[p.row0 + c] : -2;
    }
    named_bar_sync(1, EPI_THREADS);
  }
  const uint32_t idesc = idesc_bf16_f32(BM, p.n_mma);

  if (warp == 0) {
    // ------------------------------------------------------------ W producer
    if (lane == 0) {
      const uint64_t pol_w = l2_policy_evict_first();
      int stage = 0;
      uint32_t phase = 0;
      uint32_t issued_mask = 0, issued_parity = 0;   // last load per stage (stages <= 16)
      bool ok = true;
      // A warp's bulk copies are processed one after another, so the W boxes
      // (this warp) and the hidden-row boxes (warp H_WARP) come from two
      // warps, each arriving on the stage barrier with its own bytes.  The
      // first ring's worth of W stages streams before the wait for the
      // previous kernel (W does not depend on it).
      const int my_tiles = blockIdx.x < p.num_tiles ? (p.num_tiles - 1 - blockIdx.x) / gridDim.x + 1 : 0;
      const int npre = min(p.stages, my_tiles * kblocks);
      for (int i = 0; i < npre; ++i) {
        const int tile = blockIdx.x + (i / kblocks) * gridDim.x, kb = i % kblocks;
        mbar_arrive_expect_tx(&full[i], (uint32_t)A_BYTES);
        tma_load_2d(smem_u32(smem + L.a_off + (uint32_t)i * A_BYTES), &tmap_w, &full[i], kb * BK,
                    tile * BM, pol_w);
      }
      int li = 0;                        // loads so far, in (tile, k-block) order
      for (int tile = blockIdx.x; tile < p.num_tiles && ok; tile += gridDim.x) {
        for (int kb = 0; kb < kblocks; ++kb, ++li) {
          if (li >= npre) {
            if (!mbar_wait(&empty[stage], phase ^ 1u, WAIT_NS) || *abort_flag) {
              ok = false;
              break;
            }
            const uint32_t sa = smem_u32(smem + L.a_off + (uint32_t)stage * A_BYTES);
            mbar_arrive_expect_tx(&full[stage], (uint32_t)A_BYTES);
            tma_load_2d(sa, &tmap_w, &full[stage], kb * BK, tile * BM, pol_w);
          }
          issued_mask |= 1u << stage;
          issued_parity = (issued_parity & ~(1u << stage)) | (phase << stage);
          if (++stage == p.stages) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      if (!ok) {
        set_err(p.err, ERR_TIMEOUT);
        *abort_flag = 1;
        // let every issued copy land before shared memory is released
        for (int s = 0; s < p.stages; ++s)
          if (issued_mask & (1u << s)) mbar_wait(&full[s], (issued_parity >> s) & 1u, WAIT_NS);
      }
    }
  } else if (warp == H_WARP) {
    // ------------------------------------------------------------ hidden-row producer
    // (after the wait on the previous kernel: the hidden rows may come from it)
    if (lane == 0) {
      const uint64_t pol_h = l2_policy_evict_last();
      int stage = 0;
      uint32_t phase = 0;
      uint32_t issued_mask = 0, issued_parity = 0;
      bool ok = true;
      int li = 0;
      for (int tile = blockIdx.x; tile < p.num_tiles && ok; tile += gridDim.x) {
        for (int kb = 0; kb < kblocks; ++kb, ++li) {
          if (li >= p.stages && (!mbar_wait(&empty[stage], phase ^ 1u, WAIT_NS) || *abort_flag)) {
            ok = false;
            break;
          }
          const uint32_t sb = smem_u32(smem + L.b_off + (uint32_t)stage * b_bytes);
          mbar_arrive_expect_tx(&full[stage], b_bytes);
          tma_load_2d(sb, &tmap_h, &full[stage], kb * BK, p.row0, pol_h);
          issued_mask |= 1u << stage;
          issued_parity = (issued_parity & ~(1u << stage)) | (phase << stage);
          if (++stage == p.stages) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      if (!ok) {
        set_err(p.err, ERR_TIMEOUT);
        *abort_flag = 1;
        for (int s = 0; s < p.stages; ++s)
          if (issued_mask & (1u << s)) mbar_wait(&full[s], (issued_parity >> s) & 1u, WAIT_NS);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      int it = 0;
      for (int tile = blockIdx.x; tile < p.num_tiles && ok; tile += gridDim.x, ++it) {
        const int acc = it & 1;
        const uint32_t aph = (uint32_t)(it >> 1) & 1u;
        if (!mbar_wait(&tempty[acc], aph ^ 1u, WAIT_NS) || *abort_flag) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(acc * p.n_mma);
        for (int kb = 0; kb < kblocks; ++kb) {
          if (!mbar_wait(&full[stage], phase, WAIT_NS) || *abort_flag) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sa = smem_u32(smem + L.a_off + (uint32_t)stage * A_BYTES);
          const uint32_t sb = smem_u32(smem + L.b_off + (uint32_t)stage * b_bytes);
#pragma unroll
          for (int k = 0; k < BK / 16; ++k) {
            umma_bf16(d_tmem, smem_desc_sw128(sa + k * 32), smem_desc_sw128(sb + k * 32), idesc,
                      (kb | k) != 0 ? 1u : 0u);
          }
          umma_commit(&empty[stage]);
          if (++stage == p.stages) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        umma_commit(&tfull[acc]);
      }
      if (!ok) {
        set_err(p.err, ERR_TIMEOUT);
        *abort_flag = 1;
      }
      // every MMA issued by this thread completes before TMEM is released
      umma_commit(mma_done);
      mbar_wait(mma_done, 0, WAIT_NS);
    }
  } else {
    // ------------------------------------------------------------ epilogue
    const int q = warp & 3;               // TMEM lane quarter this warp may access
    const int ew = warp - 2;              // epilogue warp index
    const int half = ew >> 2;             // which alternate 16-column chunks it takes
    const int etid = tid - 64;
    const int nchunks = (p.n_rows + 15) / 16;
    int it = 0;
    for (int tile = blockIdx.x; tile < p.num_tiles; tile += gridDim.x, ++it) {
      const int acc = it & 1;
      const uint32_t aph = (uint32_t)(it >> 1) & 1u;
      // The epilogue warps take the abort decision together (named
      // barrier + shared flags) so none of them is left waiting at a barrier.
      const bool ok = __all_sync(0xffffffffu, mbar_wait(&tfull[acc], aph, WAIT_NS));
      if (lane == 0) s_fail[ew] = ok ? 0 : 1;
      named_bar_sync(1, EPI_THREADS);
      int any_fail = 0;
#pragma unroll
      for (int w = 0; w < EPI_WARPS; ++w) any_fail |= s_fail[w];
      if (any_fail) {
        if (etid == 0) {
          set_err(p.err, ERR_TIMEOUT);
          *abort_flag = 1;
        }
        break;
      }
      tc_fence_after();
      const int vid = tile * BM + q * 32 + lane;
      const bool valid = vid < p.V;
      const uint32_t tbase = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * p.n_mma);
      for (int ch = half; ch < nchunks; ch += EPI_WARPS / 4) {
        float x[16];
        tmem_ld16(tbase + (uint32_t)(ch * 16), x);
        if (LOGITS) {
          // x / T, written row by row: the warp's 32 lanes hold 32 consecutive
          // vocabulary ids of one row, so each store is one 128-byte line
#pragma unroll
          for (int c = 0; c < 16; ++c) {
            x[c] *= p.inv_temp;
            const int col = ch * 16 + c;
            if (valid && col < p.n_rows) p.logits[(size_t)(p.row0 + col) * p.V + vid] = x[c];
          }
        }
#pragma unroll
        for (int c = 0; c < 16; ++c) {
          const int col = ch * 16 + c;   // < n_mma; s_draft holds -2 past n_rows
          if (valid && s_draft[col] == vid) p.stats[(size_t)(p.row0 + col) * 5 + 4] = x[c];
          if (!valid) x[c] = -INFINITY;
        }
        float key[16];
        if (KEYED) {
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const int c0 = ch * 16 + 4 * j;
            if (c0 < p.n_rows) {             // warp-uniform
              const uint4 u = philox4x32_10(
                  make_uint4((uint32_t)vid, (uint32_t)((p.row0 + c0) >> 2), 0u, 0u), seed_lo, seed_hi);
              key[4 * j + 0] = fmaf(x[4 * j + 0], p.inv_temp, gumbel_of(u.x));
              key[4 * j + 1] = fmaf(x[4 * j + 1], p.inv_temp, gumbel_of(u.y));
              key[4 * j + 2] = fmaf(x[4 * j + 2], p.inv_temp, gumbel_of(u.z));
              key[4 * j + 3] = fmaf(x[4 * j + 3], p.inv_temp, gumbel_of(u.w));
            } else {
#pragma unroll
              for (int c = 0; c < 4; ++c) key[4 * j + c] = -INFINITY;
            }
          }
        }
        const Stat r = warp_reduce16<KEYED>(x, key, lane, vid);
        const int col = ch * 16 + (lane >> 1);
        if ((lane & 1) == 0 && col < p.n_rows) {
          s_wt[q * p.n_mma + col] = make_float4(r.m, r.sec, r.s, r.t);
          s_wti[q * p.n_mma + col] = r.i;
          if (KEYED) s_wk[q * p.n_mma + col] = r.k;
        }
      }
      tc_fence_before();
      mbar_arrive(&tempty[acc]);
      named_bar_sync(1, EPI_THREADS);
      for (int col = etid; col < p.n_rows; col += EPI_THREADS) {
        const float4 rv = s_run[col];
        Stat acc_s{rv.x, s_runi[col], rv.y, rv.z, rv.w, KEYED ? s_runk[col] : 0.f};
#pragma unroll
        for (int w = 0; w < 4; ++w) {
          const float4 v = s_wt[w * p.n_mma + col];
          acc_s = stat_merge<KEYED>(acc_s, Stat{v.x, s_wti[w * p.n_mma + col], v.y, v.z, v.w,
                                                KEYED ? s_wk[w * p.n_mma + col] : 0.f});
        }
        s_run[col] = make_float4(acc_s.m, acc_s.sec, acc_s.s, acc_s.t);
        s_runi[col] = acc_s.i;
        if (KEYED) s_runk[col] = acc_s.k;
      }
      named_bar_sync(1, EPI_THREADS);
    }
    griddep_launch_dependents();
    for (int col = etid; col < p.n_rows; col += EPI_THREADS) {
      p.part[(size_t)blockIdx.x * p.n_rows + col] = s_run[col];
      p.part_idx[(size_t)blockIdx.x * p.n_rows + col] = s_runi[col];
      if (KEYED) p.part_k[(size_t)blockIdx.x * p.n_rows + col] = s_runk[col];
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) {
    __syncwarp();
    tmem_dealloc(tmem_base, p.tmem_cols);
  }
}

// Merge the per-CTA partial statistics of every row (one warp per row).
// argmax receives the sampled id when KEYED.
template <bool KEYED>
__global__ void __launch_bounds__(128) lmhead_reduce_kernel(const float4* part, const int* part_idx,
                                                            const float* part_k, int nparts,
                                                            int row0, int n_rows, int V,
                                                            const int32_t* draft_for_row,
                                                            int32_t* argmax, float* stats, int* err) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int row = blockIdx.x * 4 + warp;
  griddep_wait();
  griddep_launch_dependents();
  if (row >= n_rows) return;
  Stat a = stat_identity();
  for (int c = lane; c < nparts; c += 32) {
    const float4 v = part[(size_t)c * n_rows + row];
    a = stat_merge<KEYED>(a, Stat{v.x, part_idx[(size_t)c * n_rows + row], v.y, v.z, v.w,
                                  KEYED ? part_k[(size_t)c * n_rows + row] : 0.f});
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) a = stat_merge<KEYED>(a, stat_shfl_xor<KEYED>(a, off));
  if (lane == 0) {
    const int m = row0 + row;
    float* st = stats + (size_t)m * 5;
    const float ls = logf(a.s);
    argmax[m] = a.i;
    st[0] = a.m;
    st[1] = a.sec;
    st[2] = a.m + ls;
    st[3] = ls - a.t / a.s;
    const int dft = draft_for_row[m];
    if (dft == -1) {
      st[4] = __int_as_float(0x7fc00000);
    } else if (dft < -1 || dft >= V) {
      st[4] = __int_as_float(0x7fc00000);
      set_err(err, ERR_TOKEN);
    }
  }
}

// 2-D bf16 row-major [rows, cols] map with a {64, box_rows} box and 128B swizzle.
bool make_map(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows) {
  const uint64_t dims[2] = {cols, rows};
  const uint64_t strides[1] = {cols * 2};
  const uint32_t box[2] = {(uint32_t)BK, box_rows};
  return encode_tensor_map_bf16(map, base, 2, dims, strides, box);
}

}  // namespace

// Limits already set on each variant of the kernel.
template <int MODE>
KernelLimits& lm_limits() {
  static KernelLimits lim;
  return lim;
}

LmheadPlan plan_lmhead(int M, int d, int V, int num_sms) {
  LmheadPlan pl{};
  // Rows beyond 256 take several passes over W, of equal size: a pass of
  // 256 rows is tensor-bound while a short one is bound by streaming W, so
  // 384 rows run as 2 x 192 rather than 256 + 128.  Pass p covers rows
  // [p * n_mma, min(M, (p + 1) * n_mma)).
  pl.passes = (M + MAX_ROWS - 1) / MAX_ROWS;
  const int rows = (M + pl.passes - 1) / pl.passes;
  pl.n_mma = (rows + 15) / 16 * 16;
  if (pl.n_mma < 16) pl.n_mma = 16;
  pl.num_tiles = (V + BM - 1) / BM;
  pl.grid = pl.num_tiles < num_sms ? pl.num_tiles : num_sms;
  // One plan serves both variants: shared memory is sized for the keyed
  // layout, which only adds to the end of the greedy one.
  const uint32_t budget = 227u * 1024u - 1024u;
  const uint32_t fixed = lm_layout(0, pl.n_mma, true).total;
  const uint32_t per_stage = A_BYTES + (uint32_t)pl.n_mma * 128u;
  int st = (int)((budget - fixed) / per_stage);
  if (st > 12) st = 12;
  while (st > 2 && lm_layout(st, pl.n_mma, true).total > budget) --st;
  pl.stages = st;
  pl.smem_bytes = lm_layout(st, pl.n_mma, true).total + 1024;
  const size_t per_part = (size_t)1024 * MAX_ROWS;  // upper bound on CTAs x rows
  pl.ws_bytes = per_part * (sizeof(float4) + sizeof(int) + sizeof(float));
  return pl;
}

cudaError_t launch_lmhead(int M, int d, int V, const __nv_bfloat16* hidden,
                          const __nv_bfloat16* w, const int32_t* draft_for_row, int32_t* argmax,
                          float* stats, void* ws, const LmheadPlan& pl, int* err,
                          cudaStream_t stream, const unsigned long long* seed, float inv_temp,
                          float* logits) {
  const bool keyed = seed != nullptr;
  const int mode = keyed ? MODE_KEYED : logits ? MODE_LOGITS : MODE_GREEDY;
  CUtensorMap map_w, map_h;
  if (!make_map(&map_w, w, (uint64_t)V, (uint64_t)d, BM)) return cudaErrorInvalidValue;
  if (!make_map(&map_h, hidden, (uint64_t)M, (uint64_t)d, (uint32_t)pl.n_mma))
    return cudaErrorInvalidValue;
  {
    const cudaError_t e =
        mode == MODE_KEYED
            ? ensure_kernel_limits((const void*)lmhead_kernel<MODE_KEYED>, lm_limits<MODE_KEYED>(),
                                   227 * 1024, false)
        : mode == MODE_LOGITS
            ? ensure_kernel_limits((const void*)lmhead_kernel<MODE_LOGITS>,
                                   lm_limits<MODE_LOGITS>(), 227 * 1024, false)
            : ensure_kernel_limits((const void*)lmhead_kernel<MODE_GREEDY>,
                                   lm_limits<MODE_GREEDY>(), 227 * 1024, false);
    if (e != cudaSuccess) return e;
  }
  float4* part = static_cast<float4*>(ws);
  int* part_idx = reinterpret_cast<int*>(part + (size_t)1024 * MAX_ROWS);
  float* part_k = reinterpret_cast<float*>(part_idx + (size_t)1024 * MAX_ROWS);
  uint32_t tmem_cols = 32;
  while (tmem_cols < (uint32_t)(2 * pl.n_mma)) tmem_cols <<= 1;
  for (int pass = 0; pass < pl.passes; ++pass) {
    LmParams p{};
    p.draft_for_row = draft_for_row;
    p.stats = stats;
    p.part = part;
    p.part_idx = part_idx;
    p.part_k = part_k;
    p.seed = seed;
    p.inv_temp = inv_temp;
    p.logits = logits;
    p.row0 = pass * pl.n_mma;
    p.n_rows = (M - p.row0) < pl.n_mma ? (M - p.row0) : pl.n_mma;
    p.n_mma = pl.n_mma;
    p.d = d;
    p.V = V;
    p.num_tiles = pl.num_tiles;
    p.stages = pl.stages;
    p.tmem_cols = tmem_cols;
    p.err = err;
    const dim3 rgrid((p.n_rows + 3) / 4);
    cudaError_t e;
    if (keyed) {
      e = launch_pdl(lmhead_kernel<MODE_KEYED>, dim3(pl.grid), dim3(NUM_THREADS), pl.smem_bytes,
                     stream, map_w, map_h, p);
      if (e != cudaSuccess) return e;
      e = launch_pdl(lmhead_reduce_kernel<true>, rgrid, dim3(128), 0, stream, (const float4*)part,
                     (const int*)part_idx, (const float*)part_k, pl.grid, p.row0, p.n_rows, V,
                     draft_for_row, argmax, stats, err);
    } else {
      e = mode == MODE_LOGITS
              ? launch_pdl(lmhead_kernel<MODE_LOGITS>, dim3(pl.grid), dim3(NUM_THREADS),
                           pl.smem_bytes, stream, map_w, map_h, p)
              : launch_pdl(lmhead_kernel<MODE_GREEDY>, dim3(pl.grid), dim3(NUM_THREADS),
                           pl.smem_bytes, stream, map_w, map_h, p);
      if (e != cudaSuccess) return e;
      e = launch_pdl(lmhead_reduce_kernel<false>, rgrid, dim3(128), 0, stream, (const float4*)part,
                     (const int*)part_idx, (const float*)nullptr, pl.grid, p.row0, p.n_rows, V,
                     draft_for_row, argmax, stats, err);
    }
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

// ---------------------------------------------------------------------------
// Allocation-free variant of the LM-head call.
//
// Some callers cannot give this library device memory: a serving engine that
// reserves almost all of HBM for its KV cache up front and forbids any other
// allocation during decoding, or a plug-in running inside a host framework
// that owns the device's memory and exposes no workspace.  For them the
// per-CTA partial statistics live in one fixed scratch array compiled into
// the library (resident on every GPU that loads it, until the process exits)
// instead of a caller-provided workspace.
//
// The array below is a device symbol: in host code its name is only a
// stand-in, never a device address.  Its address is looked up with
// cudaGetSymbolAddress once per device, on that device's first call.
namespace {

constexpr int NOALLOC_MAX_CTAS = 256;                 // persistent CTAs (one per SM)
constexpr int NOALLOC_MAX_M = 512;                    // rows per call (two 256-row passes)
constexpr size_t NOALLOC_ENTRIES = (size_t)NOALLOC_MAX_CTAS * MAX_ROWS;
// [NOALLOC_ENTRIES] float4 (m, second, s, t) then [NOALLOC_ENTRIES] int (argmax)
static __device__ __align__(256) unsigned char g_lmhead_scratch[NOALLOC_ENTRIES * (sizeof(float4) + sizeof(int))];

std::atomic<void*> g_scratch_addr[64];   // per device; a race only repeats the lookup

// The scratch's device address on the current device, looked up on the
// device's first call; the CUDA error of a failed lookup otherwise.
cudaError_t scratch_address(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  void* addr = g_scratch_addr[dev].load(std::memory_order_acquire);
  if (!addr) {
    e = cudaGetSymbolAddress(&addr, g_lmhead_scratch);
    if (e != cudaSuccess) return e;
    g_scratch_addr[dev].store(addr, std::memory_order_release);
  }
  *out = addr;
  return cudaSuccess;
}

}  // namespace

}  // namespace cospec

extern "C" COSPEC_API int cospec_lmhead_argmax_features_noalloc(
    int M, int d, int V, const uint16_t* hidden, const uint16_t* w, const int32_t* draft_for_row,
    int32_t* argmax, float* stats, void* stream) {
  using namespace cospec;
  if (M < 0 || d <= 0 || V <= 0) return COSPEC_ERR_INVALID_ARG;
  if (M == 0) return COSPEC_OK;
  if (!hidden || !w || !draft_for_row || !argmax || !stats) return COSPEC_ERR_INVALID_ARG;
  if (d % 64 != 0 || (long long)V > 0x7fffff00LL) return COSPEC_ERR_UNSUPPORTED;
  if ((reinterpret_cast<uintptr_t>(hidden) & 15u) || (reinterpret_cast<uintptr_t>(w) & 15u))
    return COSPEC_ERR_INVALID_ARG;
  if (M > NOALLOC_MAX_M) return COSPEC_ERR_UNSUPPORTED;          // beyond the fixed scratch
  const int sms = device_num_sms();
  if (sms <= 0) return cuda_lookup_failed();
  const LmheadPlan pl = plan_lmhead(M, d, V, sms);
  if (pl.grid > NOALLOC_MAX_CTAS) return COSPEC_ERR_UNSUPPORTED;  // beyond the fixed scratch
  void* scratch = nullptr;
  const cudaError_t se = scratch_address(&scratch);
  if (se != cudaSuccess) return cuda_status(se);
  int* err = device_error_word();
  if (!err) return cuda_lookup_failed();
  float4* part = static_cast<float4*>(scratch);
  int* part_idx = reinterpret_cast<int*>(part + NOALLOC_ENTRIES);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  CUtensorMap map_w, map_h;
  if (!make_map(&map_w, w, (uint64_t)V, (uint64_t)d, BM) ||
      !make_map(&map_h, hidden, (uint64_t)M, (uint64_t)d, (uint32_t)pl.n_mma))
    return cuda_status(cudaErrorInvalidValue);      // as the workspace entry point reports it
  const cudaError_t le =
      ensure_kernel_limits((const void*)lmhead_kernel<MODE_GREEDY>, lm_limits<MODE_GREEDY>(),
                           227 * 1024, false);
  if (le != cudaSuccess) return cuda_status(le);
  uint32_t tmem_cols = 32;
  while (tmem_cols < (uint32_t)(2 * pl.n_mma)) tmem_cols <<= 1;
  // Each pass overwrites every scratch entry its merge kernel reads, so the
  // contents left by an earlier call never need clearing.
  for (int pass = 0; pass < pl.passes; ++pass) {
    LmParams p{};
    p.draft_for_row = draft_for_row;
    p.stats = stats;
    p.part = part;
    p.part_idx = part_idx;
    p.row0 = pass * pl.n_mma;
    p.n_rows = (M - p.row0) < pl.n_mma ? (M - p.row0) : pl.n_mma;
    p.n_mma = pl.n_mma;
    p.d = d;
    p.V = V;
    p.num_tiles = pl.num_tiles;
    p.stages = pl.stages;
    p.tmem_cols = tmem_cols;
    p.err = err;
    cudaError_t e = launch_pdl(lmhead_kernel<MODE_GREEDY>, dim3(pl.grid), dim3(NUM_THREADS),
                               pl.smem_bytes, st, map_w, map_h, p);
    if (e == cudaSuccess)
      e = launch_pdl(lmhead_reduce_kernel<false>, dim3((p.n_rows + 3) / 4), dim3(128), 0, st,
                     (const float4*)part, (const int*)part_idx, (const float*)nullptr, pl.grid,
                     p.row0, p.n_rows, V, draft_for_row, argmax, stats, err);
    if (e != cudaSuccess) return cuda_status(e);
  }
  return COSPEC_OK;
}
