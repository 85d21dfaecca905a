// Verify attention of the K+1 block rows over a paged bf16 KV cache
// (teacher-forced verification pass, Sec. 3.1 Eq. 2 of the paper).
//
// One CTA owns (sequence b, KV head, KV split).  It loads each 64-token K/V
// tile of its split once (cp.async, 16-byte chunks, 3-stage ring, XOR-swizzled
// rows) and multiplies it against ALL query rows that read this KV head: the
// G = Hq/Hkv heads of the group times the R block rows (row index j*G + g).
// Q.K^T and P.V run on bf16 tensor cores (mma.m16n8k16, fp32 accumulate);
// the softmax is online in base 2.  Warps split the rows (16 per warp) and,
// when there are few rows, the keys of a tile; their partial (m, l, O) merge
// in shared memory.  Splits of one (b, head) merge through a workspace: the
// last CTA to finish (atomic ticket, no waiting) combines them.
#include <math.h>

#include "cospec_device.cuh"
#include "cospec_internal.h"

namespace cospec {

namespace {

constexpr int KT = 64;        // keys per tile (4 pages of 16)
constexpr int NSTAGE = 3;     // cp.async ring depth
constexpr int PAGE = 16;      // page size (fixed)

struct AttnParams {
  const __nv_bfloat16* q;
  const __nv_bfloat16* k_blk;
  const __nv_bfloat16* v_blk;
  const __nv_bfloat16* k_pages;
  const __nv_bfloat16* v_pages;
  const int32_t* page_table;
  const int32_t* ctx_len;
  __nv_bfloat16* out;
  float* ws_o;     // [B*Hkv][max_splits][nrp][D] un-normalised partial outputs
  float2* ws_ml;   // [B*Hkv][max_splits][nrp] (running max, running sum), log2 domain
  int* tickets;    // [B*Hkv] arrival counters, left at zero
  int B, R, Hq, Hkv, G, NR, nrp;
  int max_pages, num_pages;
  int tiles_per_split, max_splits;
  float scale_log2;
  int* err;
};

template <int D, int MT, int WK>
__global__ void __launch_bounds__(MT* WK * 32) verify_attn_kernel(const AttnParams p) {
  constexpr int NWARPS = MT * WK;
  constexpr int NT = NWARPS * 32;
  constexpr int KW = KT / WK;          // keys of a tile handled by one warp
  constexpr int CH = D / 8;            // 16-byte chunks per key row
  constexpr int TILE = KT * D;         // elements per K (or V) tile
  constexpr int NRP = MT * 16;         // padded query rows
  static_assert(KW % 16 == 0, "keys per warp must be a multiple of 16");

  extern __shared__ __align__(128) uint8_t smem_raw[];
  __nv_bfloat16* sK = reinterpret_cast<__nv_bfloat16*>(smem_raw);
  __nv_bfloat16* sV = sK + NSTAGE * TILE;
  __shared__ int s_last;

  const int split = blockIdx.x, kvh = blockIdx.y, b = blockIdx.z;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int wr = warp / WK, wk = warp % WK;

  const int C = p.ctx_len[b];
  const int T = C + p.R;
  const int ntiles = (T + KT - 1) / KT;
  const int nsplit = (ntiles + p.tiles_per_split - 1) / p.tiles_per_split;
  if (C < 0 || C > p.max_pages * PAGE || nsplit > p.max_splits) {
    if (split == 0 && kvh == 0 && tid == 0) set_err(p.err, ERR_CTX);
    return;
  }
  if (split >= nsplit) return;
  const int t_begin = split * p.tiles_per_split;
  const int t_end = min(ntiles, t_begin + p.tiles_per_split);
  const int* ptab = p.page_table + (size_t)b * p.max_pages;

  auto load_tile = [&](int t, int st) {
    const uint32_t sk = smem_u32(sK + st * TILE);
    const uint32_t sv = smem_u32(sV + st * TILE);
#pragma unroll 4
    for (int c = tid; c < KT * CH; c += NT) {
      const int key = c / CH, ch = c % CH;
      const int pos = t * KT + key;
      const __nv_bfloat16* gk = p.k_pages;
      const __nv_bfloat16* gv = p.v_pages;
      bool valid = false;
      if (pos < C) {
        const int page = __ldg(ptab + pos / PAGE);
        if ((unsigned)page < (unsigned)p.num_pages) {
          const size_t off =
              (((size_t)page * p.Hkv + kvh) * PAGE + (pos % PAGE)) * D + (size_t)ch * 8;
          gk += off;
          gv += off;
          valid = true;
        } else if (ch == 0) {
          set_err(p.err, ERR_PAGE);
        }
      } else if (pos < T) {
        const size_t off = (((size_t)b * p.R + (pos - C)) * p.Hkv + kvh) * D + (size_t)ch * 8;
        gk = p.k_blk + off;
        gv = p.v_blk + off;
        valid = true;
      }
      const uint32_t so = (uint32_t)(key * D + ((ch ^ (key & 7)) * 8)) * 2u;
      cp_async16(sk + so, gk, valid);
      cp_async16(sv + so, gv, valid);
    }
  };

  // Issue the first tiles before anything else so the loads overlap set-up.
#pragma unroll
  for (int s = 0; s < NSTAGE - 1; ++s) {
    if (t_begin + s < t_end) load_tile(t_begin + s, s);
    cp_async_commit();
  }

  // Query fragments (A operand, 16 rows x D) of this warp's row tile.
  const int g_row = lane >> 2, c4 = lane & 3;
  const int r0 = wr * 16 + g_row, r1 = r0 + 8;
  uint32_t qf[D / 16][4];
  {
    auto row_ptr = [&](int r) -> const __nv_bfloat16* {
      if (r >= p.NR) return nullptr;
      const int j = r / p.G, g = r % p.G;
      return p.q + (((size_t)b * p.R + j) * p.Hq + (size_t)kvh * p.G + g) * D;
    };
    const __nv_bfloat16* q0 = row_ptr(r0);
    const __nv_bfloat16* q1 = row_ptr(r1);
#pragma unroll
    for (int kk = 0; kk < D / 16; ++kk) {
      const int col = kk * 16 + 2 * c4;
      qf[kk][0] = q0 ? __ldg(reinterpret_cast<const uint32_t*>(q0 + col)) : 0u;
      qf[kk][1] = q1 ? __ldg(reinterpret_cast<const uint32_t*>(q1 + col)) : 0u;
      qf[kk][2] = q0 ? __ldg(reinterpret_cast<const uint32_t*>(q0 + col + 8)) : 0u;
      qf[kk][3] = q1 ? __ldg(reinterpret_cast<const uint32_t*>(q1 + col + 8)) : 0u;
    }
  }
  // Block row of this thread's two query rows; a row j sees positions <= C + j.
  const int lim0 = C + min(r0 / p.G, p.R - 1);
  const int lim1 = C + min(r1 / p.G, p.R - 1);

  float o[D / 8][4];
#pragma unroll
  for (int i = 0; i < D / 8; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;

  for (int t = t_begin, it = 0; t < t_end; ++t, ++it) {
    cp_async_wait<NSTAGE - 2>();
    __syncthreads();
    {
      const int tn = t + NSTAGE - 1;
      if (tn < t_end) load_tile(tn, (it + NSTAGE - 1) % NSTAGE);
      cp_async_commit();
    }
    const int st = it % NSTAGE;
    const uint32_t sk = smem_u32(sK + st * TILE);
    const uint32_t sv = smem_u32(sV + st * TILE);

    // S = Q K^T over this warp's KW keys.
    float s[KW / 8][4];
#pragma unroll
    for (int nt = 0; nt < KW / 8; ++nt) {
      s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.f;
      const int key = wk * KW + nt * 8 + (lane & 7);
#pragma unroll
      for (int kk = 0; kk < D / 16; kk += 2) {
        const int ch = kk * 2 + (lane >> 3);
        uint32_t b0, b1, b2, b3;
        ldsm_x4(sk + (uint32_t)(key * D + ((ch ^ (key & 7)) * 8)) * 2u, b0, b1, b2, b3);
        mma_16816(s[nt], qf[kk], b0, b1);
        mma_16816(s[nt], qf[kk + 1], b2, b3);
      }
    }

    // Scale, causal mask on block positions, online softmax (log2 domain).
    const int kbase = t * KT + wk * KW;
    const bool need_mask = (t * KT + KT) > C;
    float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
    for (int nt = 0; nt < KW / 8; ++nt) {
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int pos = kbase + nt * 8 + 2 * c4 + e;
        float v0 = s[nt][e] * p.scale_log2;
        float v1 = s[nt][2 + e] * p.scale_log2;
        if (need_mask) {
          if (pos > lim0) v0 = -INFINITY;
          if (pos > lim1) v1 = -INFINITY;
        }
        s[nt][e] = v0;
        s[nt][2 + e] = v1;
        mx0 = fmaxf(mx0, v0);
        mx1 = fmaxf(mx1, v1);
      }
    }
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
    const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
    const float base0 = (mn0 == -INFINITY) ? 0.f : mn0;
    const float base1 = (mn1 == -INFINITY) ? 0.f : mn1;
    const float a0 = exp2f(m0 - base0), a1 = exp2f(m1 - base1);
    m0 = mn0;
    m1 = mn1;
    l0 *= a0;
    l1 *= a1;
#pragma unroll
    for (int i = 0; i < D / 8; ++i) {
      o[i][0] *= a0;
      o[i][1] *= a0;
      o[i][2] *= a1;
      o[i][3] *= a1;
    }
    uint32_t pf[KW / 16][4];
#pragma unroll
    for (int nt = 0; nt < KW / 8; ++nt) {
      const float p0 = exp2f(s[nt][0] - base0), p1 = exp2f(s[nt][1] - base0);
      const float p2 = exp2f(s[nt][2] - base1), p3 = exp2f(s[nt][3] - base1);
      l0 += p0 + p1;
      l1 += p2 + p3;
      pf[nt / 2][(nt % 2) * 2 + 0] = pack_bf16(p0, p1);
      pf[nt / 2][(nt % 2) * 2 + 1] = pack_bf16(p2, p3);
    }

    // O += P V.
#pragma unroll
    for (int kk2 = 0; kk2 < KW / 16; ++kk2) {
      const int key = wk * KW + kk2 * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
#pragma unroll
      for (int nd = 0; nd < D / 8; nd += 2) {
        const int ch = nd + (lane >> 4);
        uint32_t b0, b1, b2, b3;
        ldsm_x4_t(sv + (uint32_t)(key * D + ((ch ^ (key & 7)) * 8)) * 2u, b0, b1, b2, b3);
        mma_16816(o[nd], pf[kk2], b0, b1);
        mma_16816(o[nd + 1], pf[kk2], b2, b3);
      }
    }
  }
  cp_async_wait<0>();
  __syncthreads();

  // Row sums live spread over the 4 threads of a quad.
  l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
  l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 2);

  // Merge the WK key groups of each row tile in shared memory.
  float* red_o = reinterpret_cast<float*>(smem_raw);           // [NWARPS][16][D]
  float2* red_ml = reinterpret_cast<float2*>(red_o + NWARPS * 16 * D);  // [NWARPS][16]
  {
    float* wo = red_o + warp * 16 * D;
#pragma unroll
    for (int nd = 0; nd < D / 8; ++nd) {
      const int col = nd * 8 + 2 * c4;
      *reinterpret_cast<float2*>(wo + g_row * D + col) = make_float2(o[nd][0], o[nd][1]);
      *reinterpret_cast<float2*>(wo + (g_row + 8) * D + col) = make_float2(o[nd][2], o[nd][3]);
    }
    if (c4 == 0) {
      red_ml[warp * 16 + g_row] = make_float2(m0, l0);
      red_ml[warp * 16 + g_row + 8] = make_float2(m1, l1);
    }
  }
  __syncthreads();

  const bool single = (nsplit == 1);
  const size_t bh = (size_t)b * p.Hkv + kvh;
  float* part_o = p.ws_o + (bh * p.max_splits + split) * (size_t)p.nrp * D;
  float2* part_ml = p.ws_ml + (bh * p.max_splits + split) * (size_t)p.nrp;
  for (int e = tid; e < NRP * (D / 4); e += NT) {
    const int r = e / (D / 4), c = (e % (D / 4)) * 4;
    const int rt = r / 16, ri = r % 16;
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < WK; ++w) M = fmaxf(M, red_ml[(rt * WK + w) * 16 + ri].x);
    float L = 0.f;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    if (M != -INFINITY) {
#pragma unroll
      for (int w = 0; w < WK; ++w) {
        const float2 ml = red_ml[(rt * WK + w) * 16 + ri];
        const float sc = exp2f(ml.x - M);
        L += ml.y * sc;
        const float4 v = *reinterpret_cast<const float4*>(red_o + ((rt * WK + w) * 16 + ri) * D + c);
        acc.x += v.x * sc;
        acc.y += v.y * sc;
        acc.z += v.z * sc;
        acc.w += v.w * sc;
      }
    }
    if (single) {
      if (r < p.NR) {
        const float inv = 1.f / L;
        const int j = r / p.G, g = r % p.G;
        __nv_bfloat16* dst = p.out + (((size_t)b * p.R + j) * p.Hq + (size_t)kvh * p.G + g) * D + c;
        uint2 pk;
        pk.x = pack_bf16(acc.x * inv, acc.y * inv);
        pk.y = pack_bf16(acc.z * inv, acc.w * inv);
        *reinterpret_cast<uint2*>(dst) = pk;
      }
    } else {
      *reinterpret_cast<float4*>(part_o + (size_t)r * D + c) = acc;
      if (c == 0) part_ml[r] = make_float2(M, L);
    }
  }
  if (single) return;

  // Last arriving split of this (b, head) merges every split.
  __threadfence();
  __syncthreads();
  if (tid == 0) {
    const int prev = atomicAdd(p.tickets + bh, 1);
    s_last = (prev == nsplit - 1);
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();

  float* wsc = reinterpret_cast<float*>(smem_raw);      // [nsplit][NRP] weights
  float* inv_l = wsc + nsplit * NRP;                    // [NRP]
  const float* all_o = p.ws_o + bh * p.max_splits * (size_t)p.nrp * D;
  const float2* all_ml = p.ws_ml + bh * p.max_splits * (size_t)p.nrp;
  for (int r = tid; r < NRP; r += NT) {
    float M = -INFINITY;
    for (int s2 = 0; s2 < nsplit; ++s2) M = fmaxf(M, __ldcg(&all_ml[(size_t)s2 * p.nrp + r].x));
    float L = 0.f;
    for (int s2 = 0; s2 < nsplit; ++s2) {
      const float2 ml = __ldcg(&all_ml[(size_t)s2 * p.nrp + r]);
      const float sc = (ml.x == -INFINITY) ? 0.f : exp2f(ml.x - M);
      wsc[s2 * NRP + r] = sc;
      L += ml.y * sc;
    }
    inv_l[r] = (L > 0.f) ? 1.f / L : 0.f;
  }
  __syncthreads();
  for (int e = tid; e < p.NR * (D / 4); e += NT) {
    const int r = e / (D / 4), c = (e % (D / 4)) * 4;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int s2 = 0; s2 < nsplit; ++s2) {
      const float sc = wsc[s2 * NRP + r];
      const float4 v = __ldcg(reinterpret_cast<const float4*>(all_o + ((size_t)s2 * p.nrp + r) * D + c));
      acc.x += v.x * sc;
      acc.y += v.y * sc;
      acc.z += v.z * sc;
      acc.w += v.w * sc;
    }
    const float inv = inv_l[r];
    const int j = r / p.G, g = r % p.G;
    __nv_bfloat16* dst = p.out + (((size_t)b * p.R + j) * p.Hq + (size_t)kvh * p.G + g) * D + c;
    uint2 pk;
    pk.x = pack_bf16(acc.x * inv, acc.y * inv);
    pk.y = pack_bf16(acc.z * inv, acc.w * inv);
    *reinterpret_cast<uint2*>(dst) = pk;
  }
  if (tid == 0) p.tickets[bh] = 0;
}

template <int D, int MT, int WK>
size_t attn_smem_bytes(int max_splits) {
  const size_t pipe = (size_t)2 * NSTAGE * KT * D * sizeof(__nv_bfloat16);
  const size_t red = (size_t)MT * WK * 16 * D * sizeof(float) + (size_t)MT * WK * 16 * sizeof(float2);
  const size_t comb = ((size_t)max_splits * MT * 16 + MT * 16) * sizeof(float);
  size_t s = pipe;
  if (red > s) s = red;
  if (comb > s) s = comb;
  return s;
}

template <int D, int MT, int WK>
cudaError_t launch_t(const AttnParams& p, dim3 grid, cudaStream_t stream) {
  const size_t smem = attn_smem_bytes<D, MT, WK>(p.max_splits);
  static bool configured[64] = {false};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 64 && !configured[dev]) {
    cudaError_t e = cudaFuncSetAttribute(verify_attn_kernel<D, MT, WK>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024);
    if (e != cudaSuccess) return e;
    configured[dev] = true;
  }
  verify_attn_kernel<D, MT, WK><<<grid, MT * WK * 32, smem, stream>>>(p);
  return cudaGetLastError();
}

}  // namespace

AttnPlan plan_verify_attn(int B, int R, int Hq, int Hkv, int D, int max_ctx, int num_sms) {
  AttnPlan pl{};
  const int G = Hq / Hkv;
  const int NR = G * R;
  int mt = (NR + 15) / 16;
  if (mt <= 1) mt = 1;
  else if (mt <= 2) mt = 2;
  else if (mt <= 4) mt = 4;
  else mt = 8;
  pl.mt = mt;
  pl.wk = (mt >= 4) ? 1 : 4 / mt;
  pl.nrp = mt * 16;
  const int tiles_max = (max_ctx + R + KT - 1) / KT;
  const long long work = (long long)B * Hkv * tiles_max;
  const int ctas_per_sm = (D == 64) ? 4 : 2;
  const long long target = (long long)num_sms * ctas_per_sm * 6;   // about six waves
  int tps = (int)((work + target - 1) / target);
  if (tps < 2) tps = 2;
  const int max_split_cap = 96;
  if ((tiles_max + tps - 1) / tps > max_split_cap) tps = (tiles_max + max_split_cap - 1) / max_split_cap;
  pl.tiles_per_split = tps;
  pl.max_splits = (tiles_max + tps - 1) / tps;
  pl.ticket_bytes = (((size_t)B * Hkv * sizeof(int)) + 255) / 256 * 256;
  pl.partial_bytes = pl.max_splits > 1
                         ? (size_t)B * Hkv * pl.max_splits * pl.nrp * D * sizeof(float)
                         : 0;
  pl.ml_bytes = pl.max_splits > 1 ? (size_t)B * Hkv * pl.max_splits * pl.nrp * sizeof(float2) : 0;
  pl.ml_bytes = (pl.ml_bytes + 255) / 256 * 256;
  pl.total_bytes = pl.ticket_bytes + pl.partial_bytes + pl.ml_bytes;
  return pl;
}

cudaError_t launch_verify_attn(const AttnArgs& a, const AttnPlan& pl, int* err,
                               cudaStream_t stream) {
  AttnParams p{};
  p.q = a.q;
  p.k_blk = a.k_blk;
  p.v_blk = a.v_blk;
  p.k_pages = a.k_pages;
  p.v_pages = a.v_pages;
  p.page_table = a.page_table;
  p.ctx_len = a.ctx_len;
  p.out = a.out;
  uint8_t* ws = static_cast<uint8_t*>(a.ws);
  p.tickets = reinterpret_cast<int*>(ws);
  p.ws_ml = reinterpret_cast<float2*>(ws + pl.ticket_bytes);
  p.ws_o = reinterpret_cast<float*>(ws + pl.ticket_bytes + pl.ml_bytes);
  p.B = a.B;
  p.R = a.R;
  p.Hq = a.Hq;
  p.Hkv = a.Hkv;
  p.G = a.Hq / a.Hkv;
  p.NR = p.G * a.R;
  p.nrp = pl.nrp;
  p.max_pages = a.max_pages;
  p.num_pages = a.num_pages;
  p.tiles_per_split = pl.tiles_per_split;
  p.max_splits = pl.max_splits;
  p.scale_log2 = a.scale * 1.4426950408889634f;
  p.err = err;
  dim3 grid(pl.max_splits, a.Hkv, a.B);
#define COSPEC_ATTN_CASE(DD, MM, WW) \
  if (a.D == DD && pl.mt == MM && pl.wk == WW) return launch_t<DD, MM, WW>(p, grid, stream);
  COSPEC_ATTN_CASE(128, 1, 4)
  COSPEC_ATTN_CASE(128, 2, 2)
  COSPEC_ATTN_CASE(128, 4, 1)
  COSPEC_ATTN_CASE(128, 8, 1)
  COSPEC_ATTN_CASE(64, 1, 4)
  COSPEC_ATTN_CASE(64, 2, 2)
  COSPEC_ATTN_CASE(64, 4, 1)
  COSPEC_ATTN_CASE(64, 8, 1)
#undef COSPEC_ATTN_CASE
  return cudaErrorInvalidValue;
}

}  // namespace cospec
