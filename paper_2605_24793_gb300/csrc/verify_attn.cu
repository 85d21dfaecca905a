// Verify attention of the K+1 block rows over a paged bf16 KV cache
// (teacher-forced verification pass, Sec. 3.1 Eq. 2 of the paper).
//
// One CTA owns (sequence b, KV head, row group of <= 64 query rows, KV
// split).  The KV range of a (b, head) is split over the CTAs of one
// thread-block cluster; every CTA streams its 64-token K/V tiles (4 pages)
// once with TMA tensor loads -- one 3-D box per page and tensor brings both
// 128-byte halves of the page's 16 rows, 128B-swizzled, into a 3-stage
// mbarrier ring; one producer warp issues the K boxes and another the V
// boxes (a warp's bulk copies are processed one after another) -- and
// multiplies each tile against ALL query rows of the group that read this
// KV head (the G = Hq/Hkv heads times the block rows, row index j*G + g).
// Q.K^T and P.V run on bf16 tensor cores (mma.m16n8k16, fp32 accumulation),
// the softmax is online in base 2.  The block's own keys (causal inside the
// block, or all of them with the full mask) land in a region of their own
// and are taken after the cache tiles by the last CTA of the cluster.
// Partial (max, sum, O) of the cluster merge through distributed shared
// memory, each CTA finishing a slice of the rows, so no workspace and no
// extra launch are needed.
#include <cuda.h>
#include <math.h>

#include "cospec_device.cuh"
#include "cospec_internal.h"

namespace cospec {

namespace {

constexpr int KT = 64;            // keys per cache tile (4 pages)
constexpr int PAGE = 16;          // page size (fixed)
constexpr int ROWB = 128;         // bytes of one swizzled smem row (64 bf16)
constexpr int NSTAGE = 3;

struct AttnParams {
  const __nv_bfloat16* q;
  const int32_t* page_table;
  const int32_t* ctx_len;
  __nv_bfloat16* out;
  int B, R, Hq, Hkv, G;
  int NRT;         // query rows of a (sequence, KV head): G * R
  int RG;          // row groups of at most 64 rows per (sequence, KV head)
  int max_pages, num_pages;
  float scale_log2;
  int kv_stable;
  int block_full;  // block rows see every block row (not only rows <= their own)
  int* err;
};

template <int D, int MT, int WK>
struct Layout {
  static constexpr int H = D / 64;                 // 128-byte halves of a key row
  static constexpr int PAGEB = H * PAGE * ROWB;    // one page of K (or V): [H][16 rows][128 B]
  static constexpr int KV = 4 * PAGEB;             // K (or V) of a 64-key tile
  static constexpr int STAGE = 2 * KV;             // K then V
  static constexpr int NRP = MT * 16;
  static constexpr int PD = D + 8;                 // padded fp32 row of a partial (no bank conflicts)
  static constexpr int ROWP = PD * 4;              // bytes of a partial row: O[D], (m, l), pad
  static constexpr int RED = (WK > 1) ? MT * WK * 16 * ROWP : 0;
  // After the last tile the ring holds, in order: RED (per-warp partials
  // when keys are split over warps), PART (this CTA's partial, NRP rows) and
  // RECV [S][rows per owner] (S * ceil(NR / S) <= NRP + 15 rows), where the
  // cluster's CTAs push their partials.  RECV overlaps neither RED nor PART,
  // so peers may push while this CTA still reduces its own partial.
  static constexpr int PART = RED;
  static constexpr int PART_END = PART + NRP * ROWP;
  static constexpr int RECV = PART_END;
  static constexpr int RECV_END = RECV + (NRP + 15) * ROWP;
  static_assert(RECV_END <= NSTAGE * STAGE, "partials must fit in the stage ring");
  static constexpr int BLK = NSTAGE * STAGE;       // block K/V (1024-aligned)
  // the block region holds 2*H halves of KBR rows (KBR = 16, 32, 48 or 64, runtime)
  static constexpr int blk_half(int kbr) { return kbr * ROWB; }
  static constexpr int total(int kbr) { return BLK + 2 * H * kbr * ROWB; }
  // The launch adds 1024 bytes to align the base; the 2*NSTAGE+2 barriers
  // (full[NSTAGE], empty[NSTAGE], block, received partials) and the index of
  // the CTA's sequence take 80 bytes of that slack, before the aligned base
  // or after the end, whichever side has room, so that two CTAs of 32 block
  // rows still share one SM.
  static constexpr int NBAR_BYTES = (2 * NSTAGE + 2) * 8 + 16;   // + the sequence slot
};

// Shared-memory byte offset of 16-byte chunk `ch` (of D/8) of key row `key`
// in a region laid out as groups of 16 keys (`group_bytes` apart), each group
// holding its 128-byte half rows half by half (`half_bytes` apart), every
// 128-byte row swizzled by the TMA 128B pattern.
CS_DEV uint32_t kv_off(int key, int ch, uint32_t group_bytes, uint32_t half_bytes) {
  return (uint32_t)(key >> 4) * group_bytes + (uint32_t)(ch >> 3) * half_bytes +
         (uint32_t)(key & 15) * ROWB + (uint32_t)(((ch & 7) ^ (key & 7)) * 16);
}

// Online-softmax update of one warp's 16 rows with NK keys held in shared
// memory (K and V regions laid out as in kv_off).  Key k of the region sits
// at row key0 + k and has index kidx0 + k for masking; row r sees key index
// <= lim_r.
template <int D, int NK>
CS_DEV void attend(uint32_t sk, uint32_t sv, uint32_t group_bytes, uint32_t half_bytes,
                   int key0, int kidx0,
                   bool need_mask, int lim0, int lim1, float scale_log2,
                   const uint32_t (&qf)[D / 16][4], float (&o)[D / 8][4], float& m0, float& m1,
                   float& l0, float& l1, int lane) {
  const int c4 = lane & 3;
  float s[NK / 8][4];
#pragma unroll
  for (int nt = 0; nt < NK / 8; ++nt) s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.f;
#pragma unroll
  for (int kk = 0; kk < D / 16; kk += 2) {
    const int ch = kk * 2 + (lane >> 3);            // 16-byte chunk of the key row
#pragma unroll
    for (int nt = 0; nt < NK / 8; ++nt) {
      const int key = key0 + nt * 8 + (lane & 7);
      const uint32_t addr = sk + kv_off(key, ch, group_bytes, half_bytes);
      uint32_t b0, b1, b2, b3;
      ldsm_x4(addr, b0, b1, b2, b3);
      mma_16816(s[nt], qf[kk], b0, b1);
      mma_16816(s[nt], qf[kk + 1], b2, b3);
    }
  }
  float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
  for (int nt = 0; nt < NK / 8; ++nt) {
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      const int kidx = kidx0 + nt * 8 + 2 * c4 + e;
      float v0 = s[nt][e] * scale_log2;
      float v1 = s[nt][2 + e] * scale_log2;
      if (need_mask) {
        if (kidx > lim0) v0 = -INFINITY;
        if (kidx > lim1) v1 = -INFINITY;
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
  const float a0 = exp2_approx(m0 - base0), a1 = exp2_approx(m1 - base1);
  // Rescale the running output only when some row's maximum moved.
  if (__any_sync(0xffffffffu, mn0 != m0 || mn1 != m1)) {
    l0 *= a0;
    l1 *= a1;
#pragma unroll
    for (int i = 0; i < D / 8; ++i) {
      o[i][0] *= a0;
      o[i][1] *= a0;
      o[i][2] *= a1;
      o[i][3] *= a1;
    }
  }
  m0 = mn0;
  m1 = mn1;
  uint32_t pf[NK / 16][4];
#pragma unroll
  for (int nt = 0; nt < NK / 8; ++nt) {
    const float p0 = exp2_approx(s[nt][0] - base0), p1 = exp2_approx(s[nt][1] - base0);
    const float p2 = exp2_approx(s[nt][2] - base1), p3 = exp2_approx(s[nt][3] - base1);
    l0 += p0 + p1;
    l1 += p2 + p3;
    pf[nt / 2][(nt % 2) * 2 + 0] = pack_bf16(p0, p1);
    pf[nt / 2][(nt % 2) * 2 + 1] = pack_bf16(p2, p3);
  }
#pragma unroll
  for (int kk2 = 0; kk2 < NK / 16; ++kk2) {
    const int key = key0 + kk2 * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
#pragma unroll
    for (int nd = 0; nd < D / 8; nd += 2) {
      const int ch = nd + (lane >> 4);
      const uint32_t addr = sv + kv_off(key, ch, group_bytes, half_bytes);
      uint32_t b0, b1, b2, b3;
      ldsm_x4_t(addr, b0, b1, b2, b3);
      mma_16816(o[nd], pf[kk2], b0, b1);
      mma_16816(o[nd + 1], pf[kk2], b2, b3);
    }
  }
}

// GEN 0: the verify block (causal, <= 32 rows), a specialised block path.
// GEN 1 / 2: blocks of more than 32 rows or a full block mask (the
// arbitrator's region) take a general block path; 2 marks more than 32 block
// keys in the 64-row variant.
// The 64-row variant with at most 32 block keys declares room for two CTAs of
// six warps per SM, which holds it at 168 registers: two of its five-warp
// CTAs then fit the register file of each SM sub-partition (three warps of
// 168).  With more block keys the shared memory allows one CTA per SM, and
// it keeps its registers (no spills).
template <int D, int MT, int WK, int GEN>
__global__ void __launch_bounds__(MT >= 4 && GEN < 2 ? 192 : MT * WK * 32 + 64,
                                  MT >= 4 && GEN < 2 ? 2 : (GEN == 2 ? 1 : 0))
    verify_attn_kernel(const __grid_constant__ CUtensorMap map_kp,
                       const __grid_constant__ CUtensorMap map_vp,
                       const __grid_constant__ CUtensorMap map_kb,
                       const __grid_constant__ CUtensorMap map_vb, const AttnParams p) {
  using LY = Layout<D, MT, WK>;
  constexpr int NWARPS = MT * WK;        // consumer warps; warps NWARPS (K) and NWARPS+1 (V) issue the loads
  constexpr int NTC = NWARPS * 32;
  constexpr int NTT = NTC + 64;
  constexpr int KW = KT / WK;            // cache keys of a tile handled by one warp
  constexpr int H = LY::H;
  constexpr int NRP = LY::NRP;
  constexpr int PD = LY::PD;
  static_assert(KW % 16 == 0, "keys per warp must be a multiple of 16");

  extern __shared__ __align__(16) uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(
      smem - smem_raw >= LY::NBAR_BYTES ? smem_raw : smem + LY::total((p.R + 15) & ~15));
  uint64_t* empty = full + NSTAGE;
  uint64_t* blk_full = empty + NSTAGE;
  uint64_t* recv_bar = blk_full + 1;     // partials received from the cluster
  volatile int* seq_slot = reinterpret_cast<volatile int*>(recv_bar + 1);   // this CTA's sequence
  uint8_t* blk_k = smem + LY::BLK;       // block keys: 2*H halves of KBR rows

  const int S = (int)cluster_nctarank();
  const int rank = (int)cluster_ctarank();
  const int kvh = blockIdx.y / p.RG, rg = blockIdx.y % p.RG;
  const int row_g0 = rg * 64;                      // first query row of this group
  const int NR = min(64, p.NRT - row_g0);          // rows of this group (<= NRP)
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  if (tid == 0) {
    for (int s2 = 0; s2 < NSTAGE; ++s2) {
      mbar_init(&full[s2], 2);           // the K and the V producer
      mbar_init(&empty[s2], NWARPS);
    }
    mbar_init(blk_full, 1);
    mbar_init(recv_bar, 1);
    fence_barrier_init();
  }
  __syncthreads();
  // Let the next kernel of the stream start launching right away: its CTAs
  // take the SMs' free slots and, with the stable-cache promise, stream their
  // cache tiles while this kernel computes (their own waits keep the order).
  griddep_launch_dependents();
  // Without the stable-cache promise, wait for the previous kernel before
  // reading anything; with it, only q and the block K/V (read below, after
  // the wait) may come from that kernel, so the cache stream starts now.
  if (!p.kv_stable) griddep_wait();

  // Sequences are taken longest context first (blockIdx.z = rank, ties by
  // index), so that the long ones start early and the short ones fill in
  // behind them at the end of the launch.
  const int b = (p.B > 1 && p.B <= RANK_MAX_B) ? sequence_by_rank(p.ctx_len, p.B, (int)blockIdx.z, seq_slot)
                        : (int)blockIdx.z;
  const int C = p.ctx_len[b];
  const bool bad = (C < 0) || (C > p.max_pages * PAGE);
  if (bad && rank == 0 && kvh == 0 && tid == 0) set_err(p.err, ERR_CTX);
  // No early exit: every CTA of the cluster takes part in the merge below.
  const int nct = bad ? 0 : (C + KT - 1) / KT;               // cache tiles of this sequence
  const int tps = (nct + S - 1) / S;
  const int t_begin = min(nct, rank * tps);
  const int n = min(nct, t_begin + tps) - t_begin;
  // The block's own keys go to the last CTA, which never has more cache tiles.
  const bool do_blk = !bad && rank == S - 1;
  const int nv = n;
  const int npages = (C + PAGE - 1) / PAGE;
  const int KBR = (p.R + 15) & ~15;                          // block keys padded to 16
  uint8_t* blk_v = blk_k + H * KBR * ROWB;                   // each [H][KBR rows][128 B]

  float o[D / 8][4];
  float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
  const int g_row = lane >> 2, c4 = lane & 3;
  const int wr = warp / WK, wk = warp % WK;
  const int r0 = wr * 16 + g_row, r1 = r0 + 8;

  if (warp >= NWARPS) {
    // ---------------------------------------------------------- producer warps
    // A warp's bulk copies are processed one after another; two warps (one
    // for K, one for V) double the rate at which a CTA can pull tiles.
    const int tensor = warp - NWARPS;    // 0: K, 1: V
    if (lane == 0) {
      tma_prefetch_desc(&map_kp);
      tma_prefetch_desc(&map_vp);
    }
    // KV is read once per row group: with several groups per (sequence, head)
    // (running side by side) keep it in L2 for the siblings
    const uint64_t pol = p.RG > 1 ? l2_policy_evict_normal() : l2_policy_evict_first();
    bool waited = !p.kv_stable;
    // The block K/V is written by the previous kernel: the V producer of the
    // CTA that owns the block fills its ring with cache tiles first (they
    // may stream early), then waits for that kernel and loads the block.
    const bool blk_here = do_blk && tensor == 1;
    const int blk_after = min(nv, NSTAGE);   // cache tiles issued before the block
    auto issue_block = [&]() {
      if (!waited) {
        griddep_wait();
        waited = true;
      }
      if (lane == 0) {
        // one box per tensor: KBR rows from block row 0 of this head, both
        // halves (rows past R belong to the next sequence or are zero-filled;
        // masked)
        mbar_arrive_expect_tx(blk_full, (uint32_t)(H * 2 * ROWB * KBR));   // KBR-row boxes
        tma_load_4d(smem_u32(blk_k), &map_kb, blk_full, 0, b * p.R, 0, kvh, pol);
        tma_load_4d(smem_u32(blk_v), &map_vb, blk_full, 0, b * p.R, 0, kvh, pol);
      }
      __syncwarp();
    };
    if (blk_here && blk_after == 0) issue_block();
    const int* ptab = p.page_table + (size_t)b * p.max_pages + (size_t)t_begin * 4;
    const int my_pages = min(n * 4, npages - t_begin * 4);   // page-table entries of this CTA
    int pid = 0;
    for (int vt = 0; vt < nv; ++vt) {
      if ((vt & 7) == 0) {                 // 32 page ids = the next 8 tiles, one per lane
        const int e = vt * 4 + lane;
        pid = (e < my_pages) ? __ldg(ptab + e) : 0;
      }
      const int st = vt % NSTAGE;
      if (vt >= NSTAGE && !mbar_wait(&empty[st], (uint32_t)((vt / NSTAGE) - 1) & 1u))
        set_err(p.err, ERR_TIMEOUT);
      uint8_t* kb = smem + st * LY::STAGE;
      {
        const int np = min(4, npages - (t_begin + vt) * 4);
        // lanes 0..3: page `lane` of the tile, this warp's tensor
        int pgid = __shfl_sync(0xffffffffu, pid, (vt & 7) * 4 + (lane & 3));
        if (lane == 0) mbar_arrive_expect_tx(&full[st], (uint32_t)(np * LY::PAGEB));
        __syncwarp();
        if (lane < np) {
          if ((unsigned)pgid >= (unsigned)p.num_pages) {
            set_err(p.err, ERR_PAGE);
            pgid = 0;
          }
          const int y = (pgid * p.Hkv + kvh) * PAGE;
          tma_load_3d(smem_u32(kb + tensor * LY::KV + lane * LY::PAGEB),
                      tensor ? (const void*)&map_vp : (const void*)&map_kp, &full[st], 0, y, 0, pol);
        }
      }
      if (vt == NSTAGE - 1) {
        // The ring is full: pull the next two tiles' pages into L2 so their
        // loads, issued once stages free up, skip most of the HBM latency.
        const int e = NSTAGE * 4 + lane;                         // lanes 0..7: 8 pages
        const int pg = __shfl_sync(0xffffffffu, pid, e & 31);
        if (lane < 8 && e < my_pages && (unsigned)pg < (unsigned)p.num_pages)
          tma_prefetch_l2_3d(tensor ? (const void*)&map_vp : (const void*)&map_kp, 0,
                             (pg * p.Hkv + kvh) * PAGE, 0);
      }
      __syncwarp();
      if (blk_here && vt == blk_after - 1) issue_block();
    }
    if (!waited) griddep_wait();
  } else {
    // ---------------------------------------------------------- consumer warps
    if (p.kv_stable) {
      // Warm L2 with this CTA's query rows (writes by the previous kernel
      // still land in L2 first), then wait for that kernel.
      for (int e = tid; e < NR * (D * 2 / 128); e += NTC) {
        const int r = row_g0 + e / (D * 2 / 128), part_ = e % (D * 2 / 128);
        const int j = r / p.G, g = r % p.G;
        prefetch_l2(p.q + (((size_t)b * p.R + j) * p.Hq + (size_t)kvh * p.G + g) * D + part_ * 64);
      }
      griddep_wait();                    // q is written by the previous kernel
    }
    // Query fragments (A operand, 16 rows x D) of this warp's row tile.
    uint32_t qf[D / 16][4];
    {
      auto row_ptr = [&](int r) -> const __nv_bfloat16* {
        if (r >= NR) return nullptr;
        const int j = (row_g0 + r) / p.G, g = (row_g0 + r) % p.G;
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
    const int j0 = min((row_g0 + r0) / p.G, p.R - 1), j1 = min((row_g0 + r1) / p.G, p.R - 1);
#pragma unroll
    for (int i = 0; i < D / 8; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;

    for (int it = 0; it < n; ++it) {
      const int st = it % NSTAGE;
      if (!mbar_wait(&full[st], (uint32_t)(it / NSTAGE) & 1u)) set_err(p.err, ERR_TIMEOUT);
      uint8_t* kb = smem + st * LY::STAGE;
      uint8_t* vb = kb + LY::KV;
      // Rows past the valid keys of this tile may hold stale or unwritten
      // bytes: zero their V rows so that 0-weight keys contribute exactly 0.
      const int valid_rows = min(KT, C - (t_begin + it) * KT);
      if (valid_rows < KT) {
        const int nz = (KT - valid_rows) * H * (ROWB / 16);
        for (int e = tid; e < nz; e += NTC) {
          const int row = valid_rows + e / (H * (ROWB / 16));
          const int rem = e % (H * (ROWB / 16));
          *reinterpret_cast<uint4*>(vb + (row >> 4) * LY::PAGEB + (rem / (ROWB / 16)) * (PAGE * ROWB) +
                                    (row & 15) * ROWB + (rem % (ROWB / 16)) * 16) =
              make_uint4(0u, 0u, 0u, 0u);
        }
        fence_proxy_async_smem();
        named_bar_sync(1, NTC);
      }
      const int kidx0 = (t_begin + it) * KT + wk * KW;
      attend<D, KW>(smem_u32(kb), smem_u32(vb), LY::PAGEB, PAGE * ROWB, wk * KW, kidx0,
                    valid_rows < KT, C - 1, C - 1, p.scale_log2, qf, o, m0, m1, l0, l1, lane);
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty[st]);
    }
    if (do_blk) {
      if (!mbar_wait(blk_full, 0)) set_err(p.err, ERR_TIMEOUT);
      // rows R..KBR-1 of the block region were never written: zero their V
      const int nz = (KBR - p.R) * H * (ROWB / 16);
      for (int e = tid; e < nz; e += NTC) {
        const int row = p.R + e / (H * (ROWB / 16));
        const int rem = e % (H * (ROWB / 16));
        *reinterpret_cast<uint4*>(blk_v + (rem / (ROWB / 16)) * KBR * ROWB + row * ROWB +
                                  (rem % (ROWB / 16)) * 16) = make_uint4(0u, 0u, 0u, 0u);
      }
      named_bar_sync(1, NTC);
      if (wk == 0) {
        const uint32_t sk = smem_u32(blk_k), sv = smem_u32(blk_v);
        if constexpr (GEN == 0) {
          // causal: block key j is seen by the rows of block rows >= j
          if (KBR == 16)
            attend<D, 16>(sk, sv, PAGE * ROWB, 16 * ROWB, 0, 0, true, j0, j1, p.scale_log2, qf, o,
                          m0, m1, l0, l1, lane);
          else
            attend<D, 32>(sk, sv, PAGE * ROWB, 32 * ROWB, 0, 0, true, j0, j1, p.scale_log2, qf, o,
                          m0, m1, l0, l1, lane);
        } else {
          // any block length up to 64, causal or full (every block row seen
          // by every row): 16 keys at a time
          const int b0 = p.block_full ? p.R - 1 : j0, b1 = p.block_full ? p.R - 1 : j1;
          for (int g0 = 0; g0 < KBR; g0 += 16)
            attend<D, 16>(sk, sv, PAGE * ROWB, KBR * ROWB, g0, g0, true, b0, b1, p.scale_log2, qf, o,
                          m0, m1, l0, l1, lane);
        }
      }
    }
    // After a timed-out wait a copy may still be in flight: wait (bounded)
    // for the last fill of every stage before the ring is reused.
    if (tid == 0) {
      for (int st = 0; st < NSTAGE && st < nv; ++st) {
        const int last = st + ((nv - 1 - st) / NSTAGE) * NSTAGE;
        mbar_wait(&full[st], (uint32_t)(last / NSTAGE) & 1u);
      }
      if (do_blk) mbar_wait(blk_full, 0);
    }
    l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
    l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
    l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
    l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
  }
  __syncthreads();
  // The ring is idle from here on.  Tell the cluster (its CTAs may push into
  // RECV once every CTA has arrived) and build this CTA's partial meanwhile.
  const int rpo = (NR + S - 1) / S;      // rows finished by each owner
  if (S > 1) {
    if (tid == 0) mbar_arrive_expect_tx(recv_bar, (uint32_t)(S * rpo * LY::ROWP));
    cluster_arrive_relaxed();
  }

  // CTA partial: rows of every warp, key groups merged (stage ring reused).
  float* part = reinterpret_cast<float*>(smem + LY::PART);
  if constexpr (WK > 1) {
    // Key groups of a row tile merge pairwise in registers: every lane of a
    // partner warp holds the same (row, column) elements, so one writes its
    // (O, m, l) and the other folds them in (a tree over the WK groups).
    float* red = reinterpret_cast<float*>(smem);                          // [NWARPS][16][PD]
#pragma unroll
    for (int step = 1; step < WK; step <<= 1) {
      const bool writer = warp < NWARPS && (wk % (2 * step)) == step;
      const bool reader = warp < NWARPS && (wk % (2 * step)) == 0;
      if (writer) {
        float* wo = red + warp * 16 * PD;
#pragma unroll
        for (int nd = 0; nd < D / 8; ++nd) {
          const int col = nd * 8 + 2 * c4;
          *reinterpret_cast<float2*>(wo + g_row * PD + col) = make_float2(o[nd][0], o[nd][1]);
          *reinterpret_cast<float2*>(wo + (g_row + 8) * PD + col) = make_float2(o[nd][2], o[nd][3]);
        }
        if (c4 == 0) {
          *reinterpret_cast<float2*>(wo + g_row * PD + D) = make_float2(m0, l0);
          *reinterpret_cast<float2*>(wo + (g_row + 8) * PD + D) = make_float2(m1, l1);
        }
      }
      __syncthreads();
      if (reader) {
        const float* po = red + (warp + step) * 16 * PD;
        const float2 ml0 = *reinterpret_cast<const float2*>(po + g_row * PD + D);
        const float2 ml1 = *reinterpret_cast<const float2*>(po + (g_row + 8) * PD + D);
        const float M0 = fmaxf(m0, ml0.x), M1 = fmaxf(m1, ml1.x);
        const float a0 = (M0 == -INFINITY) ? 0.f : exp2_approx(m0 - M0);
        const float b0 = (M0 == -INFINITY) ? 0.f : exp2_approx(ml0.x - M0);
        const float a1 = (M1 == -INFINITY) ? 0.f : exp2_approx(m1 - M1);
        const float b1 = (M1 == -INFINITY) ? 0.f : exp2_approx(ml1.x - M1);
#pragma unroll
        for (int nd = 0; nd < D / 8; ++nd) {
          const int col = nd * 8 + 2 * c4;
          const float2 v0 = *reinterpret_cast<const float2*>(po + g_row * PD + col);
          const float2 v1 = *reinterpret_cast<const float2*>(po + (g_row + 8) * PD + col);
          o[nd][0] = o[nd][0] * a0 + v0.x * b0;
          o[nd][1] = o[nd][1] * a0 + v0.y * b0;
          o[nd][2] = o[nd][2] * a1 + v1.x * b1;
          o[nd][3] = o[nd][3] * a1 + v1.y * b1;
        }
        l0 = l0 * a0 + ml0.y * b0;
        l1 = l1 * a1 + ml1.y * b1;
        m0 = M0;
        m1 = M1;
      }
      if (2 * step < WK) __syncthreads();   // the next level reuses the buffer
    }
  }
  // The first key group of every row tile (all warps when WK == 1) writes
  // the CTA's partial rows: O[0..D) then (m, l) at D, D+1 (fp32, padded to PD).
  if (warp < NWARPS && wk == 0) {
#pragma unroll
    for (int nd = 0; nd < D / 8; ++nd) {
      const int col = nd * 8 + 2 * c4;
      *reinterpret_cast<float2*>(part + r0 * PD + col) = make_float2(o[nd][0], o[nd][1]);
      *reinterpret_cast<float2*>(part + r1 * PD + col) = make_float2(o[nd][2], o[nd][3]);
    }
    if (c4 == 0) {
      *reinterpret_cast<float2*>(part + r0 * PD + D) = make_float2(m0, l0);
      *reinterpret_cast<float2*>(part + r1 * PD + D) = make_float2(m1, l1);
    }
  }
  fence_proxy_async_smem();              // the bulk copies below read `part`
  __syncthreads();

  // Reduce-scatter over the cluster: owner o finishes rows [o*rpo, (o+1)*rpo).
  // Each CTA sends its partial rows to their owners with one bulk shared-
  // to-shared copy per owner (thread-level remote accesses are slow); the
  // owner merges the S received copies from its own shared memory.
  const float* src = part;
  if (S > 1) {
    cluster_wait();                      // every CTA's RECV is free and its barrier armed
    float* recv = reinterpret_cast<float*>(smem + LY::RECV);   // [S][rpo][PD] at each owner
    // one issuing thread in each of four warps: a warp's bulk copies are
    // processed one after another
    if (lane == 0 && warp < 4) {
      const uint32_t recv_u = smem_u32(recv), bar_u = smem_u32(recv_bar);
      for (int o = warp; o < S; o += 4)
        bulk_copy_s2s(dsmem_map(recv_u + (uint32_t)(rank * rpo * LY::ROWP), (uint32_t)o),
                      smem_u32(part + o * rpo * PD), (uint32_t)(rpo * LY::ROWP),
                      dsmem_map(bar_u, (uint32_t)o));
    }
    if (!mbar_wait(recv_bar, 0)) set_err(p.err, ERR_TIMEOUT);
    src = recv;
    // Everything addressed to this CTA has landed.  Once every CTA has said
    // so, no copy reads or writes this CTA's shared memory any more: arrive
    // now, wait at the very end, and merge in between.
    cluster_arrive_relaxed();
  }
  const int row0 = rank * rpo;
  // Per owned row: one warp forms the common maximum over the S partials and
  // each partial's weight exp2(m_s - M) / L (kept in the idle block region);
  // then every output chunk is a plain weighted sum.
  float* scl = reinterpret_cast<float*>(blk_k);            // [S][rpo]
  for (int rr = warp; rr < rpo; rr += NTT / 32) {
    if (row0 + rr >= NR) break;
    const float2 ml = (lane < S) ? *reinterpret_cast<const float2*>(src + (lane * rpo + rr) * PD + D)
                                 : make_float2(-INFINITY, 0.f);
    float M = ml.x;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, off));
    const float sc = (M == -INFINITY || ml.x == -INFINITY) ? 0.f : exp2_approx(ml.x - M);
    float L = ml.y * sc;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) L += __shfl_xor_sync(0xffffffffu, L, off);
    if (lane < S) scl[lane * rpo + rr] = (L > 0.f) ? sc / L : 0.f;
  }
  __syncthreads();
  for (int e = tid; e < rpo * (D / 4); e += NTT) {
    const int rr = e / (D / 4), c = (e % (D / 4)) * 4;
    const int r = row0 + rr;
    if (r >= NR) break;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 4
    for (int s2 = 0; s2 < S; ++s2) {
      const float w = scl[s2 * rpo + rr];
      const float4 v = *reinterpret_cast<const float4*>(src + (s2 * rpo + rr) * PD + c);
      acc.x += v.x * w;
      acc.y += v.y * w;
      acc.z += v.z * w;
      acc.w += v.w * w;
    }
    const int j = (row_g0 + r) / p.G, g = (row_g0 + r) % p.G;
    // the sequence index is read again here rather than kept through the loop
    const int bo = (p.B > 1 && p.B <= RANK_MAX_B) ? *seq_slot : (int)blockIdx.z;
    __nv_bfloat16* dst = p.out + (((size_t)bo * p.R + j) * p.Hq + (size_t)kvh * p.G + g) * D + c;
    uint2 pk;
    pk.x = pack_bf16(acc.x, acc.y);
    pk.y = pack_bf16(acc.z, acc.w);
    *reinterpret_cast<uint2*>(dst) = pk;
  }
  if (S > 1) cluster_wait();             // every copy out of this CTA has landed
}


// Limits already set on each instantiation of the kernel.
template <int D, int MT, int WK, int GEN>
KernelLimits& attn_limits() {
  static KernelLimits lim;
  return lim;
}

template <int D, int MT, int WK, int GEN>
cudaError_t launch_t(const CUtensorMap* maps, const AttnParams& p, int S, int B, int Hkv,
                     cudaStream_t stream) {
  using LY = Layout<D, MT, WK>;
  const size_t smem = LY::total((p.R + 15) & ~15) + 1024;
  auto kern = verify_attn_kernel<D, MT, WK, GEN>;
  const cudaError_t e = ensure_kernel_limits((const void*)kern, attn_limits<D, MT, WK, GEN>(), smem, true);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(S, Hkv * p.RG, B);
  cfg.blockDim = dim3(MT * WK * 32 + 64, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = S;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, kern, maps[0], maps[1], maps[2], maps[3], p);
}

template <int D, int MT, int WK>
int max_cluster_t(int S, int Hkv, int B, int kbr) {
  using LY = Layout<D, MT, WK>;
  // every block path has the same shared-memory layout for a block size, and
  // the paths used with a block size the same register budget; the occupancy
  // query needs the limit at least at the queried size
  constexpr int GW = MT >= 4 ? 2 : 1;
  auto kern = kbr > 32 ? verify_attn_kernel<D, MT, WK, GW> : verify_attn_kernel<D, MT, WK, 0>;
  KernelLimits& lim = kbr > 32 ? attn_limits<D, MT, WK, GW>() : attn_limits<D, MT, WK, 0>();
  if (ensure_kernel_limits((const void*)kern, lim, LY::total(kbr) + 1024, true) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(S, Hkv, B);
  cfg.blockDim = dim3(MT * WK * 32 + 64, 1, 1);
  cfg.dynamicSmemBytes = LY::total(kbr) + 1024;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = S;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return n;
}

int variant_mt(int NR) {   // NR <= 64
  if (NR <= 16) return 1;
  if (NR <= 32) return 2;
  return 4;
}

#define COSPEC_ATTN_VARIANTS(X) \
  X(128, 1, 4) X(128, 2, 2) X(128, 4, 1) X(64, 1, 4) X(64, 2, 2) X(64, 4, 1)

}  // namespace

AttnPlan plan_verify_attn(int B, int R, int Hq, int Hkv, int D, int max_ctx, int num_sms,
                          bool kv_stable, const ResidentFn& resident) {
  AttnPlan pl{};
  const int NRT = (Hq / Hkv) * R;
  const int RG = (NRT + 63) / 64;                  // row groups of at most 64 rows
  const int NR = NRT < 64 ? NRT : 64;
  pl.mt = variant_mt(NR);
  pl.wk = (pl.mt >= 4) ? 1 : 4 / pl.mt;
  pl.nrp = pl.mt * 16;
  const int G = Hq / Hkv;
  // More than 32 query rows per KV head: the mma.sync kernel is bound by its
  // legacy tensor-core rate there and the tcgen05 kernel (one CTA per SM,
  // deep ring, every row of a head in one CTA) takes over at every batch
  // size.  Up to 32 rows the mma.sync kernel keeps the latency-bound small
  // batches and the two-CTAs-per-SM streaming of the large ones.
  int S = 1;
  const int jb = G <= 128 ? 128 / G : 1;
  const int jbq = R < jb ? R : jb;
  if (tcq_attn_supported(D, G) && G <= 64 && G * jbq > 32) {
    // tcgen05 kernel with the query rows as the MMA M dimension: row groups
    // of whole block rows, at most 128 query rows, so a KV head's rows share
    // one cache stream (K <= 31 at G = 4, K <= 15 at G = 8)
    pl.kind = 1;
    pl.jb = jb;
    pl.jbq = jbq;
    pl.rg = (R + pl.jb - 1) / pl.jb;
    pl.nt = 128;
    // 128-key tiles; one CTA per SM (a 192 KB stage ring); about one wave
    // of CTAs or a little more (with the longest contexts started first the
    // tail balances itself and every further split only adds merges), at
    // least eight tiles per CTA unless the batch is small (the prologue, the
    // query load and the merge are fixed costs), no CTA with more than 256
    // tiles.
    const int tiles_tc = (max_ctx + 127) / 128;
    pl.units = (long long)B * Hkv * pl.rg;
    const long long wave_tc = ((long long)num_sms + pl.units - 1) / (pl.units > 0 ? pl.units : 1);
    const long long len_tc = (tiles_tc + 255) / 256;
    const long long want_tc = wave_tc > len_tc ? wave_tc : len_tc;
    // a small batch (latency-bound): every cluster resident at once, and
    // down to two tiles per CTA
    pl.one_wave = (pl.units * 4 <= num_sms && len_tc <= 1) ? 1 : 0;
    if (pl.one_wave) {
      int s = 16;
      while (s > 1 && (s * 2 > tiles_tc || resident(pl, s) < pl.units)) --s;
      pl.cluster = s;
      return pl;
    }
    const int min_tiles = 8;
    while (S < 16 && S < want_tc && (S * 2) * min_tiles <= tiles_tc) S *= 2;
  } else {
    // Split each (sequence, head, row group) over a cluster of S CTAs: about
    // one wave of CTAs (as many as are resident at once), no CTA with more
    // than 256 cache tiles (long contexts), at least 4 tiles per CTA, at
    // most 16 CTAs per cluster.
    pl.kind = 0;
    const int tiles = (max_ctx + KT - 1) / KT;
    pl.units = (long long)B * Hkv * RG;
    long long slots = resident(pl, 1);
    if (slots < 1) slots = num_sms;
    const long long want_wave = (slots + pl.units - 1) / (pl.units > 0 ? pl.units : 1);
    const long long want_len = (tiles + 255) / 256;
    const long long want = want_wave > want_len ? want_wave : want_len;
    while (S < 16 && S < want && (S * 2) * 4 <= tiles) S *= 2;
    // A batch of a few units (at most a quarter of the slots) is bound by the
    // latency of one CTA's tile loop and the cluster merge, and a second wave
    // of clusters (the GPU places whole clusters inside one GPC) doubles it:
    // take the largest even split up to 16, at least four tiles per CTA,
    // whose clusters are all resident at once (Qwen3-8B batch 2: 12 splits
    // 10.7 us per layer, 8 12.5 us, 16 -- a second wave -- 16.2 us; at two
    // CTAs per SM an odd cluster leaves an SM shared with another cluster:
    // 13 splits 11.9 us).
    // A launch that may not overlap the kernel before it (no stable-cache
    // promise) starts on an idle GPU, where at batch 1 12 splits ran 8.2-8.9 us
    // against 10.3-10.9 us with 16; back to back, 16 stays faster (8.8 against
    // 9.8 us with 12).
    pl.one_wave = (pl.units * 4 <= slots && want_len <= 1) ? 1 : 0;
    if (pl.one_wave) {
      int s = kv_stable ? 16 : 12;
      while (s > 1 && (s * 4 > tiles || resident(pl, s) < pl.units)) s = s > 2 ? s - 2 : 1;
      pl.cluster = s;
      return pl;
    }
  }
  // the largest cluster not above S that can be scheduled at all
  while (S > 1 && resident(pl, S) <= 0) S >>= 1;
  pl.cluster = S;
  return pl;
}

int attn_max_active_clusters(int D, int mt, int wk, int S, int Hkv, int B, int kbr) {
#define X(DD, MM, WW) \
  if (D == DD && mt == MM && wk == WW) return max_cluster_t<DD, MM, WW>(S, Hkv, B, kbr);
  COSPEC_ATTN_VARIANTS(X)
#undef X
  return 0;
}

cudaError_t launch_verify_attn(const AttnArgs& a, const AttnPlan& pl, int* err,
                               cudaStream_t stream) {
  if (pl.kind == 1) return launch_verify_attn_tcq(a, pl, err, stream);
  // Pool as {64 columns, rows, half}: a {64, 16, H} box is one page of one
  // head, both 128-byte halves, landing as [half][16 rows][128 B].
  CUtensorMap maps[4];
  const int H = a.D / 64;
  const uint64_t pool_rows = (uint64_t)a.num_pages * a.Hkv * PAGE;
  const uint64_t dp[3] = {64, pool_rows, (uint64_t)H};
  const uint64_t sp[2] = {(uint64_t)a.D * 2, 128};
  const uint32_t bp[3] = {64, PAGE, (uint32_t)H};
  // Block K/V as {64 columns, batch*rows, half, head}: one box per (b, head).
  const uint64_t db[4] = {64, (uint64_t)a.B * a.R, (uint64_t)H, (uint64_t)a.Hkv};
  const uint64_t sb[3] = {(uint64_t)a.Hkv * a.D * 2, 128, (uint64_t)a.D * 2};
  const uint32_t bb[4] = {64, (uint32_t)((a.R + 15) & ~15), (uint32_t)H, 1};
  if (!encode_tensor_map_bf16(&maps[0], a.k_pages, 3, dp, sp, bp) ||
      !encode_tensor_map_bf16(&maps[1], a.v_pages, 3, dp, sp, bp) ||
      !encode_tensor_map_bf16(&maps[2], a.k_blk, 4, db, sb, bb) ||
      !encode_tensor_map_bf16(&maps[3], a.v_blk, 4, db, sb, bb))
    return cudaErrorInvalidValue;
  AttnParams p{};
  p.q = a.q;
  p.page_table = a.page_table;
  p.ctx_len = a.ctx_len;
  p.out = a.out;
  p.B = a.B;
  p.R = a.R;
  p.Hq = a.Hq;
  p.Hkv = a.Hkv;
  p.G = a.Hq / a.Hkv;
  p.NRT = p.G * a.R;
  p.RG = (p.NRT + 63) / 64;
  p.max_pages = a.max_pages;
  p.num_pages = a.num_pages;
  p.scale_log2 = a.scale * 1.4426950408889634f;
  p.kv_stable = a.kv_stable;
  p.block_full = a.block_full;
  p.err = err;
  const bool general = a.R > 32 || a.block_full;
  const bool wide = ((a.R + 15) & ~15) > 32;
#define X(DD, MM, WW)                                                                    \
  if (a.D == DD && pl.mt == MM && pl.wk == WW)                                           \
    return !general ? launch_t<DD, MM, WW, 0>(maps, p, pl.cluster, a.B, a.Hkv, stream)    \
           : (MM >= 4 && wide)                                                           \
               ? launch_t<DD, MM, WW, (MM >= 4 ? 2 : 1)>(maps, p, pl.cluster, a.B, a.Hkv, stream) \
               : launch_t<DD, MM, WW, 1>(maps, p, pl.cluster, a.B, a.Hkv, stream);
  COSPEC_ATTN_VARIANTS(X)
#undef X
  return cudaErrorInvalidValue;
}

}  // namespace cospec
