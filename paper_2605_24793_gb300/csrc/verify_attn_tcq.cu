// Verify attention on the tcgen05 tensor cores with the query rows as the
// MMA M dimension (teacher-forced verification pass, Sec. 3.1 Eq. 2 of the
// paper): the K+1 block rows of every query head of a KV group attend to the
// paged bf16 cache and, causally (or fully, for the arbitrator's region), to
// the block.
//
// One CTA owns (sequence b, KV head, KV split, row group of <= 128 query
// rows); the splits of a (b, head, row group) form a thread-block cluster and
// merge their partial softmax states through distributed shared memory.  A
// KV head's G query heads times the block rows (up to 128 rows: K <= 31 at
// G = 4, K <= 15 at G = 8) share one CTA, so its cache streams once.  Roles
// by warp:
//   warps 0-2  TMA producers: 128-key K/V tiles (one 2-D box per page and
//              128-byte half: [half][128 keys][128 B], 128B-swizzled) into a
//              3-stage ring, the block's own K/V as a final tile;
//   warp 3     MMA issuer (one thread), which first loads the query rows of
//              the group:
//                S  = Q K^T   (M = 128 query rows, N = 128 keys, K = D) into
//                             one of three TMEM score buffers,
//                O += P V     (M = 128 query rows, N = D, K = keys) with P
//                             read from TMEM (written over its score
//                             buffer; three buffers, so S may run two
//                             tiles ahead of P.V) and V read MN-major from
//                             the V tile;
//   warps 4-11 softmax, two groups of four warps (one per TMEM lane quarter)
//              sharing every tile, group g its key columns 64 g .. 64 g + 63:
//              a thread owns one query row and half of its scores; the two
//              threads of a row swap their half maxima through shared memory,
//              turn their scores into bf16 P in place and rescale their half
//              of the row of O when the row's reference maximum moves.
// Softmax with a lazy reference maximum per row: scores are taken relative
// to m_ref, set exactly by the first tile; a later tile moves m_ref (and
// rescales O and l) only when one of its scores exceeds m_ref by more than
// 2^8 in the exp2 domain, so P stays below 256 and rescales are rare.
#include <cuda.h>
#include <math.h>

#include "cospec_device.cuh"
#include "cospec_internal.h"

namespace cospec {

namespace {

constexpr int QKT = 128;          // keys per cache tile (8 pages) = MMA N of S
constexpr int QPPT = QKT / 16;    // pages per tile
constexpr int QPAGE = 16;         // page size (fixed)
constexpr int QROWB = 128;        // bytes of one swizzled smem row
constexpr int QM = 128;           // query rows per CTA = MMA M
constexpr int Q_PROD = 3;         // producer warps
constexpr int Q_MMA_WARP = 3;     // MMA issuer warp
constexpr int Q_SOFT0 = 4;        // first softmax warp (group 0, lane quarter 0)
constexpr int Q_THREADS = 384;   // producers, MMA warp, two groups of four softmax warps
constexpr float Q_LAZY = 8.f;     // move m_ref only when a score exceeds it by this (log2)
constexpr uint64_t Q_WAIT_NS = 2000000000ull;

struct TcqParams {
  const int32_t* page_table;
  const int32_t* ctx_len;
  const __nv_bfloat16* q;  // only for the L2 warm-up of the query rows
  __nv_bfloat16* out;
  int B, R, Hq, Hkv, G;
  int JB;          // block rows (j) per row group
  int JBQ;         // block rows covered by the query box: min(R, JB)
  int RG;          // row groups
  int max_pages, num_pages;
  float scale_log2;
  int kv_stable;
  int block_full;  // block rows see every block row (not only rows <= their own)
  int* err;
};

template <int D>
struct TcqLayout {
  static constexpr int H = D / 64;                  // 128-byte halves of a key row
  static constexpr int KVB = H * QKT * QROWB;       // K (or V) of a tile: [half][128 keys][128 B]
  static constexpr int STAGE = 2 * KVB;             // K then V
  static constexpr int NS = 3;                      // 192 KB (D = 128) / 96 KB ring
  static constexpr int RING = NS * STAGE;
  static constexpr int QH = QM * QROWB;             // one half of the query rows
  static constexpr int QOFF = RING;
  static constexpr int MISC = QOFF + H * QH;
  // barriers: full_k[NS], full_v[NS], empty_k[NS], empty_v[NS], q_full, s_full[NSB],
  // p_full[NSB], pv_done, mma_done, recv_bar
  static constexpr int NSB = 3;                     // TMEM score buffers
  static constexpr int NBAR = 4 * NS + 2 * NSB + 4;
  static constexpr int HOLDER = MISC + NBAR * 8;    // TMEM base address
  static constexpr int FLAGS = HOLDER + 16;         // abort, tiles issued [2], sequence slot, row-pair votes [8]
  static constexpr int XCH = FLAGS + 64;            // float [2][QM]: the groups' row maxima / sums
  static constexpr int TOTAL = XCH + 2 * QM * 4;
  // partial rows after the last tile, in the idle ring: PART [QM], RECV [QM + 15]
  static constexpr int PD = D + 4;                  // O[D], m, l, pad: conflict-free row stores
  static constexpr int ROWP = PD * 4;
  static constexpr int PART = 0;
  static constexpr int RECV = QM * ROWP;
  static_assert(RECV + (QM + 15) * ROWP <= RING, "partials must fit in the ring");
  static_assert(ROWP % 16 == 0, "bulk copies move whole 16-byte chunks");
  // TMEM columns: score buffers at 0, 128 and 256, O at 384
  static constexpr uint32_t TCOLS = 512u;
  static constexpr uint32_t OCOL = NSB * QKT;
  static_assert(OCOL + D <= TCOLS, "the O accumulator after the score buffers");
};

// 32 lanes x 32 bit, 16 consecutive columns per thread (no wait).
CS_DEV void tq_ld16(uint32_t taddr, float* v) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,"
      "%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}
CS_DEV void tq_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
CS_DEV void tq_st16(uint32_t taddr, const uint32_t* v) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,"
      "%14,%15,%16};" ::"r"(taddr),
      "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]),
      "r"(v[8]), "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]),
      "r"(v[15])
      : "memory");
}
CS_DEV void tq_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

// D[tmem] (+)= A[tmem] * B[smem desc], bf16 inputs, fp32 accumulate.  A is
// M x 16 with row m in TMEM lane m and two bf16 per 32-bit column.
CS_DEV void umma_bf16_tmem_a(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                             uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n}\n" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Descriptor of an MN-major operand in the 128B-swizzle layout: 64-element
// rows of 128 bytes along MN, consecutive rows = consecutive K; `lbo` bytes
// between the 64-element groups along MN, 1024 bytes between 8-row groups
// along K.
CS_DEV uint64_t tq_desc_mn_sw128(uint32_t saddr, uint32_t lbo) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFF) >> 4);
  d |= (uint64_t)((lbo >> 4) & 0x3FFF) << 16;
  d |= (uint64_t)(1024 >> 4) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
}


template <int D>
__global__ void __launch_bounds__(Q_THREADS, 1)
    verify_attn_tcq_kernel(const __grid_constant__ CUtensorMap map_kp,
                           const __grid_constant__ CUtensorMap map_vp,
                           const __grid_constant__ CUtensorMap map_kb,
                           const __grid_constant__ CUtensorMap map_vb,
                           const __grid_constant__ CUtensorMap map_q, const TcqParams p) {
  using LY = TcqLayout<D>;
  constexpr int H = LY::H;
  constexpr int NS = LY::NS;
  constexpr int PD = LY::PD;

  extern __shared__ __align__(16) uint8_t smem_raw[];
  // 1024-byte aligned base (TMA 128B swizzle, UMMA descriptors), kept as an
  // offset from the shared array so that accesses stay shared-memory ones.
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  // A stage's K and V halves fill and free separately: K is dead once its
  // score product completes, well before P.V frees V, so K refills early.
  uint64_t* full_k = reinterpret_cast<uint64_t*>(smem + LY::MISC);
  uint64_t* full_v = full_k + NS;
  uint64_t* empty_k = full_v + NS;
  uint64_t* empty_v = empty_k + NS;
  uint64_t* q_full = empty_v + NS;
  uint64_t* s_full = q_full + 1;      // [NSB]
  uint64_t* p_full = s_full + LY::NSB;  // [NSB]
  uint64_t* pv_done = p_full + LY::NSB;
  uint64_t* mma_done = pv_done + 1;
  uint64_t* recv_bar = mma_done + 1;  // partials received from the cluster
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(smem + LY::HOLDER);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + LY::FLAGS);
  volatile int* n_issued = abort_flag + 1;   // [2]: tiles whose K / V loads were issued (abort tail)
  volatile int* seq_slot = abort_flag + 3;
  volatile int* xvote = abort_flag + 4;      // [2 groups][4 quarters]: this tile's waits succeeded
  uint8_t* qs = smem + LY::QOFF;

  const int S = (int)cluster_nctarank();
  const int rank = (int)cluster_ctarank();
  const int kvh = blockIdx.y / p.RG, rg = blockIdx.y % p.RG;
  const int j0 = rg * p.JB;                          // first block row of this group
  const int nj = min(p.JB, p.R - j0);
  const int NR = nj * p.G;                           // query rows of this group (<= QM)
  const int qrows = p.G * p.JBQ;                     // rows the query box writes
  const int nsw = (NR + 31) >> 5;                    // softmax warps that own rows
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  if (tid == 0) {
    for (int s = 0; s < NS; ++s) {
      mbar_init(&full_k[s], 2);            // the two K producer warps
      mbar_init(&full_v[s], 1);            // the V producer warp
      mbar_init(&empty_k[s], 1);
      mbar_init(&empty_v[s], 1);
    }
    mbar_init(q_full, 1);
    for (int i = 0; i < LY::NSB; ++i) {
      mbar_init(&s_full[i], 1);
      mbar_init(&p_full[i], (uint32_t)(2 * nsw));   // both softmax groups' warps with rows
    }
    mbar_init(pv_done, 1);
    mbar_init(mma_done, 1);
    mbar_init(recv_bar, 1);
    abort_flag[0] = 0;
    abort_flag[1] = 0;
    abort_flag[2] = 0;
    fence_barrier_init();
  }
  if (warp == Q_MMA_WARP) {
    tmem_alloc(tmem_holder, LY::TCOLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_holder;
  // Let the next kernel of the stream start launching; with the stable-cache
  // promise its CTAs stream their cache tiles while this one computes.
  griddep_launch_dependents();
  if (!p.kv_stable) griddep_wait();

  // Sequences are taken longest context first (blockIdx.z = rank, ties by
  // index), so that the long ones start early and the short ones fill in
  // behind them at the end of the launch.
  const int b = (p.B > 1 && p.B <= RANK_MAX_B) ? sequence_by_rank(p.ctx_len, p.B, (int)blockIdx.z, seq_slot)
                        : (int)blockIdx.z;
  const int C = p.ctx_len[b];
  const bool bad = (C < 0) || (C > p.max_pages * QPAGE);
  if (bad && rank == 0 && kvh == 0 && rg == 0 && tid == 0) set_err(p.err, ERR_CTX);
  const int nct = bad ? 0 : (C + QKT - 1) / QKT;
  const int tps = (nct + S - 1) / S;
  const int t_begin = min(nct, rank * tps);
  const int n = min(nct, t_begin + tps) - t_begin;   // cache tiles of this CTA
  const bool do_blk = !bad && rank == S - 1;         // the block's keys: last CTA
  const int T = n + (do_blk ? 1 : 0);
  const int npages = (C + QPAGE - 1) / QPAGE;
  const int KBR = (p.R + 15) & ~15;                  // block keys padded to 16
  float mref = -INFINITY, l = 0.f;                   // softmax threads: this row's m_ref and sum

  if (warp < Q_PROD) {
    // ------------------------------------------------------------ producers
    // A warp's bulk copies are processed one after another, which holds one
    // warp to about 45 GB/s of 2 KB boxes: warps 0 and 1 split each tile's K
    // boxes, warp 2 issues its V boxes (needed later, at P.V).
    const int pw = warp;
    const int tensor = pw == 2 ? 1 : 0;                 // 0: K, 1: V
    constexpr int NKB = H * QPPT;                       // boxes of a tensor's tile: page x half
    const int kb0 = tensor ? 0 : pw * (NKB / 2);        // this warp's first box
    const int nkb = tensor ? NKB : NKB / 2;             // and its boxes per tile
    const int e = kb0 + lane;                           // this lane's box
    const bool mine = lane < nkb;
    uint64_t* my_full = tensor ? full_v : full_k;
    uint64_t* my_empty = tensor ? empty_v : empty_k;
    if (pw == 0 && lane == 0) {
      tma_prefetch_desc(&map_kp);
      tma_prefetch_desc(&map_vp);
      tma_prefetch_desc(&map_q);
    }
    const uint64_t pol = p.RG > 1 ? l2_policy_evict_normal() : l2_policy_evict_first();
    const int* ptab = p.page_table + (size_t)b * p.max_pages + (size_t)t_begin * QPPT;
    const int my_pages = min(n * QPPT, npages - t_begin * QPPT);
    int pid = 0;
    bool ok = true;
    int issued = 0;                      // tiles whose loads were issued
    auto issue_cache = [&](int t) {
      const int st = t % NS;
      uint8_t* sb = smem + st * LY::STAGE;
      if ((t & 3) == 0) {                // 32 page ids = the next 4 tiles, one per lane
        const int e2 = t * QPPT + lane;
        pid = (e2 < my_pages) ? __ldg(ptab + e2) : 0;
      }
      const int np = min(QPPT, npages - (t_begin + t) * QPPT);
      // box e of a tensor: page e / H, half e % H
      const int pg = e / H;
      int pgid = __shfl_sync(0xffffffffu, pid, (t & 3) * QPPT + (pg & 7));
      if (lane == 0) {
        // this warp's boxes within the tile's np pages
        const int hi = min(kb0 + nkb, np * H);
        mbar_arrive_expect_tx(&my_full[st], (uint32_t)(max(0, hi - kb0) * QPAGE * QROWB));
      }
      __syncwarp();
      if (mine && pg < np) {
        if ((unsigned)pgid >= (unsigned)p.num_pages) {
          set_err(p.err, ERR_PAGE);
          pgid = 0;
        }
        const int h = e % H;
        tma_load_3d(smem_u32(sb + tensor * LY::KVB + h * (QKT * QROWB) + pg * (QPAGE * QROWB)),
                    tensor ? (const void*)&map_vp : (const void*)&map_kp, &my_full[st], 0,
                    (pgid * p.Hkv + kvh) * QPAGE, h, pol);
      }
      __syncwarp();
    };
    auto wait_slot = [&](int t) -> bool {
      if (t < NS) return true;
      const int st = t % NS;
      const bool w = mbar_wait(&my_empty[st], (uint32_t)((t / NS) - 1) & 1u, Q_WAIT_NS);
      return __all_sync(0xffffffffu, w) && !*abort_flag;
    };
    const int pre = min(n, NS);
    for (int t = 0; t < pre; ++t) {      // with the stable-cache promise: before the wait
      issue_cache(t);
      ++issued;
    }
    if (pw == 0 && pre == NS && n > NS) {
      // The ring is full: pull the next tile's pages into L2.
      const int e2 = NS * QPPT + (lane >> 1);
      const int pg = __shfl_sync(0xffffffffu, pid, e2 & 31);
      if (lane < 2 * QPPT && e2 < my_pages && (unsigned)pg < (unsigned)p.num_pages)
        for (int h = 0; h < H; ++h)
          tma_prefetch_l2_3d((lane & 1) ? (const void*)&map_vp : (const void*)&map_kp, 0,
                             (pg * p.Hkv + kvh) * QPAGE, h);
    }
    // the block K/V comes from the previous kernel; the other producers
    // read only the (stable) cache
    if (p.kv_stable && pw == 0) griddep_wait();
    for (int t = pre; t < n && ok; ++t) {
      if (!wait_slot(t)) {
        ok = false;
        break;
      }
      issue_cache(t);
      ++issued;
    }
    if (ok && do_blk) {
      const int t = n;
      if (wait_slot(t)) {
        const int st = t % NS;
        uint8_t* sb = smem + st * LY::STAGE;
        // one box per tensor: KBR rows from block row 0 of this head, all
        // halves, landing as [half][KBR rows][128 B]
        if (pw == 0 && lane == 0) {
          mbar_arrive_expect_tx(&full_k[st], (uint32_t)(H * KBR * QROWB));
          tma_load_4d(smem_u32(sb), &map_kb, &full_k[st], 0, b * p.R, 0, kvh, pol);
        } else if (pw == 1 && lane == 0) {
          mbar_arrive(&full_k[st]);
        } else if (pw == 2 && lane == 0) {
          mbar_arrive_expect_tx(&full_v[st], (uint32_t)(H * KBR * QROWB));
          tma_load_4d(smem_u32(sb + LY::KVB), &map_vb, &full_v[st], 0, b * p.R, 0, kvh, pol);
        }
        ++issued;
      } else {
        ok = false;
      }
    }
    if (!ok && lane == 0) {
      set_err(p.err, ERR_TIMEOUT);
      *abort_flag = 1;
    }
    if (pw != 1 && lane == 0) n_issued[tensor] = issued;
  } else if (warp == Q_MMA_WARP) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0 && T > 0) {
      const uint32_t idesc_pv = idesc_bf16_f32(QM, D) | (1u << 16);   // B (V) MN-major
      const uint32_t q0 = smem_u32(qs);
      {
        // The query rows come from the previous kernel: this thread loads
        // them as soon as that kernel is done, while the producer warps are
        // still issuing the first cache tiles (a warp's bulk copies run one
        // after another; behind three tiles' boxes the rows landed ~2 us
        // later at batch 1).
        if (p.kv_stable) griddep_wait();
        const uint64_t qpol = p.RG > 1 ? l2_policy_evict_normal() : l2_policy_evict_first();
        mbar_arrive_expect_tx(q_full, (uint32_t)(H * qrows * QROWB));
        for (int h = 0; h < H; ++h)
          tma_load_4d(smem_u32(qs + h * LY::QH), &map_q, q_full, 0, kvh * p.G, b * p.R + j0, h, qpol);
      }
      bool ok = mbar_wait(q_full, 0, Q_WAIT_NS);
      auto issue_s = [&](int t) {
        const int st = t % NS;
        const uint32_t kb = smem_u32(smem + st * LY::STAGE);
        const bool blk = do_blk && t == n;
        const int nk = blk ? KBR : QKT;
        const uint32_t khalf = (uint32_t)(nk * QROWB);
        const uint32_t idesc_qk = idesc_bf16_f32(QM, nk);
#pragma unroll
        for (int h = 0; h < H; ++h)
#pragma unroll
          for (int ks = 0; ks < 4; ++ks)
            umma_bf16(tmem_base + (uint32_t)((t % LY::NSB) * QKT), smem_desc_sw128(q0 + h * LY::QH + ks * 32),
                      smem_desc_sw128(kb + h * khalf + ks * 32), idesc_qk, (h | ks) != 0 ? 1u : 0u);
        umma_commit(&empty_k[st]);         // K of this stage is free once S is done
        umma_commit(&s_full[t % LY::NSB]);
      };
      auto issue_pv = [&](int u) {
        const int st = u % NS;
        const uint32_t vb = smem_u32(smem + st * LY::STAGE + LY::KVB);
        const bool blk = do_blk && u == n;
        const int nk = blk ? KBR : QKT;
        const uint32_t vhalf = (uint32_t)(nk * QROWB);
        // P of tile u: 16 keys = 8 TMEM columns per step
        for (int ks = 0; ks < nk / 16; ++ks)
          umma_bf16_tmem_a(tmem_base + LY::OCOL,
                           tmem_base + (uint32_t)((u % LY::NSB) * QKT + ks * 8),
                           tq_desc_mn_sw128(vb + ks * 2048, vhalf), idesc_pv,
                           (u > 0 || ks > 0) ? 1u : 0u);
        umma_commit(&empty_v[st]);
        umma_commit(pv_done);
      };
      // Issue whichever product is ready, so that a P.V product (which frees
      // a ring stage for the producer) never waits behind the next tile's
      // load.  S of tile ts goes to buffer ts % 3, last read (as P) by the
      // P.V product of tile ts - 3: tcgen05 MMAs of one thread run in issue
      // order, so S may be issued once that product is.  At most two tiles'
      // S run ahead of the oldest pending P.V, which also keeps every
      // barrier within one phase of the parity tested here.
      int ts = 0, tp = 0, idle = 0;
      uint64_t t_last = global_timer_ns();
      while (ok && tp < T) {
        bool did = false;
        if (tp < ts && mbar_test(&p_full[tp % LY::NSB], (uint32_t)(tp / LY::NSB) & 1u) &&
            mbar_test(&full_v[tp % NS], (uint32_t)(tp / NS) & 1u)) {
          tc_fence_after();
          issue_pv(tp);
          ++tp;
          did = true;
        }
        if (ts < T && ts <= tp + 2 && mbar_test(&full_k[ts % NS], (uint32_t)(ts / NS) & 1u)) {
          tc_fence_after();
          issue_s(ts);
          ++ts;
          did = true;
        }
        // the clock is read only every 256 idle polls (the limit stays bounded)
        if (did) {
          idle = 0;
        } else if ((++idle & 255) == 0) {
          const uint64_t now = global_timer_ns();
          if (idle == 256) t_last = now;
          else if (*abort_flag || now - t_last > Q_WAIT_NS) ok = false;
        }
      }
      if (!ok) {
        set_err(p.err, ERR_TIMEOUT);
        *abort_flag = 1;
      }
      // every MMA issued by this thread completes before TMEM is released
      umma_commit(mma_done);
      mbar_wait(mma_done, 0, Q_WAIT_NS);
    }
  } else {
    // ------------------------------------------------------------ softmax
    // Two groups of four warps (one warp per TMEM lane quarter each) share
    // every tile: group g takes its key columns 64 g .. 64 g + 63.  A thread
    // owns one query row; the two threads of a row (same lane, warps q and
    // q + 4) swap their half-tile maxima through shared memory, so both move
    // the row's reference maximum together and their P, written over their
    // own columns of the score buffer, share one O accumulator.
    const int sw = warp - Q_SOFT0;
    const int grp = sw >> 2;             // key-column half of every tile
    const int q = sw & 3;                // TMEM lane quarter of this warp
    const int r = q * 32 + lane;         // this thread's query row
    const int gtid = q * 32 + lane;      // thread index within the group
    const int kc0 = grp * (QKT / 2);     // first key column of this half
    float* xch = reinterpret_cast<float*>(smem + LY::XCH);   // [2][QM]
    if (p.kv_stable) {
      // warm L2 with the group's query rows before the producer's TMA
      for (int e = sw * 32 + lane; e < NR * (D * 2 / 128); e += 256) {
        const int rr = e / (D * 2 / 128), part_ = e % (D * 2 / 128);
        const int j = j0 + rr / p.G, g = rr % p.G;
        prefetch_l2(p.q + (((size_t)b * p.R + j) * p.Hq + (size_t)kvh * p.G + g) * D + part_ * 64);
      }
    }
    const bool rvalid = r < NR;
    const int jr = j0 + (rvalid ? r / p.G : 0);      // block row of this query row
    // the last block key this row sees: its own row (causal) or the whole block
    const int blim = p.block_full ? p.R - 1 : min(jr, p.R - 1);
    const float sc = p.scale_log2;
    const uint32_t lane_base = tmem_base + ((uint32_t)(q * 32) << 16);
    const uint32_t ocol = LY::OCOL + (uint32_t)(grp * (D / 2));   // this group's half of O
    constexpr int HK = QKT / 2;          // key columns of a half
    if (q < nsw) {
      for (int t = 0; t < T; ++t) {
        const int sb_i = t % LY::NSB;
        const int st = t % NS;
        uint8_t* sb = smem + st * LY::STAGE;
        const bool blk = do_blk && t == n;
        const int nk = blk ? KBR : QKT;          // score columns of this tile
        // The two warps of a row pair decide an abort together (from both
        // votes, read after the first exchange barrier), so neither is left
        // waiting at a barrier the other no longer reaches.
        const bool okw =
            __all_sync(0xffffffffu, mbar_wait(&s_full[sb_i], (uint32_t)(t / LY::NSB) & 1u, Q_WAIT_NS)) &&
            !*abort_flag;
        if (lane == 0) xvote[grp * 4 + q] = okw ? 1 : 0;
        tc_fence_after();
        const uint32_t srow = lane_base + (uint32_t)(sb_i * QKT);
        // keys 0..lim of this tile are visible to this row (raw scores; the
        // scale is positive, so it is applied with the exponent).  Padding
        // rows (r >= NR) give rows of P and O that nothing reads, so they
        // decide neither the masking nor a rescale.
        const int lim = blk ? blim : min(QKT, C - (t_begin + t) * QKT) - 1;
        float x[HK];
#pragma unroll
        for (int c = 0; c < HK / 16; ++c) {
          if (okw && kc0 + c * 16 < nk) {
            tq_ld16(srow + kc0 + c * 16, &x[c * 16]);
          } else {
#pragma unroll
            for (int k = 0; k < 16; ++k) x[c * 16 + k] = -INFINITY;
          }
        }
        tq_wait_ld();
        if (__any_sync(0xffffffffu, rvalid && lim < kc0 + HK - 1)) {
#pragma unroll
          for (int k = 0; k < HK; ++k) x[k] = (kc0 + k <= lim) ? x[k] : -INFINITY;
        }
        float m4[4] = {x[0], x[1], x[2], x[3]};
#pragma unroll
        for (int k = 4; k < HK; ++k) m4[k & 3] = fmaxf(m4[k & 3], x[k]);
        const float mh = fmaxf(fmaxf(m4[0], m4[1]), fmaxf(m4[2], m4[3]));
        // the row's maximum over both halves (both threads have read their
        // scores by the first barrier, so P may then overwrite them; the
        // second barrier lets the buffer be rewritten at the next tile)
        xch[grp * QM + r] = mh;
        named_bar_sync(1 + q, 64);
        const float mx = fmaxf(mh, xch[(grp ^ 1) * QM + r]) * sc;
        const bool ok2 = xvote[q] != 0 && xvote[4 + q] != 0;
        named_bar_sync(1 + q, 64);
        if (!ok2) {
          if (lane == 0) {
            set_err(p.err, ERR_TIMEOUT);
            *abort_flag = 1;
          }
          break;
        }
        // move the reference only when a score exceeds it by 2^8 (the first
        // tile always sets it: m_ref starts at -inf)
        const bool up = rvalid && mx > mref + Q_LAZY;
        float alpha = 1.f;
        if (up) {
          alpha = (mref == -INFINITY) ? 0.f : exp2_approx(mref - mx);
          mref = mx;
          l *= alpha;
        }
        if (__any_sync(0xffffffffu, up && t > 0)) {
          // O holds tiles 0..t-1: wait for the last of them, then scale this
          // group's half of the row
          const bool okp =
              __all_sync(0xffffffffu, mbar_wait(pv_done, (uint32_t)(t - 1) & 1u, Q_WAIT_NS));
          tc_fence_after();
          if (okp) {
#pragma unroll 1
            for (int c = 0; c < D / 32; ++c) {
              float o[16];
              tq_ld16(lane_base + ocol + c * 16, o);
              tq_wait_ld();
              uint32_t w[16];
#pragma unroll
              for (int k = 0; k < 16; ++k) w[k] = __float_as_uint(o[k] * alpha);
              tq_st16(lane_base + ocol + c * 16, w);
            }
          } else if (lane == 0) {
            set_err(p.err, ERR_TIMEOUT);
          }
        }
        // P = 2^(score * scale - m_ref) in bf16, two keys per TMEM column, in
        // this half's columns of the score buffer (masked keys give exactly 0)
        const float nb = (mref == -INFINITY) ? 0.f : -mref;
        float l4[4] = {0.f, 0.f, 0.f, 0.f};
        uint32_t pk[HK / 2];
#pragma unroll
        for (int k = 0; k < HK / 2; ++k) {
          const float p0 = exp2_approx(fmaf(x[2 * k], sc, nb));
          const float p1 = exp2_approx(fmaf(x[2 * k + 1], sc, nb));
          l4[k & 3] += p0 + p1;
          pk[k] = pack_bf16(p0, p1);
        }
        l += (l4[0] + l4[1]) + (l4[2] + l4[3]);
#pragma unroll
        for (int c = 0; c < HK / 32; ++c)
          if (kc0 + c * 32 < nk) tq_st16(srow + kc0 / 2 + c * 16, &pk[c * 16]);
        // V rows of keys outside the context (or past the block) may hold
        // stale bytes: group 0 zeroes them so that their zero weights
        // contribute 0 (V lands separately from K: wait for it first).
        if (grp == 0) {
          const int vr = blk ? p.R : min(QKT, C - (t_begin + t) * QKT);
          if (vr < nk &&
              __all_sync(0xffffffffu, mbar_wait(&full_v[st], (uint32_t)(t / NS) & 1u, Q_WAIT_NS))) {
            uint8_t* vb = sb + LY::KVB;
            const int vhalf = nk * QROWB;
            for (int e = gtid; e < (nk - vr) * H * 8; e += nsw * 32) {
              const int row = vr + e / (H * 8), rem = e % (H * 8);
              *reinterpret_cast<uint4*>(vb + (rem / 8) * vhalf + row * QROWB + (rem % 8) * 16) =
                  make_uint4(0u, 0u, 0u, 0u);
            }
            fence_proxy_async_smem();
          }
        }
        tq_wait_st();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&p_full[sb_i]);
      }
      if (T > 0 && !*abort_flag) {
        const bool okp =
            __all_sync(0xffffffffu, mbar_wait(pv_done, (uint32_t)(T - 1) & 1u, Q_WAIT_NS));
        if (!okp && lane == 0) {
          set_err(p.err, ERR_TIMEOUT);
          *abort_flag = 1;
        }
      }
      tc_fence_after();
    }
    // the row's sum over both halves (the exchange buffer is free: every
    // tile's second barrier has passed)
    if (q < nsw) {
      xch[grp * QM + r] = l;
      named_bar_sync(1 + q, 64);
      l += xch[(grp ^ 1) * QM + r];
    }
  }
  __syncthreads();
  tc_fence_after();

  // ---------------------------------------------------------------- output
  // The ring is idle from here on.  Unsplit, every softmax thread writes its
  // normalised row; split, it writes its partial row (O, m_ref, l) and the
  // cluster's CTAs reduce-scatter them (owner o finishes rows
  // [o * rpo, (o + 1) * rpo)).
  const bool have = T > 0 && !*abort_flag;
  const int rpo = (NR + S - 1) / S;
  if (S > 1) {
    if (tid == 0) mbar_arrive_expect_tx(recv_bar, (uint32_t)(S * rpo * LY::ROWP));
    cluster_arrive_relaxed();
  }
  float* part = reinterpret_cast<float*>(smem + LY::PART);
  if (warp >= Q_SOFT0 && ((warp - Q_SOFT0) & 3) < nsw) {
    // each group writes its half of the row's columns (both hold m_ref and l)
    const int sw = warp - Q_SOFT0, grp = sw >> 2, q = sw & 3, r = q * 32 + lane;
    const bool rvalid = r < NR;
    const int c0 = grp * (D / 32);       // first 16-column chunk of this group's half
    const uint32_t orow = tmem_base + ((uint32_t)(q * 32) << 16) + LY::OCOL;
    auto load_o = [&](int c, float (&o)[16]) {
      if (have) {
        tq_ld16(orow + c * 16, o);
        tq_wait_ld();
      } else {
#pragma unroll
        for (int i = 0; i < 16; ++i) o[i] = 0.f;
      }
    };
    if (S == 1) {
      const int j = j0 + (rvalid ? r / p.G : 0), g = rvalid ? r % p.G : 0;
      __nv_bfloat16* dst = p.out + (((size_t)b * p.R + j) * p.Hq + (size_t)kvh * p.G + g) * D;
      const float inv = (have && l > 0.f) ? 1.f / l : 0.f;
#pragma unroll 1
      for (int c = c0; c < c0 + D / 32; ++c) {
        float o[16];
        load_o(c, o);
        if (rvalid) {
          uint4 w0, w1;
          w0.x = pack_bf16(o[0] * inv, o[1] * inv);
          w0.y = pack_bf16(o[2] * inv, o[3] * inv);
          w0.z = pack_bf16(o[4] * inv, o[5] * inv);
          w0.w = pack_bf16(o[6] * inv, o[7] * inv);
          w1.x = pack_bf16(o[8] * inv, o[9] * inv);
          w1.y = pack_bf16(o[10] * inv, o[11] * inv);
          w1.z = pack_bf16(o[12] * inv, o[13] * inv);
          w1.w = pack_bf16(o[14] * inv, o[15] * inv);
          *reinterpret_cast<uint4*>(dst + c * 16) = w0;
          *reinterpret_cast<uint4*>(dst + c * 16 + 8) = w1;
        }
      }
    } else {
      float* prow = part + r * PD;
#pragma unroll 1
      for (int c = c0; c < c0 + D / 32; ++c) {
        float o[16];
        load_o(c, o);
        if (rvalid) {
#pragma unroll
          for (int i = 0; i < 16; i += 4)
            *reinterpret_cast<float4*>(prow + c * 16 + i) = make_float4(o[i], o[i + 1], o[i + 2], o[i + 3]);
        }
      }
      if (rvalid && grp == 0) {
        prow[D] = have ? mref : -INFINITY;
        prow[D + 1] = have ? l : 0.f;
      }
    }
  }
  if (S > 1) {
    fence_proxy_async_smem();            // the bulk copies below read `part`
    __syncthreads();
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
    cluster_arrive_relaxed();            // everything addressed to this CTA has landed
    const int row0 = rank * rpo;
    // Per owned row: one warp forms the common maximum over the S partials
    // and each partial's weight exp2(m_s - M) / L (kept where the query rows
    // were); then every output chunk is a plain weighted sum.
    float* scl = reinterpret_cast<float*>(qs);               // [S][rpo]
    for (int rr = warp; rr < rpo; rr += Q_THREADS / 32) {
      if (row0 + rr >= NR) break;
      const float2 ml = (lane < S) ? *reinterpret_cast<const float2*>(recv + (lane * rpo + rr) * PD + D)
                                   : make_float2(-INFINITY, 0.f);
      float M = ml.x;
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, off));
      const float w = (M == -INFINITY || ml.x == -INFINITY) ? 0.f : exp2_approx(ml.x - M);
      float L = ml.y * w;
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) L += __shfl_xor_sync(0xffffffffu, L, off);
      if (lane < S) scl[lane * rpo + rr] = (L > 0.f) ? w / L : 0.f;
    }
    __syncthreads();
    for (int e = tid; e < rpo * (D / 4); e += Q_THREADS) {
      const int rr = e / (D / 4), c = (e % (D / 4)) * 4;
      const int r = row0 + rr;
      if (r >= NR) break;
      float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 4
      for (int s2 = 0; s2 < S; ++s2) {
        const float w = scl[s2 * rpo + rr];
        const float4 v = *reinterpret_cast<const float4*>(recv + (s2 * rpo + rr) * PD + c);
        acc.x += v.x * w;
        acc.y += v.y * w;
        acc.z += v.z * w;
        acc.w += v.w * w;
      }
      const int j = j0 + r / p.G, g = r % p.G;
      __nv_bfloat16* dst = p.out + (((size_t)b * p.R + j) * p.Hq + (size_t)kvh * p.G + g) * D + c;
      uint2 pk;
      pk.x = pack_bf16(acc.x, acc.y);
      pk.y = pack_bf16(acc.z, acc.w);
      *reinterpret_cast<uint2*>(dst) = pk;
    }
    cluster_wait();                      // every copy out of this CTA has landed
  }

  // After an abort a copy may still be in flight: wait (bounded) for the
  // last fill of every stage the producer used before shared memory goes.
  if (*abort_flag && tid == 0) {
    for (int tn = 0; tn < 2; ++tn) {
      const int ni = n_issued[tn];
      uint64_t* f = tn ? full_v : full_k;
      for (int st = 0; st < NS && st < ni; ++st) {
        const int last = st + ((ni - 1 - st) / NS) * NS;
        mbar_wait(&f[st], (uint32_t)(last / NS) & 1u, Q_WAIT_NS);
      }
    }
    if (T > 0) mbar_wait(q_full, 0, Q_WAIT_NS);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == Q_MMA_WARP) {
    __syncwarp();
    tmem_dealloc(tmem_base, LY::TCOLS);
  }
}

template <int D>
size_t tcq_smem_bytes() {
  return (size_t)TcqLayout<D>::TOTAL + 1024;
}

// Limits already set on each instantiation of the kernel.
template <int D>
KernelLimits& tcq_limits() {
  static KernelLimits lim;
  return lim;
}

template <int D>
cudaError_t launch_tcq_t(const CUtensorMap* maps, const TcqParams& p, int S, int B, int Hkv, int RG,
                         cudaStream_t stream) {
  const size_t smem = tcq_smem_bytes<D>();
  auto kern = verify_attn_tcq_kernel<D>;
  const cudaError_t e = ensure_kernel_limits((const void*)kern, tcq_limits<D>(), smem, true);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(S, Hkv * RG, B);
  cfg.blockDim = dim3(Q_THREADS, 1, 1);
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
  return cudaLaunchKernelEx(&cfg, kern, maps[0], maps[1], maps[2], maps[3], maps[4], p);
}

template <int D>
int max_cluster_tcq_t(int S, int Hkv, int B, int RG) {
  const size_t smem = tcq_smem_bytes<D>();
  auto kern = verify_attn_tcq_kernel<D>;
  if (ensure_kernel_limits((const void*)kern, tcq_limits<D>(), smem, true) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(S, Hkv * RG, B);
  cfg.blockDim = dim3(Q_THREADS, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = S;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int nclu = 0;
  if (cudaOccupancyMaxActiveClusters(&nclu, kern, &cfg) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return nclu;
}

}  // namespace

bool tcq_attn_supported(int D, int G) { return (D == 64 || D == 128) && G >= 1 && G <= QM; }

int attn_tcq_max_active_clusters(int D, int S, int Hkv, int B, int RG) {
  if (D == 128) return max_cluster_tcq_t<128>(S, Hkv, B, RG);
  if (D == 64) return max_cluster_tcq_t<64>(S, Hkv, B, RG);
  return 0;
}

cudaError_t launch_verify_attn_tcq(const AttnArgs& a, const AttnPlan& pl, int* err,
                                   cudaStream_t stream) {
  const int H = a.D / 64;
  const int G = a.Hq / a.Hkv;
  if (G * pl.jbq > QM || pl.jb * G > QM) return cudaErrorInvalidValue;
  CUtensorMap maps[5];
  // Pool as {64 columns, rows, half}: a {64, 16, 1} box is one 128-byte half
  // of one page of one head.
  const uint64_t pool_rows = (uint64_t)a.num_pages * a.Hkv * QPAGE;
  const uint64_t dp[3] = {64, pool_rows, (uint64_t)H};
  const uint64_t sp[2] = {(uint64_t)a.D * 2, 128};
  const uint32_t bp[3] = {64, QPAGE, 1};
  // Block K/V as {64 columns, batch*rows, half, head}: one box per (b, head).
  const int KBR = (a.R + 15) & ~15;
  const uint64_t db[4] = {64, (uint64_t)a.B * a.R, (uint64_t)H, (uint64_t)a.Hkv};
  const uint64_t sb[3] = {(uint64_t)a.Hkv * a.D * 2, 128, (uint64_t)a.D * 2};
  const uint32_t bb[4] = {64, (uint32_t)KBR, (uint32_t)H, 1};
  // Query rows as {64 columns, head, batch*rows, half}: a {64, G, JBQ, 1}
  // box is one half of the rows (j, g) of a row group, in order j*G + g.
  const uint64_t dq[4] = {64, (uint64_t)a.Hq, (uint64_t)a.B * a.R, (uint64_t)H};
  const uint64_t sq[3] = {(uint64_t)a.D * 2, (uint64_t)a.Hq * a.D * 2, 128};
  const uint32_t bq[4] = {64, (uint32_t)G, (uint32_t)pl.jbq, 1};
  if (!encode_tensor_map_bf16(&maps[0], a.k_pages, 3, dp, sp, bp) ||
      !encode_tensor_map_bf16(&maps[1], a.v_pages, 3, dp, sp, bp) ||
      !encode_tensor_map_bf16(&maps[2], a.k_blk, 4, db, sb, bb) ||
      !encode_tensor_map_bf16(&maps[3], a.v_blk, 4, db, sb, bb) ||
      !encode_tensor_map_bf16(&maps[4], a.q, 4, dq, sq, bq))
    return cudaErrorInvalidValue;
  TcqParams p{};
  p.page_table = a.page_table;
  p.ctx_len = a.ctx_len;
  p.q = a.q;
  p.out = a.out;
  p.B = a.B;
  p.R = a.R;
  p.Hq = a.Hq;
  p.Hkv = a.Hkv;
  p.G = G;
  p.JB = pl.jb;
  p.JBQ = pl.jbq;
  p.RG = pl.rg;
  p.max_pages = a.max_pages;
  p.num_pages = a.num_pages;
  p.scale_log2 = a.scale * 1.4426950408889634f;
  p.kv_stable = a.kv_stable;
  p.block_full = a.block_full;
  p.err = err;
  if (a.D == 128) return launch_tcq_t<128>(maps, p, pl.cluster, a.B, a.Hkv, pl.rg, stream);
  if (a.D == 64) return launch_tcq_t<64>(maps, p, pl.cluster, a.B, a.Hkv, pl.rg, stream);
  return cudaErrorInvalidValue;
}

}  // namespace cospec
