// Verify attention on the tcgen05 tensor cores (teacher-forced verification
// pass, Sec. 3.1 Eq. 2 of the paper): the K+1 block rows of every query head
// of a KV group attend to the paged bf16 cache and, causally, to the block.
//
// One CTA owns (sequence b, KV head, KV split, row group); the splits of a
// (b, head, row group) form a thread-block cluster and merge their partial
// softmax states through distributed shared memory, as in the mma.sync
// variant.  Inside a CTA the roles are split by warp:
//   warps 0-2   TMA producers: 128-key K/V tiles (one 2-D box per page and
//               128-byte half, so each tile lands as [half][128 keys][128 B],
//               128B-swizzled) into a ring of stages, the query rows of the
//               group once, the block's own K/V as a final tile.  A warp
//               issues its bulk copies one after another, which holds one
//               warp to about 45 GB/s of 2 KB boxes; three warps split each
//               tile's 32 boxes;
//   warp 3      MMA issuer (one thread):
//                 S^T = K Q^T   (M = 128 keys, N = query rows, K = D),
//                 O^T += V^T P^T (M = D, N = query rows, K = keys; V^T is
//                               read MN-major straight from the V tile);
//               S^T is double-buffered in TMEM, O^T accumulates in TMEM;
//   warps 4-11  softmax: one thread per key (TMEM lane) turns a tile of S^T
//               into P^T (bf16, written over the tile's K, which the MMA no
//               longer needs), rescales O^T when needed and reads it out at
//               the end.  Two warps share each TMEM lane quarter and split
//               the query-row columns, so every SM sub-partition holds two
//               softmax warps that hide each other's latencies.
// Keys are the MMA M dimension because a verify block has few query rows
// (G * (K+1)): spreading keys over threads keeps every softmax lane busy.
//
// Softmax with a lazy reference maximum: per row, scores are taken relative
// to m_ref, set exactly from the first tile; a later tile changes m_ref (and
// rescales O^T and the partial sums) only when one of its scores exceeds
// m_ref by more than 2^8 in the exp2 domain, so P stays below 256.  The sum
// l = sum_k exp2(x_k - m_ref) is kept per thread and reduced once at the end.
#include <cuda.h>
#include <math.h>

#include "cospec_device.cuh"
#include "cospec_internal.h"

namespace cospec {

namespace {

constexpr int TKT = 128;          // keys per cache tile (8 pages) = MMA M
constexpr int TPPT = TKT / 16;    // pages per tile
constexpr int TPAGE = 16;         // page size (fixed)
constexpr int TROWB = 128;        // bytes of one swizzled smem row
constexpr int TC_PROD = 3;        // producer warps
constexpr int TC_MMA_WARP = 3;    // MMA issuer warp
constexpr int TC_SOFT0 = 4;       // first softmax warp
constexpr int TC_THREADS = 384;   // producer warps, MMA warp, 8 softmax warps
constexpr int TC_SOFT = 256;      // softmax threads
constexpr float LAZY_LOG2 = 8.f;  // rescale only when a score exceeds m_ref by this (log2)
constexpr uint64_t TC_WAIT_NS = 2000000000ull;

struct TcParams {
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

template <int D, int NT>
struct TcLayout {
  static constexpr int H = D / 64;                  // 128-byte halves of a key row
  static constexpr int KVB = H * TKT * TROWB;       // K (or V) of a tile: [half][128 keys][128 B]
  static constexpr int STAGE = 2 * KVB;             // K then V
  static constexpr int NS = 3;                      // 192 KB (D = 128) / 96 KB ring
  static constexpr int PCS = 8192;                  // P^T: two 64-key chunks [N rows][128 B], 8 KB apart
  static constexpr int RING = NS * STAGE;
  static constexpr int QH = NT * TROWB;             // one half of the query rows
  static constexpr int QOFF = RING;
  static constexpr int MISC = QOFF + H * QH;
  // barriers: full[NS], empty[NS], q_full, s_full[2], s_empty[2], p_full[2], pv_done,
  // mma_done, recv_bar
  static constexpr int NBAR = 2 * NS + 10;
  static constexpr int HOLDER = MISC + NBAR * 8;            // TMEM base address
  static constexpr int FLAGS = HOLDER + 16;                 // int [2][8] votes, [2] rescale, abort
  static constexpr int MREF = FLAGS + 128;                  // float [NT] reference maxima
  static constexpr int ALPHA = MREF + NT * 4;               // float [NT]
  static constexpr int RED = ALPHA + NT * 4;                // float [4][NT]
  static constexpr int LSUM = RED + 4 * NT * 4;             // float [NT]
  static constexpr int TOTAL = LSUM + NT * 4;
  // partial rows after the last tile, in the idle ring: PART [NT], RECV [NT + 15]
  static constexpr int PD = D + 8;
  static constexpr int ROWP = PD * 4;
  static constexpr int PART = 0;
  static constexpr int RECV = NT * ROWP;
  static_assert(RECV + (NT + 15) * ROWP <= RING, "partials must fit in the ring");
  // TMEM columns: S^T buffers at 0 and NT, O^T at 2 NT
  static constexpr uint32_t TCOLS = (3 * NT <= 128) ? 128u : 256u;
};

CS_DEV void tmem_ld16_async(uint32_t taddr, float* v) {
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
CS_DEV void tmem_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
CS_DEV void tmem_st16(uint32_t taddr, const float* v) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,"
      "%14,%15,%16};" ::"r"(taddr),
      "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])),
      "r"(__float_as_uint(v[3])), "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])),
      "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])), "r"(__float_as_uint(v[8])),
      "r"(__float_as_uint(v[9])), "r"(__float_as_uint(v[10])), "r"(__float_as_uint(v[11])),
      "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])), "r"(__float_as_uint(v[14])),
      "r"(__float_as_uint(v[15]))
      : "memory");
}
CS_DEV void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

// Descriptor of an MN-major operand in the 128B-swizzle layout: 64-element
// rows of 128 bytes along M, consecutive rows = consecutive K; `lbo` bytes
// between the 64-element groups along M, 1024 bytes between 8-row groups
// along K.
CS_DEV uint64_t smem_desc_mn_sw128(uint32_t saddr, uint32_t lbo) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFF) >> 4);
  d |= (uint64_t)((lbo >> 4) & 0x3FFF) << 16;
  d |= (uint64_t)(1024 >> 4) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
}

// Column reduction of a [32 lanes][C] register block: afterwards lane l
// holds, in v[0 .. C/32), the reductions over all 32 lanes of columns
// l*C/32 .. l*C/32 + C/32 - 1.  Each butterfly level hands half of the
// remaining columns to the partner lane.
template <int C, bool MAX>
CS_DEV void warp_col_reduce(float (&v)[C], int lane) {
#pragma unroll
  for (int lvl = 0; lvl < 5; ++lvl) {
    const int off = 16 >> lvl;
    const int w = C >> lvl;          // columns still held
    const bool up = (lane & off) != 0;
#pragma unroll
    for (int i = 0; i < w / 2; ++i) {
      const float send = up ? v[i] : v[i + w / 2];
      const float keep = up ? v[i + w / 2] : v[i];
      const float recv = __shfl_xor_sync(0xffffffffu, send, off);
      v[i] = MAX ? fmaxf(keep, recv) : keep + recv;
    }
  }
}

// The N (<= NT) columns of one S^T buffer for this warp's 32 TMEM lanes;
// columns past N read as 0.
template <int NT>
CS_DEV void load_s(uint32_t taddr, int N, float (&x)[NT]) {
#pragma unroll
  for (int c = 0; c < NT / 16; ++c) {
    if (c * 16 < N) {
      tmem_ld16_async(taddr + c * 16, &x[c * 16]);
    } else {
#pragma unroll
      for (int i = 0; i < 16; ++i) x[c * 16 + i] = 0.f;
    }
  }
  tmem_wait_ld();
}

template <int D, int NT>
__global__ void __launch_bounds__(TC_THREADS, 1)
    verify_attn_tc_kernel(const __grid_constant__ CUtensorMap map_kp,
                          const __grid_constant__ CUtensorMap map_vp,
                          const __grid_constant__ CUtensorMap map_kb,
                          const __grid_constant__ CUtensorMap map_vb,
                          const __grid_constant__ CUtensorMap map_q, const TcParams p) {
  using LY = TcLayout<D, NT>;
  constexpr int H = LY::H;
  constexpr int NS = LY::NS;
  constexpr int PD = LY::PD;

  extern __shared__ __align__(16) uint8_t smem_raw[];
  // 1024-byte aligned base (TMA 128B swizzle, UMMA descriptors), kept as an
  // offset from the shared array so that accesses stay shared-memory ones.
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + LY::MISC);
  uint64_t* empty = full + NS;
  uint64_t* q_full = empty + NS;
  uint64_t* s_full = q_full + 1;      // [2]
  uint64_t* s_empty = s_full + 2;     // [2]
  uint64_t* p_full = s_empty + 2;     // [2]
  uint64_t* pv_done = p_full + 2;
  uint64_t* mma_done = pv_done + 1;
  uint64_t* recv_bar = mma_done + 1;  // partials received from the cluster
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(smem + LY::HOLDER);
  volatile int* votes = reinterpret_cast<volatile int*>(smem + LY::FLAGS);   // [2][8]
  volatile int* resc = votes + 16;                                            // [2]
  volatile int* abort_flag = votes + 18;
  volatile int* n_issued = votes + 19;     // tiles the producer loaded (abort tail)
  float* m_ref = reinterpret_cast<float*>(smem + LY::MREF);
  float* alpha_s = reinterpret_cast<float*>(smem + LY::ALPHA);
  float* red = reinterpret_cast<float*>(smem + LY::RED);
  float* lsum = reinterpret_cast<float*>(smem + LY::LSUM);
  uint8_t* qs = smem + LY::QOFF;

  const int S = (int)cluster_nctarank();
  const int rank = (int)cluster_ctarank();
  const int kvh = blockIdx.y / p.RG, rg = blockIdx.y % p.RG;
  const int j0 = rg * p.JB;                          // first block row of this group
  const int nj = min(p.JB, p.R - j0);
  const int NR = nj * p.G;                           // query rows of this group (<= NT)
  const int N = (NR + 15) & ~15;                     // MMA N
  const int qrows = p.G * p.JBQ;                     // rows the query box writes
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  if (tid == 0) {
    for (int s = 0; s < NS; ++s) {
      mbar_init(&full[s], TC_PROD);        // one arrival per producer warp
      mbar_init(&empty[s], 1);
    }
    mbar_init(q_full, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&s_full[i], 1);
      mbar_init(&s_empty[i], 1);
      mbar_init(&p_full[i], 1);
    }
    mbar_init(pv_done, 1);
    mbar_init(mma_done, 1);
    mbar_init(recv_bar, 1);
    for (int i = 0; i < 20; ++i) votes[i] = 0;
    fence_barrier_init();
  }
  if (warp == TC_MMA_WARP) {
    tmem_alloc(tmem_holder, LY::TCOLS);
    tmem_relinquish();
  }
  // Query rows past the box (MMA padding) are zeroed once, so every S^T
  // column stays finite.
  for (int e = tid; e < H * (N - qrows) * 8; e += TC_THREADS) {
    const int h = e / ((N - qrows) * 8), rem = e % ((N - qrows) * 8);
    *reinterpret_cast<uint4*>(qs + h * LY::QH + (qrows + rem / 8) * TROWB + (rem % 8) * 16) =
        make_uint4(0u, 0u, 0u, 0u);
  }
  for (int r = tid; r < NT; r += TC_THREADS) {
    // +inf marks padding rows: their scores become -inf, their weights 0
    m_ref[r] = (r < NR) ? -INFINITY : INFINITY;
    lsum[r] = 0.f;
  }
  fence_proxy_async_smem();
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
  const int b = p.B > 1 ? sequence_by_rank(p.ctx_len, p.B, (int)blockIdx.z,
                                           reinterpret_cast<volatile int*>(red))
                        : (int)blockIdx.z;
  const int C = p.ctx_len[b];
  const bool bad = (C < 0) || (C > p.max_pages * TPAGE);
  if (bad && rank == 0 && kvh == 0 && rg == 0 && tid == 0) set_err(p.err, ERR_CTX);
  const int nct = bad ? 0 : (C + TKT - 1) / TKT;
  const int tps = (nct + S - 1) / S;
  const int t_begin = min(nct, rank * tps);
  const int n = min(nct, t_begin + tps) - t_begin;   // cache tiles of this CTA
  const bool do_blk = !bad && rank == S - 1;         // the block's keys: last CTA
  const int T = n + (do_blk ? 1 : 0);
  const int npages = (C + TPAGE - 1) / TPAGE;
  const int KBR = (p.R + 15) & ~15;                  // block keys padded to 16

  if (warp < TC_PROD) {
    // ------------------------------------------------------------ producers
    const int pw = warp;
    constexpr int NBOX = 2 * H * TPPT;                  // boxes of a full tile
    constexpr int BPW = (NBOX + TC_PROD - 1) / TC_PROD; // boxes per producer warp
    const int e = pw * BPW + lane;                      // this lane's box
    const bool mine = lane < BPW && e < NBOX;
    if (pw == 0 && lane == 0) {
      tma_prefetch_desc(&map_kp);
      tma_prefetch_desc(&map_vp);
      tma_prefetch_desc(&map_q);
    }
    // KV is read once per row group: with several groups per (sequence, head)
    // (running side by side) keep it in L2 for the siblings
    const uint64_t pol = p.RG > 1 ? l2_policy_evict_normal() : l2_policy_evict_first();
    const int* ptab = p.page_table + (size_t)b * p.max_pages + (size_t)t_begin * TPPT;
    const int my_pages = min(n * TPPT, npages - t_begin * TPPT);
    int pid = 0;
    bool ok = true;
    int issued = 0;                      // tiles whose loads were issued
    auto issue_cache = [&](int t) {
      const int st = t % NS;
      uint8_t* sb = smem + st * LY::STAGE;
      if ((t & 3) == 0) {                // 32 page ids = the next 4 tiles, one per lane
        const int e = t * TPPT + lane;
        pid = (e < my_pages) ? __ldg(ptab + e) : 0;
      }
      const int np = min(TPPT, npages - (t_begin + t) * TPPT);
      // box e: page e / (2H), tensor (e / H) & 1 (K, V), half e % H
      const int pg = e / (2 * H);
      int pgid = __shfl_sync(0xffffffffu, pid, (t & 3) * TPPT + (pg & 7));
      if (lane == 0) {
        // this warp's boxes within the tile's np pages
        const int lo = pw * BPW, hi = min(NBOX, min(lo + BPW, np * 2 * H));
        mbar_arrive_expect_tx(&full[st], (uint32_t)(max(0, hi - lo) * TPAGE * TROWB));
      }
      __syncwarp();
      if (mine && pg < np) {
        if ((unsigned)pgid >= (unsigned)p.num_pages) {
          set_err(p.err, ERR_PAGE);
          pgid = 0;
        }
        const int tensor = (e / H) & 1, h = e % H;
        tma_load_3d(smem_u32(sb + tensor * LY::KVB + h * (TKT * TROWB) + pg * (TPAGE * TROWB)),
                    tensor ? (const void*)&map_vp : (const void*)&map_kp, &full[st], 0,
                    (pgid * p.Hkv + kvh) * TPAGE, h, pol);
      }
      __syncwarp();
    };
    auto wait_slot = [&](int t) -> bool {
      if (t < NS) return true;
      const int st = t % NS;
      const bool w = mbar_wait(&empty[st], (uint32_t)((t / NS) - 1) & 1u, TC_WAIT_NS);
      return __all_sync(0xffffffffu, w) && !*abort_flag;
    };
    const int pre = min(n, NS);
    for (int t = 0; t < pre; ++t) {      // with the stable-cache promise: before the wait
      issue_cache(t);
      ++issued;
    }
    if (pw == 0 && pre == NS && n > NS) {
      // The ring is full: pull the next tile's pages into L2.
      const int e = NS * TPPT + (lane >> 1);
      const int pg = __shfl_sync(0xffffffffu, pid, e & 31);
      if (lane < 2 * TPPT && e < my_pages && (unsigned)pg < (unsigned)p.num_pages)
        for (int h = 0; h < H; ++h)
          tma_prefetch_l2_3d((lane & 1) ? (const void*)&map_vp : (const void*)&map_kp, 0,
                             (pg * p.Hkv + kvh) * TPAGE, h);
    }
    // the query rows and the block K/V come from the previous kernel; the
    // other producers read only the (stable) cache
    if (p.kv_stable && pw == 0) griddep_wait();
    if (T > 0 && pw == 0 && lane == 0) {
      mbar_arrive_expect_tx(q_full, (uint32_t)(H * qrows * TROWB));
      for (int h = 0; h < H; ++h)
        tma_load_4d(smem_u32(qs + h * LY::QH), &map_q, q_full, 0, kvh * p.G, b * p.R + j0, h, pol);
    }
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
        if (pw == 0 && lane == 0) {
          // one box per tensor: KBR rows from block row 0 of this head, all
          // halves, landing as [half][KBR rows][128 B]
          mbar_arrive_expect_tx(&full[st], (uint32_t)(2 * H * KBR * TROWB));
          tma_load_4d(smem_u32(sb), &map_kb, &full[st], 0, b * p.R, 0, kvh, pol);
          tma_load_4d(smem_u32(sb + LY::KVB), &map_vb, &full[st], 0, b * p.R, 0, kvh, pol);
        } else if (lane == 0) {
          mbar_arrive(&full[st]);
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
    if (pw == 0 && lane == 0) *n_issued = issued;
  } else if (warp == TC_MMA_WARP) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0 && T > 0) {
      const uint32_t idesc_qk = idesc_bf16_f32(128, N);
      const uint32_t idesc_pv = idesc_bf16_f32(128, N) | (1u << 15);   // A (V^T) MN-major
      const uint32_t q0 = smem_u32(qs);
      bool ok = mbar_wait(q_full, 0, TC_WAIT_NS);
      auto issue_s = [&](int t) {
        const int st = t % NS;
        const uint32_t kb = smem_u32(smem + st * LY::STAGE);
        const uint32_t khalf = (do_blk && t == n) ? (uint32_t)(KBR * TROWB) : (uint32_t)(TKT * TROWB);
#pragma unroll
        for (int h = 0; h < H; ++h)
#pragma unroll
          for (int ks = 0; ks < 4; ++ks)
            umma_bf16(tmem_base + (uint32_t)((t & 1) * NT), smem_desc_sw128(kb + h * khalf + ks * 32),
                      smem_desc_sw128(q0 + h * LY::QH + ks * 32), idesc_qk, (h | ks) != 0 ? 1u : 0u);
        umma_commit(&s_full[t & 1]);
      };
      auto issue_pv = [&](int u) {
        const int st = u % NS;
        const uint32_t kb = smem_u32(smem + st * LY::STAGE);
        const bool blk = do_blk && u == n;
        const uint32_t vhalf = blk ? (uint32_t)(KBR * TROWB) : (uint32_t)(TKT * TROWB);
        const int nks = blk ? KBR / 16 : TKT / 16;
        // D = 64: the second 64-row group of M repeats the first (lbo 0)
        const uint32_t lbo = (H == 2) ? vhalf : 0u;
        for (int ks = 0; ks < nks; ++ks)
          umma_bf16(tmem_base + 2 * NT, smem_desc_mn_sw128(kb + LY::KVB + ks * 2048, lbo),
                    smem_desc_sw128(kb + (ks >> 2) * LY::PCS + (ks & 3) * 32), idesc_pv,
                    (u > 0 || ks > 0) ? 1u : 0u);
        umma_commit(&empty[st]);
        umma_commit(pv_done);
      };
      // Issue whichever product is ready, so that a P.V product (which frees
      // a ring stage for the producer) never waits behind the next tile's
      // load.  S^T of tile ts needs the tile and a free S^T buffer; at most
      // one tile's S^T runs ahead of the oldest pending P.V, which also keeps
      // every barrier within one phase of the parity tested here.
      int ts = 0, tp = 0;
      uint64_t t_last = global_timer_ns();
      while (ok && tp < T) {
        bool did = false;
        if (tp < ts && mbar_test(&p_full[tp & 1], (uint32_t)(tp >> 1) & 1u)) {
          tc_fence_after();
          issue_pv(tp);
          ++tp;
          did = true;
        }
        if (ts < T && ts <= tp + 1 && mbar_test(&full[ts % NS], (uint32_t)(ts / NS) & 1u) &&
            (ts < 2 || mbar_test(&s_empty[ts & 1], (uint32_t)((ts >> 1) - 1) & 1u))) {
          tc_fence_after();
          issue_s(ts);
          ++ts;
          did = true;
        }
        if (did) {
          t_last = global_timer_ns();
        } else if (*abort_flag || global_timer_ns() - t_last > TC_WAIT_NS) {
          ok = false;
        }
      }
      if (!ok) {
        set_err(p.err, ERR_TIMEOUT);
        *abort_flag = 1;
      }
      // every MMA issued by this thread completes before TMEM is released
      umma_commit(mma_done);
      mbar_wait(mma_done, 0, TC_WAIT_NS);
    }
  } else {
    // ------------------------------------------------------------ softmax
    constexpr int HC = NT / 2;           // query-row columns of one softmax warp
    const int q = warp & 3;              // TMEM lane quarter this warp may access
    const int ew = warp - TC_SOFT0;
    const int col0 = (ew >> 2) * HC;     // first of this warp's columns
    const int etid = tid - TC_SOFT0 * 32;
    const bool s_warp = true;            // every warp owns 32 keys (TMEM lanes)
    const int key = q * 32 + lane;
    if (p.kv_stable) {
      // warm L2 with the group's query rows before the producer's TMA
      for (int e = etid; e < NR * (D * 2 / 128); e += TC_SOFT) {
        const int r = e / (D * 2 / 128), part_ = e % (D * 2 / 128);
        const int j = j0 + r / p.G, g = r % p.G;
        prefetch_l2(p.q + (((size_t)b * p.R + j) * p.Hq + (size_t)kvh * p.G + g) * D + part_ * 64);
      }
    }
    float l_part[HC];
    float mref[HC];                      // m_ref of this warp's rows
#pragma unroll
    for (int i = 0; i < HC; ++i) {
      l_part[i] = 0.f;
      mref[i] = (col0 + i < NR) ? -INFINITY : INFINITY;
    }
    const float sc = p.scale_log2;
    bool aborted = false;
    for (int t = 0; t < T; ++t) {
      const int st = t % NS;
      uint8_t* sb = smem + st * LY::STAGE;
      const bool blk = do_blk && t == n;
      const bool okw = __all_sync(0xffffffffu, mbar_wait(&s_full[t & 1], (uint32_t)(t >> 1) & 1u, TC_WAIT_NS));
      tc_fence_after();
      const uint32_t taddr = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)((t & 1) * NT + col0);
      // cache keys below C are seen by every row; block key j < R by the
      // rows of block rows >= j (causal inside the block)
      const bool kvalid = blk ? (key < p.R) : ((t_begin + t) * TKT + key < C);
      // block key j is seen by row r iff j <= j0 + r / G, i.e. (j - j0) * G <= r
      // (causal), or by every row (full block)
      const int kg = p.block_full ? -1 : (key - j0) * p.G;
      float x[HC];
      float excess = -INFINITY;
      if (s_warp && okw) {
        load_s<HC>(taddr, N - col0, x);
        // x = score * log2(e) / sqrt(D) - m_ref; with m_ref unset (-inf) this
        // is +inf and forces the exact path below
        if (!blk) {
#pragma unroll
          for (int i = 0; i < HC; ++i) {
            x[i] = kvalid ? fmaf(x[i], sc, -mref[i]) : -INFINITY;
            excess = fmaxf(excess, x[i]);
          }
        } else {
#pragma unroll
          for (int i = 0; i < HC; ++i) {
            x[i] = (kvalid && kg <= col0 + i) ? fmaf(x[i], sc, -mref[i]) : -INFINITY;
            excess = fmaxf(excess, x[i]);
          }
        }
      }
      // vote: bit 0 = this warp saw a score above m_ref + 2^8, bit 1 = timeout
      const bool hi = __any_sync(0xffffffffu, excess > LAZY_LOG2);
      if (lane == 0) votes[(t & 1) * 8 + ew] = (hi ? 1 : 0) | (okw ? 0 : 2);
      if (etid == 0) resc[t & 1] = 0;
      named_bar_sync(1, TC_SOFT);
      int vote = 0;
#pragma unroll
      for (int w = 0; w < 8; ++w) vote |= votes[(t & 1) * 8 + w];
      if (vote & 2) {
        if (etid == 0) {
          set_err(p.err, ERR_TIMEOUT);
          *abort_flag = 1;
        }
        aborted = true;
        break;
      }
      if (vote & 1) {
        // Exact path: absolute scaled scores of the tile, their column
        // maxima, the new references and the factors for what came before.
        if (s_warp) {
          load_s<HC>(taddr, N - col0, x);
#pragma unroll
          for (int i = 0; i < HC; ++i)
            x[i] = (kvalid && (!blk || kg <= col0 + i)) ? x[i] * sc : -INFINITY;
          // column maxima over the warp's 32 keys (a 16-column half padded to 32)
          float mx[32];
#pragma unroll
          for (int i = 0; i < 32; ++i) mx[i] = (i < HC) ? x[i] : -INFINITY;
          warp_col_reduce<32, true>(mx, lane);
          if (lane < HC) red[q * NT + col0 + lane] = mx[0];
        }
        named_bar_sync(1, TC_SOFT);
        if (etid < NT) {
          const int r = etid;
          const float mo = m_ref[r];
          float mn = mo, a = 1.f;
          if (r < NR) {
            mn = fmaxf(fmaxf(mo, fmaxf(red[r], red[NT + r])), fmaxf(red[2 * NT + r], red[3 * NT + r]));
            // alpha rescales what was accumulated against mo (nothing when mo = -inf)
            a = (mn == mo) ? 1.f : (mo == -INFINITY ? 0.f : exp2_approx(mo - mn));
          }
          m_ref[r] = mn;
          alpha_s[r] = a;
          if (a < 1.f && t > 0) resc[t & 1] = 1;
        }
        named_bar_sync(1, TC_SOFT);
        if (s_warp) {
#pragma unroll
          for (int i = 0; i < HC; ++i) {
            mref[i] = m_ref[col0 + i];
            l_part[i] *= alpha_s[col0 + i];
            x[i] -= mref[i];
          }
        }
        if (resc[t & 1]) {
          // O^T holds tiles 0..t-1: wait for the last of them, then scale its columns.
          const bool okp = __all_sync(0xffffffffu, mbar_wait(pv_done, (uint32_t)(t - 1) & 1u, TC_WAIT_NS));
          tc_fence_after();
          if (okp && (H == 2 || q < 2)) {
            const uint32_t oaddr = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(2 * NT);
#pragma unroll 1
            for (int c = col0 / 16; c < (col0 + HC) / 16; ++c) {
              if (c * 16 < N) {
                float o[16];
                tmem_ld16_async(oaddr + c * 16, o);
                tmem_wait_ld();
#pragma unroll
                for (int i = 0; i < 16; ++i) o[i] *= alpha_s[c * 16 + i];
                tmem_st16(oaddr + c * 16, o);
              }
            }
            tmem_wait_st();
          }
          if (!okp && lane == 0) set_err(p.err, ERR_TIMEOUT);
        }
      }
      // P^T (bf16) over the tile's K: row r of 64 keys, 128B-swizzled.
      if (s_warp) {
        // rows past NR have x = -inf, so whole 16-row chunks are written;
        // keys 0..63 and 64..127 go to two K-major chunks of 64 keys
        const int kk = key & 63;
        uint8_t* prow = sb + (key >> 6) * LY::PCS + (kk & 7) * 2;
#pragma unroll
        for (int c = 0; c < HC / 16; ++c) {
          if (col0 + c * 16 < N) {
#pragma unroll
            for (int i = 0; i < 16; ++i) {
              const int r = col0 + c * 16 + i;
              const float pr = exp2_approx(x[c * 16 + i]);
              l_part[c * 16 + i] += pr;
              *reinterpret_cast<__nv_bfloat16*>(prow + r * TROWB + (((kk >> 3) ^ (r & 7)) << 4)) =
                  __float2bfloat16_rn(pr);
            }
          }
        }
      }
      // V rows of keys outside the context (or past the block) may hold stale
      // bytes: zero them so that their zero weights contribute exactly 0.
      {
        const int vr = blk ? p.R : min(TKT, C - (t_begin + t) * TKT);
        const int rows = blk ? KBR : TKT;
        const int vhalf = rows * TROWB;
        uint8_t* vb = sb + LY::KVB;
        for (int e = etid; e < (rows - vr) * H * 8; e += TC_SOFT) {
          const int row = vr + e / (H * 8), rem = e % (H * 8);
          *reinterpret_cast<uint4*>(vb + (rem / 8) * vhalf + row * TROWB + (rem % 8) * 16) =
              make_uint4(0u, 0u, 0u, 0u);
        }
      }
      fence_proxy_async_smem();
      tc_fence_before();
      named_bar_sync(1, TC_SOFT);
      if (etid == 0) {
        mbar_arrive(&p_full[t & 1]);
        mbar_arrive(&s_empty[t & 1]);
      }
    }
    // Totals of the partial sums, and the end of the last P.V product.
    if (s_warp) {
      float sm[32];
#pragma unroll
      for (int i = 0; i < 32; ++i) sm[i] = (i < HC) ? l_part[i] : 0.f;
      warp_col_reduce<32, false>(sm, lane);
      if (lane < HC) red[q * NT + col0 + lane] = sm[0];
    }
    if (T > 0 && !aborted) {
      const bool okp = __all_sync(0xffffffffu, mbar_wait(pv_done, (uint32_t)(T - 1) & 1u, TC_WAIT_NS));
      if (!okp && lane == 0) set_err(p.err, ERR_TIMEOUT);
    }
    tc_fence_after();
    named_bar_sync(1, TC_SOFT);
    if (etid < NT)
      lsum[etid] = (T > 0 && !aborted)
                       ? (red[etid] + red[NT + etid]) + (red[2 * NT + etid] + red[3 * NT + etid])
                       : 0.f;
  }
  __syncthreads();
  tc_fence_after();

  // The ring is idle from here on.  Tell the cluster (its CTAs may push into
  // RECV once every CTA has arrived) and write this CTA's partial meanwhile.
  const int rpo = (NR + S - 1) / S;      // rows finished by each owner
  if (S > 1) {
    if (tid == 0) mbar_arrive_expect_tx(recv_bar, (uint32_t)(S * rpo * LY::ROWP));
    cluster_arrive_relaxed();
  }
  float* part = reinterpret_cast<float*>(smem + LY::PART);
  const bool have = T > 0 && !*abort_flag;
  if (warp >= TC_SOFT0) {
    const int q = warp & 3;
    const int d = q * 32 + lane;
    const int c0 = ((warp - TC_SOFT0) >> 2) * (NT / 32);   // this warp's half of the row chunks
    if (H == 2 || q < 2) {
      const uint32_t taddr = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(2 * NT);
#pragma unroll
      for (int c = c0; c < c0 + NT / 32; ++c) {
        if (c * 16 < N) {
          float o[16];
          if (have) {
            tmem_ld16_async(taddr + c * 16, o);
            tmem_wait_ld();
          } else {
#pragma unroll
            for (int i = 0; i < 16; ++i) o[i] = 0.f;
          }
#pragma unroll
          for (int i = 0; i < 16; ++i)
            if (c * 16 + i < NR) part[(c * 16 + i) * PD + d] = o[i];
        }
      }
    }
  }
  for (int r = tid; r < NR; r += TC_THREADS) {
    part[r * PD + D] = have ? m_ref[r] : -INFINITY;
    part[r * PD + D + 1] = have ? lsum[r] : 0.f;
  }
  fence_proxy_async_smem();              // the bulk copies below read `part`
  tc_fence_before();
  __syncthreads();

  // Reduce-scatter over the cluster: owner o finishes rows [o*rpo, (o+1)*rpo).
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
    cluster_arrive_relaxed();            // everything addressed to this CTA has landed
  }
  const int row0 = rank * rpo;
  // Per owned row: one warp forms the common maximum over the S partials and
  // each partial's weight exp2(m_s - M) / L (kept in the idle reduction
  // buffer); then every output chunk is a plain weighted sum.
  float* scl = red;                                          // [S][rpo] <= 4 NT floats
  for (int rr = warp; rr < rpo; rr += TC_THREADS / 32) {
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
  for (int e = tid; e < rpo * (D / 4); e += TC_THREADS) {
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
    const int j = j0 + r / p.G, g = r % p.G;
    __nv_bfloat16* dst = p.out + (((size_t)b * p.R + j) * p.Hq + (size_t)kvh * p.G + g) * D + c;
    uint2 pk;
    pk.x = pack_bf16(acc.x, acc.y);
    pk.y = pack_bf16(acc.z, acc.w);
    *reinterpret_cast<uint2*>(dst) = pk;
  }
  if (S > 1) cluster_wait();             // every copy out of this CTA has landed

  // After an abort a copy may still be in flight: wait (bounded) for the
  // last fill of every stage the producer used before shared memory goes.
  if (*abort_flag && tid == 0) {
    const int ni = *n_issued;
    for (int st = 0; st < NS && st < ni; ++st) {
      const int last = st + ((ni - 1 - st) / NS) * NS;
      mbar_wait(&full[st], (uint32_t)(last / NS) & 1u, TC_WAIT_NS);
    }
    if (T > 0) mbar_wait(q_full, 0, TC_WAIT_NS);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == TC_MMA_WARP) {
    __syncwarp();
    tmem_dealloc(tmem_base, LY::TCOLS);
  }
}

template <int D, int NT>
size_t tc_smem_bytes() {
  return (size_t)TcLayout<D, NT>::TOTAL + 1024;
}

// Limits already set on each instantiation of the kernel.
template <int D, int NT>
KernelLimits& tc_limits() {
  static KernelLimits lim;
  return lim;
}

template <int D, int NT>
cudaError_t launch_tc_t(const CUtensorMap* maps, const TcParams& p, int S, int B, int Hkv, int RG,
                        cudaStream_t stream) {
  const size_t smem = tc_smem_bytes<D, NT>();
  auto kern = verify_attn_tc_kernel<D, NT>;
  const cudaError_t e = ensure_kernel_limits((const void*)kern, tc_limits<D, NT>(), smem, true);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(S, Hkv * RG, B);
  cfg.blockDim = dim3(TC_THREADS, 1, 1);
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

template <int D, int NT>
int max_cluster_tc_t(int S, int Hkv, int B, int RG) {
  const size_t smem = tc_smem_bytes<D, NT>();
  auto kern = verify_attn_tc_kernel<D, NT>;
  if (ensure_kernel_limits((const void*)kern, tc_limits<D, NT>(), smem, true) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(S, Hkv * RG, B);
  cfg.blockDim = dim3(TC_THREADS, 1, 1);
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

bool tc_attn_supported(int D, int G) { return (D == 64 || D == 128) && G >= 1 && G <= 64; }

int attn_tc_max_active_clusters(int D, int nt, int S, int Hkv, int B, int RG) {
  if (D == 128 && nt == 32) return max_cluster_tc_t<128, 32>(S, Hkv, B, RG);
  if (D == 128 && nt == 64) return max_cluster_tc_t<128, 64>(S, Hkv, B, RG);
  if (D == 64 && nt == 32) return max_cluster_tc_t<64, 32>(S, Hkv, B, RG);
  if (D == 64 && nt == 64) return max_cluster_tc_t<64, 64>(S, Hkv, B, RG);
  return 0;
}

cudaError_t launch_verify_attn_tc(const AttnArgs& a, const AttnPlan& pl, int* err,
                                  cudaStream_t stream) {
  const int H = a.D / 64;
  const int G = a.Hq / a.Hkv;
  CUtensorMap maps[5];
  // Pool as {64 columns, rows, half}: a {64, 16, 1} box is one 128-byte half
  // of one page of one head.
  const uint64_t pool_rows = (uint64_t)a.num_pages * a.Hkv * TPAGE;
  const uint64_t dp[3] = {64, pool_rows, (uint64_t)H};
  const uint64_t sp[2] = {(uint64_t)a.D * 2, 128};
  const uint32_t bp[3] = {64, TPAGE, 1};
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
  TcParams p{};
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
  if (a.D == 128 && pl.nt == 32) return launch_tc_t<128, 32>(maps, p, pl.cluster, a.B, a.Hkv, pl.rg, stream);
  if (a.D == 128 && pl.nt == 64) return launch_tc_t<128, 64>(maps, p, pl.cluster, a.B, a.Hkv, pl.rg, stream);
  if (a.D == 64 && pl.nt == 32) return launch_tc_t<64, 32>(maps, p, pl.cluster, a.B, a.Hkv, pl.rg, stream);
  if (a.D == 64 && pl.nt == 64) return launch_tc_t<64, 64>(maps, p, pl.cluster, a.B, a.Hkv, pl.rg, stream);
  return cudaErrorInvalidValue;
}

}  // namespace cospec
