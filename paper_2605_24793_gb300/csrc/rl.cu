// RL stage of CoSpec (Sec. 3.4): per-decision shaped rewards, rollout
// returns, rebalanced group-normalised advantages, per-decision advantages
// and the clipped objective with its entropy and KL terms.
//
// One CTA per prompt group.  A warp takes a rollout and its lanes take
// rounds: each lane scans its round's K positions once (s, i*, rho, the
// effective decisions and their g) and the warp sums the returns.  Warp 0
// then forms the group statistics (float64, so that the standardisation of
// nearly equal returns is not decided by float32 rounding), and the warps
// revisit the rounds for the decision advantages and the objective terms.
// Per-group partial sums of the objective go to the workspace and a one-CTA
// kernel adds them in a fixed order.
#include <math.h>

#include "../../include/cospec.h"
#include "cospec_device.cuh"
#include "cospec_internal.h"

namespace cospec {

namespace {

constexpr int RL_THREADS = 256;
constexpr int RL_WARPS = RL_THREADS / 32;

struct RLArgs {
  int num_groups, num_rollouts, num_rounds, K;
  const int32_t* group_off;
  const uint8_t* correct;
  const int32_t* round_off;
  const uint8_t* match;
  const uint8_t* accept;
  const float* ell;
  cospec_rl_params prm;
  const float* ratio;
  const float* p_new;
  const float* p_ref;
  float* g;
  uint8_t* eff;
  float* rho;
  float* J;
  float* Jbar;
  float* adv;
  float* adv_dec;
  double* ws_j;      // [num_rollouts] returns
  double* ws_abs;    // [num_rollouts] sum |g| of each rollout
  double* ws_adv;    // [num_rollouts] rollout advantages
  double* part;      // [num_groups][3] objective partial sums
  int* err;
};

CS_DEV double warp_sum(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// One round: s = first rejected mismatch (else K+1), i* = first mismatch,
// rho = (s - i*) / (K + 1 - i*); the effective decisions are the mismatches
// at positions <= min(s, K).  Writes g / eff / rho of the round and adds its
// returns to (sg, sa).
CS_DEV void rl_round(const RLArgs& a, int r, bool correct, double& sg, double& sa) {
  const int K = a.K;
  const uint8_t* dm = a.match + (size_t)r * K;
  const uint8_t* ac = a.accept + (size_t)r * K;
  int s = K + 1, istar = 0;
  for (int i = 1; i <= K; ++i) {
    if (dm[i - 1] == 0) {
      if (istar == 0) istar = i;
      if (ac[i - 1] == 0) {
        s = i;
        break;
      }
    }
  }
  const double rho = istar ? (double)(s - istar) / (double)(K + 1 - istar) : 0.0;
  a.rho[r] = istar ? (float)rho : __int_as_float(0x7fc00000);
  const int last = s < K ? s : K;
  const int irej = (s <= K) ? s : K + 1;
  for (int i = 1; i <= K; ++i) {
    const size_t e = (size_t)r * K + (i - 1);
    const bool effective = dm[i - 1] == 0 && i <= last;
    double gv = 0.0;
    if (effective) {
      if (correct) {
        gv = rho;
      } else {
        const bool acc = ac[i - 1] == 1 && i < irej;
        const bool rej = i == irej && irej <= K;
        gv = -(double)a.prm.alpha * fabs((double)a.ell[e]) * (acc ? 1.0 : 0.0) -
             (double)a.prm.beta * (rej ? 1.0 : 0.0);
      }
      sg += gv;
      sa += fabs(gv);
    }
    a.g[e] = (float)gv;
    a.eff[e] = effective ? 1 : 0;
  }
}

CS_DEV double bern_entropy(double p) {
  double h = 0.0;
  if (p > 0.0) h -= p * log(p);
  if (p < 1.0) h -= (1.0 - p) * log(1.0 - p);
  return h;
}

CS_DEV double bern_kl(double p, double q) {
  double k = 0.0;
  if (p > 0.0) k += p * log(p / q);
  if (p < 1.0) k += (1.0 - p) * log((1.0 - p) / (1.0 - q));
  return k;
}

__global__ void __launch_bounds__(RL_THREADS) rl_group_kernel(const RLArgs a) {
  const int x = blockIdx.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __shared__ double red[3][RL_WARPS];
  const int m0 = a.group_off[x], m1 = a.group_off[x + 1];
  if (m0 < 0 || m1 < m0 || m1 > a.num_rollouts) {
    if (threadIdx.x == 0) {
      set_err(a.err, ERR_OFFSETS);
      if (a.part) a.part[3 * x] = a.part[3 * x + 1] = a.part[3 * x + 2] = 0.0;
    }
    return;
  }
  // ---- returns: warp per rollout, lane per round
  for (int m = m0 + warp; m < m1; m += RL_WARPS) {
    const int r0 = a.round_off[m], r1 = a.round_off[m + 1];
    const bool bad = r0 < 0 || r1 < r0 || r1 > a.num_rounds;
    double sg = 0.0, sa = 0.0;
    if (!bad)
      for (int r = r0 + lane; r < r1; r += 32) rl_round(a, r, a.correct[m] != 0, sg, sa);
    sg = warp_sum(sg);
    sa = warp_sum(sa);
    if (lane == 0) {
      if (bad) set_err(a.err, ERR_OFFSETS);
      a.ws_j[m] = sg;
      a.ws_abs[m] = sa;
      a.J[m] = (float)sg;
    }
  }
  __syncthreads();
  // ---- group statistics (warp 0): gamma, Jbar, mean, population sigma, Adv
  if (warp == 0) {
    const double eps = (double)a.prm.eps;
    double pos = 0.0, negabs = 0.0, npos = 0.0, nneg = 0.0;
    for (int m = m0 + lane; m < m1; m += 32) {
      const double j = a.ws_j[m];
      if (a.correct[m]) {
        pos += j;
        npos += 1.0;
      } else {
        negabs += fabs(j);
        nneg += 1.0;
      }
    }
    pos = warp_sum(pos);
    negabs = warp_sum(negabs);
    npos = warp_sum(npos);
    nneg = warp_sum(nneg);
    const double n = npos + nneg;
    const double gamma = (npos > 0.0 && nneg > 0.0) ? negabs / (pos + eps) : 1.0;
    const double eta = (npos == 0.0) ? (double)a.prm.eta_fail : 1.0;
    double sum = 0.0;
    for (int m = m0 + lane; m < m1; m += 32) sum += a.correct[m] ? gamma * a.ws_j[m] : a.ws_j[m];
    sum = warp_sum(sum);
    const double mu = n > 0.0 ? sum / n : 0.0;
    double var = 0.0;
    for (int m = m0 + lane; m < m1; m += 32) {
      const double jb = a.correct[m] ? gamma * a.ws_j[m] : a.ws_j[m];
      var += (jb - mu) * (jb - mu);
    }
    var = warp_sum(var);
    const double sigma = n > 0.0 ? sqrt(var / n) : 0.0;
    for (int m = m0 + lane; m < m1; m += 32) {
      const double jb = a.correct[m] ? gamma * a.ws_j[m] : a.ws_j[m];
      const double ad = eta * (jb - mu) / (sigma + eps);
      a.ws_adv[m] = ad;
      a.Jbar[m] = (float)jb;
      a.adv[m] = (float)ad;
    }
  }
  __syncthreads();
  // ---- decision advantages and the objective terms
  double surr = 0.0, ent = 0.0, kl = 0.0;
  const double ce = (double)a.prm.clip_eps;
  for (int m = m0 + warp; m < m1; m += RL_WARPS) {
    const int r0 = a.round_off[m], r1 = a.round_off[m + 1];
    if (r0 < 0 || r1 < r0 || r1 > a.num_rounds) continue;
    const double adm = a.ws_adv[m], sabs = a.ws_abs[m];
    const bool corr = a.correct[m] != 0;
    for (int r = r0 + lane; r < r1; r += 32) {
      const double rho = (double)a.rho[r];
      for (int i = 0; i < a.K; ++i) {
        const size_t e = (size_t)r * a.K + i;
        if (!a.eff[e]) {
          a.adv_dec[e] = 0.f;
          continue;
        }
        const double A = corr ? rho * adm : (sabs > 0.0 ? fabs((double)a.g[e]) / sabs * adm : 0.0);
        a.adv_dec[e] = (float)A;
        if (a.ratio) {
          const double rt = (double)a.ratio[e];
          const double rc = fmin(fmax(rt, 1.0 - ce), 1.0 + ce);
          surr += fmin(rt * A, rc * A);
          ent += bern_entropy((double)a.p_new[e]);
          kl += bern_kl((double)a.p_new[e], (double)a.p_ref[e]);
        }
      }
    }
  }
  if (a.part) {
    surr = warp_sum(surr);
    ent = warp_sum(ent);
    kl = warp_sum(kl);
    if (lane == 0) {
      red[0][warp] = surr;
      red[1][warp] = ent;
      red[2][warp] = kl;
    }
    __syncthreads();
    if (threadIdx.x < 3) {
      double t = 0.0;
      for (int w = 0; w < RL_WARPS; ++w) t += red[threadIdx.x][w];
      a.part[3 * x + threadIdx.x] = t;
    }
  }
}

// Sum of the per-group partials in a fixed order; loss[3] is the objective.
__global__ void __launch_bounds__(RL_THREADS) rl_loss_kernel(const double* part, int num_groups,
                                                             cospec_rl_params prm, float* loss) {
  __shared__ double acc[3][RL_THREADS];
  double t[3] = {0.0, 0.0, 0.0};
  for (int x = threadIdx.x; x < num_groups; x += RL_THREADS)
    for (int c = 0; c < 3; ++c) t[c] += part[3 * x + c];
  for (int c = 0; c < 3; ++c) acc[c][threadIdx.x] = t[c];
  __syncthreads();
  for (int s = RL_THREADS / 2; s > 0; s >>= 1) {
    if (threadIdx.x < s)
      for (int c = 0; c < 3; ++c) acc[c][threadIdx.x] += acc[c][threadIdx.x + s];
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    loss[0] = (float)acc[0][0];
    loss[1] = (float)acc[1][0];
    loss[2] = (float)acc[2][0];
    loss[3] = (float)(-acc[0][0] - (double)prm.beta_h * acc[1][0] + (double)prm.beta_kl * acc[2][0]);
  }
}

size_t align256(size_t n) { return (n + 255) / 256 * 256; }

}  // namespace

}  // namespace cospec

extern "C" COSPEC_API size_t cospec_rl_workspace(int num_groups, int num_rollouts) {
  using namespace cospec;
  if (num_groups < 0 || num_rollouts < 0) return 0;
  return 3 * align256((size_t)num_rollouts * sizeof(double)) +
         align256((size_t)num_groups * 3 * sizeof(double)) + 256;
}

extern "C" COSPEC_API int cospec_rl_advantages(
    int num_groups, int num_rollouts, int num_rounds, int K, const int32_t* group_off,
    const uint8_t* correct, const int32_t* round_off, const uint8_t* match, const uint8_t* accept,
    const float* ell, const cospec_rl_params* params, const float* ratio, const float* p_new,
    const float* p_ref, float* g, uint8_t* eff, float* rho, float* J, float* Jbar, float* adv,
    float* adv_dec, float* loss, void* ws, size_t ws_bytes, void* stream) {
  using namespace cospec;
  if (num_groups < 0 || num_rollouts < 0 || num_rounds < 0 || K < 1 || K > 64 || !params)
    return COSPEC_ERR_INVALID_ARG;
  const cospec_rl_params& pr = *params;
  const float vals[7] = {pr.alpha, pr.beta, pr.eta_fail, pr.eps, pr.clip_eps, pr.beta_h, pr.beta_kl};
  for (float v : vals)
    if (!isfinite(v)) return COSPEC_ERR_INVALID_ARG;
  if (!(pr.eps > 0.f) || pr.clip_eps < 0.f) return COSPEC_ERR_INVALID_ARG;
  const int have_obj = (ratio != nullptr) + (p_new != nullptr) + (p_ref != nullptr);
  if (have_obj != 0 && have_obj != 3) return COSPEC_ERR_INVALID_ARG;
  if (have_obj == 3 && !loss) return COSPEC_ERR_INVALID_ARG;
  if (!group_off || !round_off) return COSPEC_ERR_INVALID_ARG;
  if (num_rollouts > 0 && (!correct || !J || !Jbar || !adv)) return COSPEC_ERR_INVALID_ARG;
  if (num_rounds > 0 && (!match || !accept || !ell || !g || !eff || !rho || !adv_dec))
    return COSPEC_ERR_INVALID_ARG;
  const size_t need = cospec_rl_workspace(num_groups, num_rollouts);
  if (!ws || ws_bytes < need) return COSPEC_ERR_WORKSPACE;
  int* err = device_error_word();
  if (!err) return cuda_lookup_failed();
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(ws) + 255) & ~uintptr_t(255));
  const size_t mb = align256((size_t)num_rollouts * sizeof(double));
  RLArgs a{};
  a.num_groups = num_groups;
  a.num_rollouts = num_rollouts;
  a.num_rounds = num_rounds;
  a.K = K;
  a.group_off = group_off;
  a.correct = correct;
  a.round_off = round_off;
  a.match = match;
  a.accept = accept;
  a.ell = ell;
  a.prm = pr;
  a.ratio = ratio;
  a.p_new = p_new;
  a.p_ref = p_ref;
  a.g = g;
  a.eff = eff;
  a.rho = rho;
  a.J = J;
  a.Jbar = Jbar;
  a.adv = adv;
  a.adv_dec = adv_dec;
  a.ws_j = reinterpret_cast<double*>(base);
  a.ws_abs = reinterpret_cast<double*>(base + mb);
  a.ws_adv = reinterpret_cast<double*>(base + 2 * mb);
  a.part = have_obj ? reinterpret_cast<double*>(base + 3 * mb) : nullptr;
  a.err = err;
  if (num_groups > 0) {
    rl_group_kernel<<<num_groups, RL_THREADS, 0, st>>>(a);
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_status(e);
  }
  if (have_obj) {
    rl_loss_kernel<<<1, RL_THREADS, 0, st>>>(a.part, num_groups, pr, loss);
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_status(e);
  }
  return COSPEC_OK;
}
