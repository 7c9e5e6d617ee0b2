// Drafter-head update (Sec. 3.4) on the replay buffer of Sec. 3.3.
//
// Rows are the buffer slots (step, sequence, block position); only rows with
// the valid flag (positions up to and including the first reject) count.
// With u = RMSNorm_final(h_k), l = logits^phi, p = softmax(z),
// z = (W^S + gamma A B) u, q = softmax(l / tau), q1 = softmax(l):
//
//  update_prep      UB[n] = B u_n                               (LoRA down)
//  (projection)     Z = U W^S^T + gamma UB A^T                  (EPI_HEAD)
//  update_rowstats  per (vocabulary chunk, row) one pass of max-shifted sums
//                   that merge across chunks; the last chunk of a row gives
//                   its log-normalisers of z, l/tau, l, KL(p||q), KL(p||q1),
//                   H[p], -log p(a), -log p(y*); the last row gives the
//                   schedule's term weights at update t, the loss, the
//                   per-row gradient coefficients, and moves the EMA
//                   baseline b after the loss is formed
//  update_grad_a    per vocabulary entry v, dL/dz_{n,v} from the closed forms
//                     KL:  p (log p - log q - KL)     CE to a: p - [v=a]
//                     -H:  p (log p + H)
//                   then dA[v] = gamma sum_n G[n][v] UB[n] and the optimizer
//                   step on A[v]; partial sums of G A for dB (old A)
//  update_ga_reduce GA[n] = sum over vocabulary tiles (fixed order)
//  update_grad_b    dB[j][c] = gamma sum_n GA[n][j] u_n[c], optimizer step;
//                   its last CTA ends the update (t += 1, empty the buffer)
//
// Full-head mode (W^S itself is trained; LoRA factors, if any, stay frozen)
// replaces grad_a .. grad_b by
//  update_g         G[n][v] = dL/dz_{n,v} (the same closed forms)
//  update_gw        dW[v][c] = sum_n G[n][v] u_n[c] and the optimizer step on
//                   W^S (its f32 master when the weights are bf16; the bf16
//                   rounding is written back for the next drafter passes)
//  update_finish    t += 1, empty the buffer
#include <cmath>

#include "common.cuh"
#include "kernels.h"

namespace dvi {

constexpr int kMaxRank = 64;

enum { RS_LSEZ = 0, RS_LSEQ, RS_LSEQ1, RS_KL, RS_KL1, RS_ENT, RS_NLLA, RS_NLLY, RS_N };
enum { CF_KL = 0, CF_KL1, CF_ENT, CF_A, CF_Y, CF_N };
// dev_state floats: 0 t, 1 b, 2 loss, 3 kl, 4 pg, 5 ce, 6 ent, 7 rl, 8 kl1, 9 accept rate,
// 10 skip flag, 11 adam steps, 12 / 13 Adam's bias-correction denominators 1 - beta^step
enum { DS_T = 0, DS_B, DS_LOSS, DS_KL, DS_PG, DS_CE, DS_ENT, DS_RL, DS_KL1, DS_ACC, DS_SKIP, DS_ADAM, DS_BC1, DS_BC2 };

__device__ __forceinline__ bool row_valid(const UpdateArgs& a, int n) { return a.log_meta[n * 6] != 0; }

// grid (cap, r), 128 threads: CTA (n, j) forms UB[n][j] = B_j . u_n, each
// thread over features tid, tid + 128, ... (all its loads independent), then
// a warp and a block sum in fixed order.
template <typename T>
__global__ void __launch_bounds__(128) update_prep_kernel(const UpdateArgs a) {
  griddep_launch();
  griddep_wait();
  __shared__ float red[4];
  const int n = blockIdx.x, j = blockIdx.y;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (!row_valid(a, n)) {
    if (tid == 0) a.ub[n * a.r + j] = 0.f;
    return;
  }
  const T* u = static_cast<const T*>(a.log_u) + static_cast<size_t>(n) * a.d;
  const float* br = a.lora_b + static_cast<size_t>(j) * a.d;
  float acc = 0.f;
#pragma unroll 16
  for (int c = tid; c < a.d; c += 128) acc = fmaf(br[c], Act<T>::ld(u + c, a.log_plane), acc);
  acc = warp_sum(acc);
  if (lane == 0) red[warp] = acc;
  __syncthreads();
  if (tid == 0) a.ub[n * a.r + j] = (red[0] + red[1]) + (red[2] + red[3]);
}

// (m, s) pairs of log-sum-exp: merge of two partial maxima and sums.
__device__ __forceinline__ void lse_merge(float& m, float& s, float m2, float s2) {
  const float M = fmaxf(m, m2);
  if (M == -INFINITY) return;
  s = (m == -INFINITY ? 0.f : s * expf(m - M)) + (m2 == -INFINITY ? 0.f : s2 * expf(m2 - M));
  m = M;
}
__device__ __forceinline__ void lse_add(float& m, float& s, float x) {
  if (x == -INFINITY) return;
  if (x > m) {
    s = (m == -INFINITY ? 0.f : s * expf(m - x)) + 1.f;
    m = x;
  } else {
    s += expf(x - m);
  }
}

// Weights of the terms at update t (Sec. 3.4's schedule; readings of the
// unnamed constants are the config's).
struct TermW { float kl, pg, ce, ent, rl, beta; };
__device__ TermW term_weights(const dvi_update_config& c, int t) {
  TermW w{0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  if (c.objective == 1) { w.kl = c.lambda0; return w; }
  if (c.objective == 2) { w.rl = 1.f; return w; }
  if (c.objective == 3) { w.pg = 1.f; return w; }
  if (t < c.t_warmup) {
    w.pg = 0.f;
    w.kl = c.lambda0;
  } else if (t < c.t_warmup + c.t_ramp) {
    const float f = static_cast<float>(t - c.t_warmup) / static_cast<float>(c.t_ramp);
    w.pg = f * c.lambda_pg_max;
    w.kl = c.lambda0 - f * (c.lambda0 - c.lambda_kl_min);
  } else {
    w.pg = c.lambda_pg_max;
    w.kl = c.lambda_kl_min;
  }
  w.ce = c.w_ce;
  w.ent = c.w_ent;
  if (t >= c.t_warmup) {
    const float f = c.t_ramp > 0 ? fminf(1.f, static_cast<float>(t - c.t_warmup) / c.t_ramp) : 1.f;
    w.rl = c.w_rl_max * f;
    w.beta = c.beta_min + (c.beta0 - c.beta_min) * expf(-static_cast<float>(t - c.t_warmup) / c.t_beta);
  }
  return w;
}

// The schedule's term weights at update t, the means that form the loss,
// the per-row gradient coefficients, the skip decision and the EMA baseline
// (one thread; reads every row's statistics).
__device__ void coef_body(const UpdateArgs& a) {
  const int t = static_cast<int>(a.dev_state[DS_T]);
  const float b = a.dev_state[DS_B];
  const TermW w = term_weights(a.cfg, t);
  int N = 0, nP = 0;
  float s_kl = 0.f, s_pg = 0.f, s_ce = 0.f, s_ent = 0.f, s_rl = 0.f, s_kl1 = 0.f, s_r = 0.f;
  for (int n = 0; n < a.cap; ++n) {
    if (!row_valid(a, n)) continue;
    const float* rs = a.rowstat + n * RS_N;
    const float r = static_cast<float>(a.log_meta[n * 6 + 2]);
    ++N;
    s_r += r;
    s_kl += rs[RS_KL];
    s_kl1 += rs[RS_KL1];
    s_ce += rs[RS_NLLY];
    s_ent += rs[RS_ENT];
    s_rl += (r - b) * rs[RS_NLLA];
    if (r == 1.f) { ++nP; s_pg += rs[RS_NLLA]; }
  }
  const float fN = N > 0 ? static_cast<float>(N) : 1.f;
  const float kl = N ? s_kl / fN : 0.f, kl1 = N ? s_kl1 / fN : 0.f, ce = N ? s_ce / fN : 0.f;
  const float ent = N ? s_ent / fN : 0.f, rl = N ? s_rl / fN : 0.f, pg = nP ? s_pg / nP : 0.f;
  const float loss = w.kl * kl + w.pg * pg + w.ce * ce - w.ent * ent + w.rl * rl + w.beta * kl1;
  const bool skip = (N == 0) || !isfinite(loss);
  if (N > 0 && !isfinite(loss)) flag_status(a.status, DVI_DEV_NONFINITE);
  a.dev_state[DS_LOSS] = loss;
  a.dev_state[DS_KL] = kl;
  a.dev_state[DS_PG] = pg;
  a.dev_state[DS_CE] = ce;
  a.dev_state[DS_ENT] = ent;
  a.dev_state[DS_RL] = rl;
  a.dev_state[DS_KL1] = kl1;
  a.dev_state[DS_ACC] = N ? s_r / fN : 0.f;
  a.dev_state[DS_SKIP] = skip ? 1.f : 0.f;
  for (int n = 0; n < a.cap; ++n) {
    float* cf = a.coef + n * CF_N;
    if (skip || !row_valid(a, n)) {
      for (int q = 0; q < CF_N; ++q) cf[q] = 0.f;
      continue;
    }
    const float r = static_cast<float>(a.log_meta[n * 6 + 2]);
    cf[CF_KL] = w.kl / fN;
    cf[CF_KL1] = w.beta / fN;
    cf[CF_ENT] = w.ent / fN;
    cf[CF_A] = (r == 1.f && nP ? w.pg / nP : 0.f) + w.rl * (r - b) / fN;
    cf[CF_Y] = w.ce / fN;
  }
  if (!skip) {
    const float rho = a.cfg.baseline_rho;
    a.dev_state[DS_B] = rho * b + (1.f - rho) * (s_r / fN);
    a.dev_state[DS_ADAM] += 1.f;
  }
  // Adam's bias-correction denominators of this step, once for all entries
  const float step = a.dev_state[DS_ADAM];
  a.dev_state[DS_BC1] = 1.f - powf(a.cfg.beta1, step);
  a.dev_state[DS_BC2] = 1.f - powf(a.cfg.beta2, step);
}

// Row statistics in one pass.  With p = softmax(z), q = softmax(l / tau),
// q1 = softmax(l) and a row's log-normalisers lz, lq, lq1:
//   KL(p||q)  = E_p[z] - E_p[l / tau] - lz + lq,   KL(p||q1) = E_p[z] - E_p[l] - lz + lq1,
//   H[p]      = lz - E_p[z],
// so every statistic follows from max-shifted sums that merge across parts of
// the row: (mz, sz = sum e^(z-mz), e^(z-mz) z, e^(z-mz) l/tau, e^(z-mz) l)
// and the (max, sum) pairs of l / tau and l.
enum { PS_MZ = 0, PS_SZ, PS_TZ, PS_TQ, PS_TQ1, PS_MQ, PS_SQ, PS_MQ1, PS_SQ1, PS_N };

// Merge of part `b` into part `a` (both in PS_ layout).
__device__ __forceinline__ void part_merge(float* a, const float* b) {
  const float M = fmaxf(a[PS_MZ], b[PS_MZ]);
  if (M != -INFINITY) {
    const float fa = a[PS_MZ] == -INFINITY ? 0.f : expf(a[PS_MZ] - M);
    const float fb = b[PS_MZ] == -INFINITY ? 0.f : expf(b[PS_MZ] - M);
    a[PS_SZ] = a[PS_SZ] * fa + b[PS_SZ] * fb;
    a[PS_TZ] = a[PS_TZ] * fa + b[PS_TZ] * fb;
    a[PS_TQ] = a[PS_TQ] * fa + b[PS_TQ] * fb;
    a[PS_TQ1] = a[PS_TQ1] * fa + b[PS_TQ1] * fb;
    a[PS_MZ] = M;
  }
  lse_merge(a[PS_MQ], a[PS_SQ], b[PS_MQ], b[PS_SQ]);
  lse_merge(a[PS_MQ1], a[PS_SQ1], b[PS_MQ1], b[PS_SQ1]);
}


constexpr int kStatThreads = 256;
constexpr int kStatPer = 8;                               // vocabulary entries per thread
constexpr int kStatChunk = kStatThreads * kStatPer;       // per CTA

// The merged part of row n over vocabulary chunk c of kStatThreads * PER
// entries (kStatThreads threads of the CTA together; one thread writes
// `out[PS_N]`).
template <int PER>
__device__ void chunk_part(const UpdateArgs& a, int n, int c, float* out, float (*wp)[PS_N]) {
  constexpr int kStatPer = PER;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const float it = 1.f / a.cfg.tau;
  const int i0 = c * kStatThreads * PER + tid * kStatPer;
  const float* z = a.Z + static_cast<size_t>(n) * a.V;
  const float* l = a.log_logits + static_cast<size_t>(n) * a.V;
  float zv[kStatPer], lv[kStatPer];
#pragma unroll
  for (int e = 0; e < kStatPer; ++e) {
    const int i = i0 + e;
    zv[e] = i < a.V ? __ldcg(z + i) : -INFINITY;
    lv[e] = i < a.V ? __ldcg(l + i) : -INFINITY;
  }
  float pt[PS_N];
  float mz = -INFINITY, mq = -INFINITY, mq1 = -INFINITY;
#pragma unroll
  for (int e = 0; e < kStatPer; ++e) {
    mz = fmaxf(mz, zv[e]);
    mq = fmaxf(mq, lv[e] * it);
    mq1 = fmaxf(mq1, lv[e]);
  }
  float sz = 0.f, tz = 0.f, tq = 0.f, tq1 = 0.f, sq = 0.f, sq1 = 0.f;
#pragma unroll
  for (int e = 0; e < kStatPer; ++e) {
    if (zv[e] == -INFINITY) continue;
    const float w = expf(zv[e] - mz);
    sz += w;
    tz = fmaf(w, zv[e], tz);
    tq = fmaf(w, lv[e] * it, tq);
    tq1 = fmaf(w, lv[e], tq1);
    sq += expf(lv[e] * it - mq);
    sq1 += expf(lv[e] - mq1);
  }
  pt[PS_MZ] = mz; pt[PS_SZ] = sz; pt[PS_TZ] = tz; pt[PS_TQ] = tq; pt[PS_TQ1] = tq1;
  pt[PS_MQ] = mq; pt[PS_SQ] = sq; pt[PS_MQ1] = mq1; pt[PS_SQ1] = sq1;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    float other[PS_N];
#pragma unroll
    for (int q = 0; q < PS_N; ++q) other[q] = __shfl_xor_sync(0xffffffffu, pt[q], o);
    // merge in lane order so every lane holds the same, order-fixed result
    if (lane & o) {
      part_merge(other, pt);
#pragma unroll
      for (int q = 0; q < PS_N; ++q) pt[q] = other[q];
    } else {
      part_merge(pt, other);
    }
  }
  if (lane == 0)
#pragma unroll
    for (int q = 0; q < PS_N; ++q) wp[warp][q] = pt[q];
  __syncthreads();
  if (tid == 0) {
    float acc[PS_N];
#pragma unroll
    for (int q = 0; q < PS_N; ++q) acc[q] = wp[0][q];
    for (int w = 1; w < kStatThreads / 32; ++w) part_merge(acc, wp[w]);
#pragma unroll
    for (int q = 0; q < PS_N; ++q) out[q] = acc[q];
  }
  __syncthreads();   // wp is free for the next call
}

// Row n's statistics from its nc chunk parts, merged in chunk order (one
// thread): log-normalisers, KL(p||q), KL(p||q1), H[p], -log p(a), -log p(y*)
// into rs[RS_N] (zeros for a row that is not valid).
__device__ void row_stats(const UpdateArgs& a, int n, int nc, bool valid, float* rs) {
  if (!valid) {
    for (int q = 0; q < RS_N; ++q) rs[q] = 0.f;
    return;
  }
  const float* parts = a.stat_part + static_cast<size_t>(n) * nc * PS_N;
  float acc[PS_N];
#pragma unroll
  for (int q = 0; q < PS_N; ++q) acc[q] = __ldcg(parts + q);
#pragma unroll 8
  for (int k = 1; k < nc; ++k) {
    float b[PS_N];
#pragma unroll
    for (int q = 0; q < PS_N; ++q) b[q] = __ldcg(parts + k * PS_N + q);
    part_merge(acc, b);
  }
  const float lz = acc[PS_MZ] + logf(acc[PS_SZ]);
  const float lq = acc[PS_MQ] + logf(acc[PS_SQ]);
  const float lq1 = acc[PS_MQ1] + logf(acc[PS_SQ1]);
  const float ez = acc[PS_TZ] / acc[PS_SZ];
  const float eq = acc[PS_TQ] / acc[PS_SZ];
  const float eq1 = acc[PS_TQ1] / acc[PS_SZ];
  const int* meta = a.log_meta + n * 6;
  const float* z = a.Z + static_cast<size_t>(n) * a.V;
  rs[RS_LSEZ] = lz;
  rs[RS_LSEQ] = lq;
  rs[RS_LSEQ1] = lq1;
  rs[RS_KL] = (ez - eq) - (lz - lq);
  rs[RS_KL1] = (ez - eq1) - (lz - lq1);
  rs[RS_ENT] = lz - ez;
  rs[RS_NLLA] = lz - __ldcg(z + meta[1]);
  rs[RS_NLLY] = lz - __ldcg(z + meta[5]);
}

// grid (ceil(V / kStatChunk), cap): CTA (c, n) forms the merged part of row n
// over its chunk; the last CTA of a row merges the row's parts in chunk
// order into the row statistics, and the last row to finish forms the loss
// and the per-row coefficients (coef_body).
__global__ void __launch_bounds__(kStatThreads) update_rowstats_kernel(const UpdateArgs a) {
  griddep_launch();
  griddep_wait();
  __shared__ float wp[kStatThreads / 32][PS_N];
  __shared__ int last_chunk, last_row;
  const int c = blockIdx.x, n = blockIdx.y, nc = gridDim.x;
  const int tid = threadIdx.x;
  const bool valid = row_valid(a, n);
  float* parts = a.stat_part + static_cast<size_t>(n) * nc * PS_N;
  if (valid) chunk_part<kStatPer>(a, n, c, parts + c * PS_N, wp);
  // the last chunk of the row merges the row's parts in chunk order
  __threadfence();
  __syncthreads();
  if (tid == 0) last_chunk = atomicAdd(a.ctr + 2 + n, 1) == nc - 1;
  __syncthreads();
  if (!last_chunk) return;
  if (tid == 0) {
    __threadfence();
    a.ctr[2 + n] = 0;
    row_stats(a, n, nc, valid, a.rowstat + n * RS_N);
    // every row's statistics are in place before the last row reads them
    __threadfence();
    last_row = atomicAdd(a.ctr, 1) == static_cast<int>(gridDim.y) - 1;
    if (last_row) {
      __threadfence();
      coef_body(a);
      *a.ctr = 0;
    }
  }
}


// One optimizer step of a parameter; bc1, bc2 = 1 - beta1^step, 1 - beta2^step.
__device__ __forceinline__ void opt_step(const dvi_update_config& c, float bc1, float bc2, float g, float* p,
                                         float* m, float* v) {
  if (c.optimizer == 1) {
    *p -= c.lr * g;
    return;
  }
  const float mn = c.beta1 * *m + (1.f - c.beta1) * g;
  const float vn = c.beta2 * *v + (1.f - c.beta2) * g * g;
  *m = mn;
  *v = vn;
  const float mh = mn / bc1;
  const float vh = vn / bc2;
  *p -= c.lr * mh / (sqrtf(vh) + c.adam_eps);
}

// dL/dz_{n,v} of a valid row n from its row statistics and term coefficients:
//   KL(p||q):  p (log p - log q - KL)      KL(p||q1): p (log p - log q1 - KL1)
//   -H[p]:     p (log p + H)               CE to a / to y*: p - [v = a / y*]
__device__ __forceinline__ float logit_grad(const UpdateArgs& a, int n, int v, float it) {
  const float* rs = a.rowstat + n * RS_N;
  const float* cf = a.coef + n * CF_N;
  const float z = a.Z[static_cast<size_t>(n) * a.V + v];
  const float l = a.log_logits[static_cast<size_t>(n) * a.V + v];
  const float lp = z - rs[RS_LSEZ];
  const float p = expf(lp);
  const float lq = l * it - rs[RS_LSEQ];
  const float lq1 = l - rs[RS_LSEQ1];
  const int* meta = a.log_meta + n * 6;
  return cf[CF_KL] * p * (lp - lq - rs[RS_KL]) + cf[CF_KL1] * p * (lp - lq1 - rs[RS_KL1]) +
         cf[CF_ENT] * p * (lp + rs[RS_ENT]) + cf[CF_A] * (p - (v == meta[1] ? 1.f : 0.f)) +
         cf[CF_Y] * (p - (v == meta[5] ? 1.f : 0.f));
}

// Per-row constants of the logit gradient, staged in shared memory: the
// log-normalisers, KL, KL1, H, the term coefficients, the ids a and y*
// (as floats) and the valid flag.
enum { RW_LZ = 0, RW_LQ, RW_LQ1, RW_KL, RW_KL1, RW_ENT, RW_CKL, RW_CKL1, RW_CENT, RW_CA, RW_CY, RW_A, RW_Y, RW_OK,
       RW_N = 16 };

__device__ __forceinline__ void stage_rows(const UpdateArgs& a, float* rw) {
  for (int n = threadIdx.x; n < a.cap; n += blockDim.x) {
    const float* rs = a.rowstat + n * RS_N;
    const float* cf = a.coef + n * CF_N;
    const int* meta = a.log_meta + n * 6;
    float* o = rw + n * RW_N;
    o[RW_LZ] = rs[RS_LSEZ]; o[RW_LQ] = rs[RS_LSEQ]; o[RW_LQ1] = rs[RS_LSEQ1];
    o[RW_KL] = rs[RS_KL]; o[RW_KL1] = rs[RS_KL1]; o[RW_ENT] = rs[RS_ENT];
    o[RW_CKL] = cf[CF_KL]; o[RW_CKL1] = cf[CF_KL1]; o[RW_CENT] = cf[CF_ENT]; o[RW_CA] = cf[CF_A]; o[RW_CY] = cf[CF_Y];
    o[RW_A] = __int_as_float(meta[1]); o[RW_Y] = __int_as_float(meta[5]); o[RW_OK] = meta[0] != 0 ? 1.f : 0.f;
  }
}

// logit_grad with the row's constants from shared memory (same closed forms).
__device__ __forceinline__ float logit_grad_rw(const float* o, float z, float l, int v, float it) {
  const float lp = z - o[RW_LZ];
  const float p = expf(lp);
  const float lq = l * it - o[RW_LQ];
  const float lq1 = l - o[RW_LQ1];
  return o[RW_CKL] * p * (lp - lq - o[RW_KL]) + o[RW_CKL1] * p * (lp - lq1 - o[RW_KL1]) +
         o[RW_CENT] * p * (lp + o[RW_ENT]) + o[RW_CA] * (p - (v == __float_as_int(o[RW_A]) ? 1.f : 0.f)) +
         o[RW_CY] * (p - (v == __float_as_int(o[RW_Y]) ? 1.f : 0.f));
}

constexpr int kGaBatch = 16;   // buffer rows whose z, l loads are issued together
constexpr size_t kGaSmemMax = 220 * 1024;

// Dynamic shared memory of update_grad_a_kernel, with or without U B^T staged.
__host__ __device__ inline size_t grad_a_smem(const UpdateArgs& a, bool stage_ub) {
  return sizeof(float) * (static_cast<size_t>(a.cap) * 128 + 128 * a.r + static_cast<size_t>(a.cap) * RW_N +
                          (stage_ub ? static_cast<size_t>(a.cap) * a.r : 0));
}

// grid = ceil(V/128); dynamic smem: G tile [cap][128], A tile [128][r], the
// rows' constants [cap][RW_N] and U B^T [cap][r].  R: a bound on the rank
// known at compile time, so the per-thread rows of dA and A stay in
// registers (16 covers the workloads; 64 is the limit).
template <int R>
__global__ void __launch_bounds__(128) update_grad_a_kernel(const UpdateArgs a) {
  griddep_launch();
  griddep_wait();
  extern __shared__ float sm[];
  if (a.dev_state[DS_SKIP] != 0.f) return;
  float* Gs = sm;                                          // [cap][128]
  float* As = Gs + static_cast<size_t>(a.cap) * 128;      // [128][r]
  float* rw = As + 128 * a.r;                              // [cap][RW_N]
  const bool stage_ub = grad_a_smem(a, true) <= kGaSmemMax;
  float* ubs = stage_ub ? rw + static_cast<size_t>(a.cap) * RW_N : a.ub;   // [cap][r]
  const int tid = threadIdx.x;
  const int v = blockIdx.x * 128 + tid;
  const bool ok = v < a.V;
  const float it = 1.f / a.cfg.tau;
  stage_rows(a, rw);
  if (stage_ub)
    for (int i = tid; i < a.cap * a.r; i += 128) ubs[i] = a.ub[i];
  float dA[R];
  float Av[R];
#pragma unroll
  for (int j = 0; j < R; ++j) {
    dA[j] = 0.f;
    Av[j] = (ok && j < a.r) ? a.lora_a[static_cast<size_t>(v) * a.r + j] : 0.f;
    if (j < a.r) As[tid * a.r + j] = Av[j];
  }
  __syncthreads();
  const size_t vv = ok ? static_cast<size_t>(v) : 0;
  for (int n0 = 0; n0 < a.cap; n0 += kGaBatch) {
    float zb[kGaBatch], lb[kGaBatch];
#pragma unroll
    for (int b = 0; b < kGaBatch; ++b) {
      const int n = n0 + b;
      const bool live = ok && n < a.cap && rw[n * RW_N + RW_OK] != 0.f;
      zb[b] = live ? __ldcg(a.Z + static_cast<size_t>(n) * a.V + vv) : 0.f;
      lb[b] = live ? __ldcg(a.log_logits + static_cast<size_t>(n) * a.V + vv) : 0.f;
    }
#pragma unroll
    for (int b = 0; b < kGaBatch; ++b) {
      const int n = n0 + b;
      if (n >= a.cap) break;
      const float* o = rw + n * RW_N;
      float G = 0.f;
      if (ok && o[RW_OK] != 0.f) {
        G = logit_grad_rw(o, zb[b], lb[b], v, it);
        const float* ub = ubs + n * a.r;
#pragma unroll
        for (int j = 0; j < R; ++j)
          if (j < a.r) dA[j] = fmaf(G, ub[j], dA[j]);
      }
      Gs[static_cast<size_t>(n) * 128 + tid] = G;
    }
  }
  __syncthreads();
  // partial G A over this vocabulary tile: pairs (n, j)
  float* part = a.ga_part + static_cast<size_t>(blockIdx.x) * a.cap * a.r;
  for (int idx = tid; idx < a.cap * a.r; idx += 128) {
    const int n = idx / a.r, j = idx % a.r;
    const float* g = Gs + static_cast<size_t>(n) * 128;
    float acc = 0.f;
    for (int q = 0; q < 128; ++q) acc = fmaf(g[q], As[q * a.r + j], acc);
    part[idx] = acc;
  }
  if (!ok) return;
  const float bc1 = a.dev_state[DS_BC1], bc2 = a.dev_state[DS_BC2];
#pragma unroll
  for (int j = 0; j < R; ++j) {
    if (j >= a.r) break;
    const float g = a.gamma * dA[j];
    const size_t i = static_cast<size_t>(v) * a.r + j;
    a.grad_a[i] = g;
    opt_step(a.cfg, bc1, bc2, g, a.lora_a + i, a.m_a + i, a.v_a + i);
  }
}

// GA[n][j] = sum over vocabulary tiles of the partials: 256 threads per row,
// thread (part, j) sums tiles t = part (mod parts), then the parts in order.
__global__ void __launch_bounds__(256) update_ga_reduce_kernel(const UpdateArgs a) {
  griddep_launch();
  griddep_wait();
  __shared__ float ps[256];
  if (a.dev_state[DS_SKIP] != 0.f) return;
  const int n = blockIdx.x, tid = threadIdx.x;
  const int parts = 256 / a.r;
  const int j = tid % a.r, part = tid / a.r;
  float acc = 0.f;
  if (part < parts) {
#pragma unroll 4
    for (int t = part; t < a.n_vtiles; t += parts) acc += a.ga_part[(static_cast<size_t>(t) * a.cap + n) * a.r + j];
  }
  ps[tid] = acc;
  __syncthreads();
  if (tid < a.r) {
    float s = 0.f;
    for (int q = 0; q < parts; ++q) s += ps[q * a.r + tid];
    a.ga[n * a.r + tid] = s;
  }
}

// The update's end: empty the buffer, advance t, count the update unless
// it was skipped.
__device__ __forceinline__ void finish_body(const UpdateArgs& a, int tid, int nthreads) {
  for (int n = tid; n < a.cap; n += nthreads) a.log_meta[n * 6] = 0;
  if (tid == 0) {
    a.dev_state[DS_T] += 1.f;
    *a.log_step = 0;
    if (a.dev_state[DS_SKIP] == 0.f) a.counters[4] += 1;
  }
}

// grid (ceil(d/128), ceil(r/4)): thread c of CTA (x, y) forms dB[j][c] for
// the four j = 4y.. of the CTA (one pass over the buffer rows) and steps
// them; the last CTA to finish then ends the update (finish_body).
template <typename T>
__global__ void __launch_bounds__(128) update_grad_b_kernel(const UpdateArgs a) {
  griddep_launch();
  griddep_wait();
  __shared__ int last;
  __shared__ float gas[kMaxTokens][4];   // G A of the CTA's four j, 0 for rows that are not valid
  __shared__ int okn[kMaxTokens];
  const int c = blockIdx.x * 128 + threadIdx.x;
  const int j0 = blockIdx.y * 4;
  const bool skip = a.dev_state[DS_SKIP] != 0.f;
  if (!skip) {
    for (int i = threadIdx.x; i < a.cap * 4; i += blockDim.x) {
      const int n = i >> 2, q = i & 3;
      gas[n][q] = (j0 + q < a.r && row_valid(a, n)) ? a.ga[n * a.r + j0 + q] : 0.f;
      if (q == 0) okn[n] = row_valid(a, n) ? 1 : 0;
    }
    __syncthreads();
  }
  if (!skip && c < a.d) {
    const float bc1 = a.dev_state[DS_BC1], bc2 = a.dev_state[DS_BC2];
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
    const T* u = static_cast<const T*>(a.log_u) + c;
    // rows that are not valid are not read (their u is whatever the buffer holds)
#pragma unroll 8
    for (int n = 0; n < a.cap; ++n) {
      const float un = okn[n] ? Act<T>::ld(u + static_cast<size_t>(n) * a.d, a.log_plane) : 0.f;
#pragma unroll
      for (int q = 0; q < 4; ++q) acc[q] = fmaf(gas[n][q], un, acc[q]);
    }
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int j = j0 + q;
      if (j >= a.r) break;
      const float g = a.gamma * acc[q];
      const size_t i = static_cast<size_t>(j) * a.d + c;
      a.grad_b[i] = g;
      opt_step(a.cfg, bc1, bc2, g, a.lora_b + i, a.m_b + i, a.v_b + i);
    }
  }
  // every CTA has read the buffer rows' flags before they are cleared
  __syncthreads();
  if (threadIdx.x == 0) last = atomicAdd(a.ctr + 1, 1) == static_cast<int>(gridDim.x * gridDim.y) - 1;
  __syncthreads();
  if (!last) return;
  __threadfence();
  finish_body(a, threadIdx.x, blockDim.x);
  if (threadIdx.x == 0) a.ctr[1] = 0;
}

// ---------------------------------------------------------------- fused LoRA update
// One cooperative launch (every CTA resident, one per SM) runs the whole
// LoRA update on the replay buffer, whose drafter logits z were logged by
// the drafter head when the tuples were drafted (A, B and W^S change only at
// an update, which empties the buffer, so they equal a recomputation), in
// three phases separated by two grid barriers:
//   A  U B^T, and the merged parts of the row statistics per (vocabulary
//      chunk, row)
//   C  every CTA merges every row's parts (chunk order) and forms the loss
//      and the per-row coefficients (the same fixed-order sums in each CTA;
//      CTA 0 publishes them); then per 256-entry vocabulary tile dL/dz,
//      dA = gamma G^T UB with Adam on A, and the CTA's partial of G A over
//      its tiles (old A)
//   E  each CTA sums, over the CTAs' partials, the G A it needs for its
//      share of B's entries, then dB = gamma (G A)^T U and Adam on B; the
//      last CTA out ends the update.
// Each barrier's wait is bounded (one second, then DVI_DEV_TIMEOUT and the
// CTAs wind down).

__device__ __forceinline__ int ld_acquire_i32(const int* p) {
  int v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void st_release_i32(int* p, int v) {
  asm volatile("st.release.gpu.global.b32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

// Grid barrier: bar[0] counts arrivals, bar[1] is the generation, which the
// last CTA to arrive advances after resetting the count.  Thread 0 of each
// CTA keeps the generation it waits for in `gen` and polls with a short
// sleep between reads.
__device__ bool grid_barrier(int* bar, int& gen, int* status, int* ok_s) {
  __syncthreads();
  if (threadIdx.x == 0) {
    int ok = 1;
    const int target = gen + 1;
    __threadfence();
    if (atomicAdd(bar, 1) == static_cast<int>(gridDim.x) - 1) {
      atomicExch(bar, 0);
      __threadfence();
      st_release_i32(bar + 1, target);
    } else {
      const uint64_t t0 = global_ns();
      while (ld_acquire_i32(bar + 1) - target < 0) {
        __nanosleep(64);
        if (global_ns() - t0 > kWaitLimitNs) {
          flag_status(status, DVI_DEV_TIMEOUT);
          ok = 0;
          break;
        }
      }
    }
    __threadfence();
    gen = target;
    *ok_s = ok;
  }
  __syncthreads();
  return *ok_s != 0;
}

constexpr int kFuThreads = 256;
constexpr int kFuPer = 16;         // vocabulary entries per thread in a statistics chunk
constexpr int kFuTile = 256;       // vocabulary entries per grad-A tile (one per thread)
constexpr int kFuRowBlk = 32;      // buffer rows per G tile in shared memory
constexpr int kFuMaxJ = 4;         // rows of B one CTA's share of B's entries may touch

// Dynamic shared memory of the fused update (floats): U B^T [cap][r], the
// rows' constants [cap][RW_N], a G tile [kFuRowBlk][kFuTile], an A tile
// [kFuTile][r], the CTA's partial of G A [cap][r], G A of its B rows
// [cap][kFuMaxJ].
__host__ __device__ inline size_t fused_update_smem(int cap, int r) {
  return sizeof(float) * (static_cast<size_t>(cap) * r * 2 + static_cast<size_t>(cap) * (RW_N + kFuMaxJ) +
                          static_cast<size_t>(kFuRowBlk) * kFuTile + static_cast<size_t>(kFuTile) * r);
}

// Block sum of one value per thread (kFuThreads), in a fixed order.
__device__ __forceinline__ float block_sum(float v, float* red) {
  v = warp_sum(v);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __syncthreads();
  if (lane == 0) red[warp] = v;
  __syncthreads();
  float t = 0.f;
#pragma unroll
  for (int w = 0; w < kFuThreads / 32; ++w) t += red[w];
  return t;
}

// Adam (or SGD) on four consecutive parameters.
__device__ __forceinline__ void opt_step4(const dvi_update_config& c, float bc1, float bc2, const float (&g)[4],
                                          float4* p, float4* m, float4* v) {
  float pv[4] = {p->x, p->y, p->z, p->w};
  if (c.optimizer == 1) {
#pragma unroll
    for (int q = 0; q < 4; ++q) pv[q] -= c.lr * g[q];
  } else {
    float mv[4] = {m->x, m->y, m->z, m->w}, sv[4] = {v->x, v->y, v->z, v->w};
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      mv[q] = c.beta1 * mv[q] + (1.f - c.beta1) * g[q];
      sv[q] = c.beta2 * sv[q] + (1.f - c.beta2) * g[q] * g[q];
      pv[q] -= c.lr * (mv[q] / bc1) / (sqrtf(sv[q] / bc2) + c.adam_eps);
    }
    *m = make_float4(mv[0], mv[1], mv[2], mv[3]);
    *v = make_float4(sv[0], sv[1], sv[2], sv[3]);
  }
  *p = make_float4(pv[0], pv[1], pv[2], pv[3]);
}

template <typename T, int R>
__global__ void __launch_bounds__(kFuThreads, 1) update_fused_kernel(const UpdateArgs a) {
  extern __shared__ float fsm[];
  __shared__ float wp[kFuThreads / 32][PS_N];
  __shared__ float red[kFuThreads / 32];
  __shared__ float sc[4];
  __shared__ int ok_s, last;
  const int tid = threadIdx.x, G = gridDim.x, c = blockIdx.x;
  const int cap = a.cap, r = a.r;
  float* ubs = fsm;                                        // [cap][r]
  float* rw = ubs + cap * r;                               // [cap][RW_N]
  float* Gs = rw + cap * RW_N;                             // [kFuRowBlk][kFuTile]
  float* As = Gs + kFuRowBlk * kFuTile;                    // [kFuTile][r]
  float* gp = As + kFuTile * r;                            // [cap][r] this CTA's partial of G A
  float* gas = gp + cap * r;                               // [cap][kFuMaxJ] G A of this CTA's B rows
  int* bar = a.ctr + 2 + cap;
  int gen = 0;
  if (tid == 0) {
    gen = ld_acquire_i32(bar + 1);
    sc[0] = a.dev_state[DS_T];
    sc[1] = a.dev_state[DS_B];
    sc[2] = a.dev_state[DS_ADAM];
  }
  constexpr int kChunk = kStatThreads * kFuPer;
  const int nc = (a.V + kChunk - 1) / kChunk;

  // ---- A: U B^T (one warp per (row, j) pair) and the parts of the row
  // statistics
  {
    const int warp = tid >> 5, lane = tid & 31;
    const T* U = static_cast<const T*>(a.log_u);
    for (int pq = c * (kFuThreads / 32) + warp; pq < cap * r; pq += G * (kFuThreads / 32)) {
      const int n = pq / r, j = pq % r;
      float acc = 0.f;
      if (row_valid(a, n)) {
        const T* u = U + static_cast<size_t>(n) * a.d;
        const float* br = a.lora_b + static_cast<size_t>(j) * a.d;
#pragma unroll 8
        for (int col = lane; col < a.d; col += 32) acc = fmaf(br[col], Act<T>::ld(u + col, a.log_plane), acc);
        acc = warp_sum(acc);
      }
      if (lane == 0) a.ub[pq] = acc;
    }
  }
  for (int q = c; q < cap * nc; q += G) {
    const int n = q / nc, k = q % nc;
    if (row_valid(a, n)) chunk_part<kFuPer>(a, n, k, a.stat_part + (static_cast<size_t>(n) * nc + k) * PS_N, wp);
  }
  if (!grid_barrier(bar, gen, a.status, &ok_s)) return;

  // ---- C: row statistics, loss and coefficients (every CTA), grad A
  const float b = sc[1];
  float rs[RS_N];
  bool ok_row = false;
  float rr = 0.f;
  if (tid < cap) {
    ok_row = row_valid(a, tid);
    rr = static_cast<float>(a.log_meta[tid * 6 + 2]);
    row_stats(a, tid, nc, ok_row, rs);
    if (c == 0)
      for (int q = 0; q < RS_N; ++q) a.rowstat[tid * RS_N + q] = rs[q];
  }
  float tot[9];
  {
    const bool on = tid < cap && ok_row;
    tot[0] = block_sum(on ? 1.f : 0.f, red);                          // N
    tot[1] = block_sum(on ? rr : 0.f, red);                           // sum r
    tot[2] = block_sum(on ? rs[RS_KL] : 0.f, red);
    tot[3] = block_sum(on ? rs[RS_KL1] : 0.f, red);
    tot[4] = block_sum(on ? rs[RS_NLLY] : 0.f, red);                  // CE to y*
    tot[5] = block_sum(on ? rs[RS_ENT] : 0.f, red);
    tot[6] = block_sum(on ? (rr - b) * rs[RS_NLLA] : 0.f, red);       // REINFORCE
    tot[7] = block_sum(on && rr == 1.f ? 1.f : 0.f, red);             // |P|
    tot[8] = block_sum(on && rr == 1.f ? rs[RS_NLLA] : 0.f, red);     // masked CE
  }
  const TermW w = term_weights(a.cfg, static_cast<int>(sc[0]));
  const float N = tot[0], nP = tot[7];
  const float fN = N > 0.f ? N : 1.f;
  const float kl = N > 0.f ? tot[2] / fN : 0.f, kl1 = N > 0.f ? tot[3] / fN : 0.f;
  const float ce = N > 0.f ? tot[4] / fN : 0.f, ent = N > 0.f ? tot[5] / fN : 0.f;
  const float rl = N > 0.f ? tot[6] / fN : 0.f, pg = nP > 0.f ? tot[8] / nP : 0.f;
  const float loss = w.kl * kl + w.pg * pg + w.ce * ce - w.ent * ent + w.rl * rl + w.beta * kl1;
  const bool skip = (N == 0.f) || !isfinite(loss);
  const float adam = sc[2] + (skip ? 0.f : 1.f);
  const float bc1 = 1.f - powf(a.cfg.beta1, adam), bc2 = 1.f - powf(a.cfg.beta2, adam);
  if (c == 0 && tid == 0) {
    if (N > 0.f && !isfinite(loss)) flag_status(a.status, DVI_DEV_NONFINITE);
    a.dev_state[DS_LOSS] = loss;
    a.dev_state[DS_KL] = kl;
    a.dev_state[DS_PG] = pg;
    a.dev_state[DS_CE] = ce;
    a.dev_state[DS_ENT] = ent;
    a.dev_state[DS_RL] = rl;
    a.dev_state[DS_KL1] = kl1;
    a.dev_state[DS_ACC] = N > 0.f ? tot[1] / fN : 0.f;
    a.dev_state[DS_SKIP] = skip ? 1.f : 0.f;
    if (!skip) a.dev_state[DS_B] = a.cfg.baseline_rho * b + (1.f - a.cfg.baseline_rho) * (tot[1] / fN);
    a.dev_state[DS_ADAM] = adam;
    a.dev_state[DS_BC1] = bc1;
    a.dev_state[DS_BC2] = bc2;
  }
  if (tid < cap) {
    const int n = tid;
    const int* meta = a.log_meta + n * 6;
    const bool ok = !skip && ok_row;
    float cf[CF_N] = {0.f, 0.f, 0.f, 0.f, 0.f};
    if (ok) {
      cf[CF_KL] = w.kl / fN;
      cf[CF_KL1] = w.beta / fN;
      cf[CF_ENT] = w.ent / fN;
      cf[CF_A] = (rr == 1.f && nP > 0.f ? w.pg / nP : 0.f) + w.rl * (rr - b) / fN;
      cf[CF_Y] = w.ce / fN;
    }
    if (c == 0)
      for (int q = 0; q < CF_N; ++q) a.coef[n * CF_N + q] = cf[q];
    float* o = rw + n * RW_N;
    o[RW_LZ] = rs[RS_LSEZ]; o[RW_LQ] = rs[RS_LSEQ]; o[RW_LQ1] = rs[RS_LSEQ1];
    o[RW_KL] = rs[RS_KL]; o[RW_KL1] = rs[RS_KL1]; o[RW_ENT] = rs[RS_ENT];
    o[RW_CKL] = cf[CF_KL]; o[RW_CKL1] = cf[CF_KL1]; o[RW_CENT] = cf[CF_ENT]; o[RW_CA] = cf[CF_A];
    o[RW_CY] = cf[CF_Y];
    o[RW_A] = __int_as_float(meta[1]); o[RW_Y] = __int_as_float(meta[5]); o[RW_OK] = ok ? 1.f : 0.f;
  }
  for (int i = tid; i < cap * r; i += kFuThreads) {
    ubs[i] = a.ub[i];
    gp[i] = 0.f;
  }
  __syncthreads();
  const bool vec4 = (r & 3) == 0 && (reinterpret_cast<uintptr_t>(a.lora_a) & 15u) == 0;
  if (!skip) {
    const float it = 1.f / a.cfg.tau;
    const int n_t = (a.V + kFuTile - 1) / kFuTile;
    for (int t = c; t < n_t; t += G) {
      const int v = t * kFuTile + tid;
      const bool vok = v < a.V;
      const size_t vv = vok ? static_cast<size_t>(v) : 0;
      float dA[R];
#pragma unroll
      for (int j = 0; j < R; ++j) {
        dA[j] = 0.f;
        if (j < r) As[tid * r + j] = vok ? a.lora_a[vv * r + j] : 0.f;
      }
      for (int n0 = 0; n0 < cap; n0 += kFuRowBlk) {
        const int nb = min(kFuRowBlk, cap - n0);
        for (int b0 = 0; b0 < nb; b0 += kGaBatch) {
          float zb[kGaBatch], lb[kGaBatch];
#pragma unroll
          for (int q = 0; q < kGaBatch; ++q) {
            const int n = n0 + b0 + q;
            const bool live = vok && b0 + q < nb && rw[n * RW_N + RW_OK] != 0.f;
            zb[q] = live ? __ldcg(a.Z + static_cast<size_t>(n) * a.V + vv) : 0.f;
            lb[q] = live ? __ldcg(a.log_logits + static_cast<size_t>(n) * a.V + vv) : 0.f;
          }
#pragma unroll
          for (int q = 0; q < kGaBatch; ++q) {
            if (b0 + q >= nb) break;
            const int n = n0 + b0 + q;
            const float* o = rw + n * RW_N;
            float g = 0.f;
            if (vok && o[RW_OK] != 0.f) {
              g = logit_grad_rw(o, zb[q], lb[q], v, it);
              const float* ub = ubs + n * r;
#pragma unroll
              for (int j = 0; j < R; ++j)
                if (j < r) dA[j] = fmaf(g, ub[j], dA[j]);
            }
            Gs[(b0 + q) * kFuTile + tid] = g;
          }
        }
        __syncthreads();
        // this tile's G A for the block's rows, added to the CTA's partial
        for (int idx = tid; idx < nb * r; idx += kFuThreads) {
          const int nn = idx / r, j = idx % r;
          const float* g = Gs + nn * kFuTile;
          float acc = 0.f;
          for (int q = 0; q < kFuTile; ++q) acc = fmaf(g[q], As[q * r + j], acc);
          gp[(n0 + nn) * r + j] += acc;
        }
        __syncthreads();
      }
      if (vok) {
        if (vec4) {
#pragma unroll
          for (int j4 = 0; j4 < R / 4; ++j4) {
            if (4 * j4 >= r) break;
            const size_t i = vv * r + 4 * j4;
            const float g[4] = {a.gamma * dA[4 * j4], a.gamma * dA[4 * j4 + 1], a.gamma * dA[4 * j4 + 2],
                                a.gamma * dA[4 * j4 + 3]};
            *reinterpret_cast<float4*>(a.grad_a + i) = make_float4(g[0], g[1], g[2], g[3]);
            opt_step4(a.cfg, bc1, bc2, g, reinterpret_cast<float4*>(a.lora_a + i),
                      reinterpret_cast<float4*>(a.m_a + i), reinterpret_cast<float4*>(a.v_a + i));
          }
        } else {
#pragma unroll
          for (int j = 0; j < R; ++j) {
            if (j >= r) break;
            const float g = a.gamma * dA[j];
            const size_t i = vv * r + j;
            a.grad_a[i] = g;
            opt_step(a.cfg, bc1, bc2, g, a.lora_a + i, a.m_a + i, a.v_a + i);
          }
        }
      }
      __syncthreads();
    }
    for (int i = tid; i < cap * r; i += kFuThreads) a.ga_part[static_cast<size_t>(c) * cap * r + i] = gp[i];
  }
  if (!grid_barrier(bar, gen, a.status, &ok_s)) return;

  // ---- E: this CTA's share of B's entries [e0, e1): G A of its rows of B
  // (summed over the CTAs' partials in CTA order), dB and Adam on B
  if (!skip) {
    const int total = r * a.d;
    const int per = (total + G - 1) / G;
    const int e0 = c * per, e1 = min(total, e0 + per);
    if (e0 < e1) {
      const int j_lo = e0 / a.d, nj = (e1 - 1) / a.d - j_lo + 1;   // <= kFuMaxJ (checked at launch)
      // 16 threads per (n, j) pair, each over every 16th CTA partial (all of
      // its loads issued together), then a fixed-order butterfly across the 16
      const int pairs = cap * nj;
      for (int p0 = 0; p0 < pairs; p0 += kFuThreads / 16) {
        const int p = p0 + tid / 16, sub = tid & 15;
        float xs[kFuThreads / 16];
        const int n = p / nj, j = j_lo + p % nj;
#pragma unroll
        for (int m = 0; m < kFuThreads / 16; ++m) {
          const int k = sub + 16 * m;
          xs[m] = (p < pairs && k < G) ? __ldcg(a.ga_part + (static_cast<size_t>(k) * cap + n) * r + j) : 0.f;
        }
        float x = 0.f;
#pragma unroll
        for (int m = 0; m < kFuThreads / 16; ++m) x += xs[m];
        x += __shfl_xor_sync(0xffffffffu, x, 1);
        x += __shfl_xor_sync(0xffffffffu, x, 2);
        x += __shfl_xor_sync(0xffffffffu, x, 4);
        x += __shfl_xor_sync(0xffffffffu, x, 8);
        if (p < pairs && sub == 0) gas[n * kFuMaxJ + p % nj] = x;
      }
      __syncthreads();
      const T* U = static_cast<const T*>(a.log_u);
      // a thread's entries e0 + tid, e0 + tid + 256, ...: two at a time, so
      // the loads of both rows of U go out together
      for (int e = e0 + tid; e < e1; e += 2 * kFuThreads) {
        const int e2 = e + kFuThreads;
        const bool two = e2 < e1;
        const int ja = e / a.d, ca = e - ja * a.d;
        const int jb = two ? e2 / a.d : ja, cb = two ? e2 - jb * a.d : ca;
        float acc_a = 0.f, acc_b = 0.f;
#pragma unroll 8
        for (int n = 0; n < cap; ++n) {
          const bool on = rw[n * RW_N + RW_OK] != 0.f;
          const T* un = U + static_cast<size_t>(n) * a.d;
          const float ua = on ? Act<T>::ld(un + ca, a.log_plane) : 0.f;
          const float ub = on && two ? Act<T>::ld(un + cb, a.log_plane) : 0.f;
          acc_a = fmaf(gas[n * kFuMaxJ + (ja - j_lo)], ua, acc_a);
          acc_b = fmaf(gas[n * kFuMaxJ + (jb - j_lo)], ub, acc_b);
        }
        const float ga = a.gamma * acc_a;
        a.grad_b[e] = ga;
        opt_step(a.cfg, bc1, bc2, ga, a.lora_b + e, a.m_b + e, a.v_b + e);
        if (two) {
          const float gb = a.gamma * acc_b;
          a.grad_b[e2] = gb;
          opt_step(a.cfg, bc1, bc2, gb, a.lora_b + e2, a.m_b + e2, a.v_b + e2);
        }
      }
    }
  }
  // the update's end, by the last CTA out (every CTA has read the rows' flags)
  __syncthreads();
  if (tid == 0) last = atomicAdd(a.ctr + 1, 1) == G - 1;
  __syncthreads();
  if (!last) return;
  __threadfence();
  finish_body(a, tid, kFuThreads);
  if (tid == 0) a.ctr[1] = 0;
}

// ---------------------------------------------------------------- full-head mode

// G[n][v] for every buffer row (zeros for rows that are not valid).
// grid = (ceil(V/256), cap), 256 threads.
__global__ void __launch_bounds__(256) update_g_kernel(const UpdateArgs a) {
  griddep_launch();
  griddep_wait();
  if (a.dev_state[DS_SKIP] != 0.f) return;
  const int n = blockIdx.y;
  const int v = blockIdx.x * 256 + threadIdx.x;
  if (v >= a.V) return;
  a.G[static_cast<size_t>(n) * a.V + v] = row_valid(a, n) ? logit_grad(a, n, v, 1.f / a.cfg.tau) : 0.f;
}

constexpr int kGwRows = 16;    // W^S rows per CTA (accumulators per thread: kGwRows x 4)
constexpr int kGwCols = 512;   // W^S columns per CTA: 128 threads x 4 consecutive columns
constexpr int kGwStage = 16;   // buffer rows staged in shared memory per round

// dW = G^T U for a [kGwRows x kGwCols] tile of W^S, then the optimizer step
// on it.  The contraction runs over the buffer rows (N <= 256), so it is a
// few FMAs per W^S entry; the kernel streams W^S (master), m and v once.
// grid = (ceil(V / kGwRows), ceil(d / kGwCols)), 128 threads.
template <typename T>
__global__ void __launch_bounds__(128) update_gw_kernel(const UpdateArgs a) {
  griddep_launch();
  griddep_wait();
  if (a.dev_state[DS_SKIP] != 0.f) return;
  __shared__ float4 us[kGwStage][kGwCols / 4];
  __shared__ float gs[kGwStage][kGwRows];
  const int tid = threadIdx.x;
  const int v0 = blockIdx.x * kGwRows;
  const int cb = blockIdx.y * kGwCols;
  const int c = cb + tid * 4;
  float4 acc[kGwRows];
#pragma unroll
  for (int i = 0; i < kGwRows; ++i) acc[i] = make_float4(0.f, 0.f, 0.f, 0.f);
  const T* U = static_cast<const T*>(a.log_u);
  for (int n0 = 0; n0 < a.cap; n0 += kGwStage) {
    __syncthreads();
    for (int i = tid; i < kGwStage * (kGwCols / 4); i += 128) {
      const int row = i / (kGwCols / 4), col = cb + (i % (kGwCols / 4)) * 4;
      const int n = n0 + row;
      float4 u = make_float4(0.f, 0.f, 0.f, 0.f);
      if (n < a.cap && col < a.d && row_valid(a, n)) {
        const T* src = U + static_cast<size_t>(n) * a.d + col;
        const size_t pl = a.log_plane;
        u = make_float4(Act<T>::ld(src, pl), Act<T>::ld(src + 1, pl), Act<T>::ld(src + 2, pl),
                        Act<T>::ld(src + 3, pl));
      }
      us[row][i % (kGwCols / 4)] = u;
    }
    for (int i = tid; i < kGwStage * kGwRows; i += 128) {
      const int row = i / kGwRows, vv = i % kGwRows;
      const int n = n0 + row, v = v0 + vv;
      gs[row][vv] = (n < a.cap && v < a.V) ? a.G[static_cast<size_t>(n) * a.V + v] : 0.f;
    }
    __syncthreads();
    const int rows = min(kGwStage, a.cap - n0);
    for (int row = 0; row < rows; ++row) {
      const float4 u = us[row][tid];
#pragma unroll
      for (int vv = 0; vv < kGwRows; ++vv) {
        const float g = gs[row][vv];
        acc[vv].x = fmaf(g, u.x, acc[vv].x);
        acc[vv].y = fmaf(g, u.y, acc[vv].y);
        acc[vv].z = fmaf(g, u.z, acc[vv].z);
        acc[vv].w = fmaf(g, u.w, acc[vv].w);
      }
    }
  }
  if (c >= a.d) return;
  const dvi_update_config& cf = a.cfg;
  const float bc1 = a.dev_state[DS_BC1], bc2 = a.dev_state[DS_BC2];
  float* master = a.w_master ? a.w_master : static_cast<float*>(a.w_head);
  // four rows at a time: their loads are issued before any store
#pragma unroll
  for (int g0 = 0; g0 < kGwRows; g0 += 4) {
    float4 p[4], m[4], s[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int v = v0 + g0 + j;
      if (v >= a.V) continue;
      const size_t i = static_cast<size_t>(v) * a.d + c;
      p[j] = *reinterpret_cast<const float4*>(master + i);
      if (cf.optimizer == 0) {
        m[j] = *reinterpret_cast<const float4*>(a.m_w + i);
        s[j] = *reinterpret_cast<const float4*>(a.v_w + i);
      }
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int v = v0 + g0 + j;
      if (v >= a.V) continue;
      const size_t i = static_cast<size_t>(v) * a.d + c;
      const float4 g = acc[g0 + j];
      if (a.keep_grad_w) *reinterpret_cast<float4*>(a.grad_w + i) = g;
      float gv[4] = {g.x, g.y, g.z, g.w};
      float pv[4] = {p[j].x, p[j].y, p[j].z, p[j].w};
      if (cf.optimizer == 1) {
#pragma unroll
        for (int q = 0; q < 4; ++q) pv[q] -= cf.lr * gv[q];
      } else {
        float mv[4] = {m[j].x, m[j].y, m[j].z, m[j].w};
        float sv[4] = {s[j].x, s[j].y, s[j].z, s[j].w};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          mv[q] = cf.beta1 * mv[q] + (1.f - cf.beta1) * gv[q];
          sv[q] = cf.beta2 * sv[q] + (1.f - cf.beta2) * gv[q] * gv[q];
          pv[q] -= cf.lr * (mv[q] / bc1) / (sqrtf(sv[q] / bc2) + cf.adam_eps);
        }
        *reinterpret_cast<float4*>(a.m_w + i) = make_float4(mv[0], mv[1], mv[2], mv[3]);
        *reinterpret_cast<float4*>(a.v_w + i) = make_float4(sv[0], sv[1], sv[2], sv[3]);
      }
      *reinterpret_cast<float4*>(master + i) = make_float4(pv[0], pv[1], pv[2], pv[3]);
      if (a.w_master) {
        uint2 packed;
        packed.x = pack_bf16x2(pv[0], pv[1]);
        packed.y = pack_bf16x2(pv[2], pv[3]);
        *reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(a.w_head) + i) = packed;
      }
    }
  }
}

// master[i] = W^S[i] (bf16 -> f32), once at context creation.
__global__ void update_master_init_kernel(const __nv_bfloat16* w, float* master, size_t n) {
  for (size_t i = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x; i < n;
       i += static_cast<size_t>(gridDim.x) * blockDim.x)
    master[i] = __bfloat162float(w[i]);
}

__global__ void update_finish_kernel(const UpdateArgs a) {
  griddep_launch();
  griddep_wait();
  finish_body(a, threadIdx.x, blockDim.x);
}

cudaError_t launch_update_prep(const UpdateArgs& a, cudaStream_t s) {
  if (a.r == 0) return cudaSuccess;
  const dim3 grid(a.cap, a.r);
  const cudaError_t e = a.dtype == DVI_BF16 ? launch_pdl(update_prep_kernel<__nv_bfloat16>, grid, dim3(128), 0, s, a)
                                            : launch_pdl(update_prep_kernel<float>, grid, dim3(128), 0, s, a);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}
cudaError_t launch_update_rowstats(const UpdateArgs& a, cudaStream_t s) {
  const dim3 grid((a.V + kStatChunk - 1) / kStatChunk, a.cap);
  const cudaError_t e = launch_pdl(update_rowstats_kernel, grid, dim3(kStatThreads), 0, s, a);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}
cudaError_t launch_update_grad_a(const UpdateArgs& a, cudaStream_t s) {
  if (a.r == 0) return cudaSuccess;
  const size_t full = grad_a_smem(a, true);
  const size_t smem = full <= kGaSmemMax ? full : grad_a_smem(a, false);
  auto kern = a.r <= 16 ? update_grad_a_kernel<16> : update_grad_a_kernel<kMaxRank>;
  // set on every call above 48 KiB (once per update; the attribute is per
  // device, and this keeps it right on whichever device is current)
  if (smem > 48 * 1024)
    cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  const cudaError_t e = launch_pdl(kern, dim3(a.n_vtiles), dim3(128), smem, s, a);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}
cudaError_t launch_update_grad_b(const UpdateArgs& a, cudaStream_t s) {
  if (a.r == 0) return cudaSuccess;
  cudaError_t e = launch_pdl(update_ga_reduce_kernel, dim3(a.cap), dim3(256), 0, s, a);
  if (e != cudaSuccess) return e;
  const dim3 grid((a.d + 127) / 128, (a.r + 3) / 4);
  e = a.dtype == DVI_BF16 ? launch_pdl(update_grad_b_kernel<__nv_bfloat16>, grid, dim3(128), 0, s, a)
                          : launch_pdl(update_grad_b_kernel<float>, grid, dim3(128), 0, s, a);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}
bool update_fused_ok(const UpdateArgs& a, int n_sms) {
  if (a.r <= 0 || a.r > kMaxRank || n_sms < 1 || a.cap > kFuThreads) return false;
  if (fused_update_smem(a.cap, a.r) > 200 * 1024) return false;
  // a CTA's share of B's entries must touch at most kFuMaxJ rows of B
  const int per = (a.r * a.d + n_sms - 1) / n_sms;
  return per / a.d + 2 <= kFuMaxJ;
}

cudaError_t launch_update_fused(const UpdateArgs& a, int n_sms, cudaStream_t s) {
  const size_t smem = fused_update_smem(a.cap, a.r);
  void (*kern)(const UpdateArgs);
  if (a.dtype == DVI_BF16) kern = a.r <= 16 ? update_fused_kernel<__nv_bfloat16, 16> : update_fused_kernel<__nv_bfloat16, kMaxRank>;
  else kern = a.r <= 16 ? update_fused_kernel<float, 16> : update_fused_kernel<float, kMaxRank>;
  if (smem > 48 * 1024) {
    const cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    if (e != cudaSuccess) return e;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(n_sms);
  cfg.blockDim = dim3(kFuThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeCooperative;   // every CTA resident: the grid barriers need it
  at[0].val.cooperative = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, kern, a);
  return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t launch_update_full(const UpdateArgs& a, cudaStream_t s) {
  cudaError_t e = launch_pdl(update_g_kernel, dim3((a.V + 255) / 256, a.cap), dim3(256), 0, s, a);
  if (e != cudaSuccess) return e;
  const dim3 grid((a.V + kGwRows - 1) / kGwRows, (a.d + kGwCols - 1) / kGwCols);
  e = a.dtype == DVI_BF16 ? launch_pdl(update_gw_kernel<__nv_bfloat16>, grid, dim3(128), 0, s, a)
                          : launch_pdl(update_gw_kernel<float>, grid, dim3(128), 0, s, a);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}
cudaError_t launch_master_init(const void* w_bf16, float* master, size_t n, cudaStream_t s) {
  update_master_init_kernel<<<1024, 256, 0, s>>>(static_cast<const __nv_bfloat16*>(w_bf16), master, n);
  return cudaGetLastError();
}
cudaError_t launch_update_finish(const UpdateArgs& a, cudaStream_t s) {
  const cudaError_t e = launch_pdl(update_finish_kernel, dim3(1), dim3(256), 0, s, a);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace dvi
