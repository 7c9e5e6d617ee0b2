// Projection kernels of the split decoder (Sec. 3.1's f_{0->k}, f_{k->L} and
// both heads): Y[tok][f] = sum_k W[f][k] * B[tok][k] for a few token rows.
//
// Decode passes carry 1..256 token rows against weight matrices of up to
// 32000 x 11008, so every launch is a weight stream: each tile of 128 output
// features (the tcgen05 M dimension) is read from HBM exactly once, and the
// token rows sit on the MMA's N dimension ("swap AB").
//
// bf16 (tcgen05): warp 4 streams the 128x64 weight tile and the matching
// activation tiles of each K block by TMA (128-byte swizzle, the K-major
// layout tcgen05 reads) into a ring of shared-memory stages; warp 5 issues
// tcgen05.mma (M=128, N=n_pad, K=16) into a TMEM accumulator and frees
// stages with tcgen05.commit; warps 0-3 then read TMEM and run the fused
// epilogue.  Activations are bf16 pairs hi + lo (two planes of the
// activation buffer) whose rows sit next to each other in a stage, so each
// K step's MMA (N = 2 n_pad) writes W.hi to accumulator columns [0, n_pad)
// and W.lo to [n_pad, 2 n_pad); the epilogue adds the two, and the product
// carries the rounding of the weights only.  A gate/up tile holds 64 rows of W_gate and the same 64 rows of
// W_up (two 64-row TMA boxes), so SwiGLU pairs rows r and r+64 of one tile.
// The RMSNorm feeding a projection is split in two: its gain is folded into
// the activation rows by the kernel that produced them, and its 1/rms (a
// per-row scalar) multiplies the accumulators in the epilogue.
// Launches use programmatic dependent launch: the weight tiles of the first
// stages (which no earlier kernel writes) stream in before the kernel waits
// for its predecessor.
//
// f32 (FP32 FMA, no TF32): the same decomposition with a shared-memory tiled
// FFMA main loop of 16 token columns per CTA.
//
// K is split over `n_splits` CTAs per tile when there are too few tiles to
// fill the GPU.  bf16: the splits of a tile form one thread-block cluster;
// each leaves its partial tile in shared memory and, after a cluster barrier,
// rank r sums the partials of all ranks in rank order through distributed
// shared memory for the token columns n = r (mod n_splits) and runs their
// epilogue.  f32: each split stores its partial in
// global scratch and the last CTA to arrive (an atomic counter per tile) sums
// them in split order.  Both are deterministic, and the split plan depends on
// the weight shape only (never on the number of decode rows).
#include <algorithm>
#include <cudaTypedefs.h>

#include "common.cuh"
#include "kernels.h"

namespace dvi {

constexpr int kGuRows = 64;   // features per gate/up tile (64 gate rows + 64 up rows)

struct EpiSmem {
  float stage[kTileRows][kChunk + 1];
  float red[4][kChunk];
  unsigned long long redk[4][kChunk];
  int flag;
};

__device__ __forceinline__ void row_seq_pos(const ProjArgs& p, int n, int& seq, int& pos) {
  seq = p.seq0 + n / p.rows_per_seq;
  pos = p.lens[seq] + p.pos_off + n % p.rows_per_seq;
}

// rstd[n] for the token rows of the launch (1 when there is no norm), and
// for the QKV flavour the cache position of every row.
__device__ __forceinline__ void compute_rstd(const ProjArgs& p, float* rstd, int* posn, int tid, int nthreads) {
  for (int n = tid; n < p.M; n += nthreads) {
    float r = 1.f;
    if (p.ss) {
      float s = 0.f;
      for (int t = 0; t < p.ss_tiles; ++t) s += p.ss[static_cast<size_t>(t) * p.ss_ld + n];
      r = rsqrtf(s / static_cast<float>(p.d_norm) + p.eps);
    }
    rstd[n] = r;
    if (p.flavor == EPI_QKV) {
      int seq, pos;
      row_seq_pos(p, n, seq, pos);
      posn[n] = pos;
    }
  }
}

// Token columns [c0, c0+16) that hold rows of the launch.
__device__ __forceinline__ uint32_t valid_cols(const ProjArgs& p, int c0) {
  const int n = min(kChunk, p.M - c0);
  return n >= kChunk ? 0xffffu : ((1u << max(n, 0)) - 1u);
}

// Fused epilogue for the token columns of [c0, c0+16) set in `own` (a
// subset of the valid ones) of one 128-feature tile.  Called by the 128
// epilogue threads together (row = feature within tile).
template <typename T>
__device__ __forceinline__ void epilogue_chunk(const ProjArgs& p, int tile, int row, int c0, float (&v)[kChunk],
                               const float* rstd, const int* posn, EpiSmem& es, uint32_t own) {
  const int warp = row >> 5, lane = row & 31;
  if (p.ss) {
#pragma unroll
    for (int j = 0; j < kChunk; ++j) v[j] *= ((own >> j) & 1u) ? rstd[c0 + j] : 0.f;
  }
  if (p.flavor == EPI_QKV) {
    const int tq = p.rows_q / kTileRows, tk = p.rows_k / kTileRows;
    int sec, lt;
    if (tile < tq) { sec = 0; lt = tile; }
    else if (tile < tq + tk) { sec = 1; lt = tile - tq; }
    else { sec = 2; lt = tile - tq - tk; }
    const int f = lt * kTileRows + row;
    const int hd = p.head_dim, half = hd >> 1;
    const int head = f / hd, dim = f % hd;
    if (sec < 2) {
#pragma unroll
      for (int j = 0; j < kChunk; ++j) es.stage[row][j] = v[j];
      named_bar(1, kTileRows);
    }
    const int prow = row + (dim < half ? half : -half);
#pragma unroll
    for (int j = 0; j < kChunk; ++j) {
      const int n = c0 + j;
      if ((own >> j) & 1u) {
        const int seq = p.seq0 + n / p.rows_per_seq;
        const int pos = posn[n];
        if (pos >= p.max_len || pos < 0) {
          flag_status(p.status, DVI_DEV_KV_FULL);
        } else {
          float val = v[j];
          if (sec < 2) {
            const float vp = es.stage[prow][j];
            const float2 cs = p.rope[static_cast<size_t>(pos) * half + (dim % half)];
            val = dim < half ? val * cs.x - vp * cs.y : val * cs.x + vp * cs.y;
          }
          if (sec == 0) {
            p.q_out[static_cast<size_t>(n) * p.ld_q + f] = val;
          } else {
            T* c = static_cast<T*>(sec == 1 ? p.kc : p.vc);
            DT<T>::st(c + ((static_cast<size_t>(seq) * p.n_kv_heads + head) * p.max_len + pos) * hd + dim, val);
          }
        }
      }
    }
    if (sec < 2) named_bar(1, kTileRows);
  } else if (p.flavor == EPI_RESID) {
    const int f = tile * kTileRows + row;
    const float g = (p.xg_out && f < p.n_out) ? p.g_next[f] : 0.f;
    float sq[kChunk];
#pragma unroll
    for (int j = 0; j < kChunk; ++j) {
      const int n = c0 + j;
      float xn = 0.f;
      if (((own >> j) & 1u) && f < p.n_out) {
        float* xp = p.x_res + static_cast<size_t>(n) * p.ld_res + f;
        xn = *xp + v[j];
        *xp = xn;
        if (p.xg_out) Act<T>::st(static_cast<T*>(p.xg_out) + static_cast<size_t>(n) * p.ld_xg + f, p.xg_plane, xn * g);
      }
      sq[j] = xn * xn;
    }
#pragma unroll
    for (int j = 0; j < kChunk; ++j) {
      const float s = warp_sum(sq[j]);
      if (lane == 0) es.red[warp][j] = s;
    }
    named_bar(1, kTileRows);
    if (row < kChunk && ((own >> row) & 1u))
      p.ss_out[static_cast<size_t>(tile) * p.ss_out_ld + c0 + row] =
          (es.red[0][row] + es.red[1][row]) + (es.red[2][row] + es.red[3][row]);
    named_bar(1, kTileRows);
  } else if (p.flavor == EPI_GATEUP) {
    // rows 0..63: W_gate, rows 64..127: W_up, same 64 features
#pragma unroll
    for (int j = 0; j < kChunk; ++j) es.stage[row][j] = v[j];
    named_bar(1, kTileRows);
    const int f = tile * kGuRows + row;
    if (row < kGuRows && f < p.n_out) {
#pragma unroll
      for (int j = 0; j < kChunk; ++j) {
        const int n = c0 + j;
        if ((own >> j) & 1u) {
          const float gt = es.stage[row][j];
          const float h = gt / (1.f + expf(-gt)) * es.stage[row + kGuRows][j];
          Act<T>::st(static_cast<T*>(p.h_out) + static_cast<size_t>(n) * p.ld_h + f, p.h_plane, h);
        }
      }
    }
    named_bar(1, kTileRows);
  } else {  // EPI_HEAD
    const int f = tile * kTileRows + row;
    const bool ok = f < p.n_out;
    float z[kChunk];
#pragma unroll
    for (int j = 0; j < kChunk; ++j) z[j] = v[j];
    if (p.lora_r > 0 && ok) {
      const float* arow = p.lora_a + static_cast<size_t>(f) * p.lora_r;
      for (int j = 0; j < kChunk; ++j) {
        const int n = c0 + j;
        if ((own >> j) & 1u) {
          const float* bu = p.lora_bu + static_cast<size_t>(n) * p.lora_r;
          float acc = 0.f;
          for (int q = 0; q < p.lora_r; ++q) acc = fmaf(arow[q], bu[q], acc);
          z[j] = fmaf(p.gamma, acc, z[j]);
        }
      }
    }
    if (p.logits_mode != 0 && ok) {
      float* dst = nullptr;
      if (p.logits_mode == 1) {
        dst = p.logits_out;
      } else {
        const int ls = *p.log_step;
        if (ls < p.log_cap_steps)
          dst = p.logits_out + static_cast<size_t>(ls) * p.log_rows_per_step * p.ld_logits;
      }
      if (dst) {
#pragma unroll
        for (int j = 0; j < kChunk; ++j) {
          int row = c0 + j;
          if (p.logits_mode == 2) {   // replay-buffer slot of (sequence, block row)
            const int i = row % p.log_src_rows;
            row = i < p.log_dst_rows ? row / p.log_src_rows * p.log_dst_rows + i : -1;
          }
          if (((own >> j) & 1u) && row >= 0) dst[static_cast<size_t>(row) * p.ld_logits + f] = z[j];
        }
      }
    }
    if (p.amax) {
#pragma unroll
      for (int j = 0; j < kChunk; ++j) {
        unsigned long long key = 0;
        if (ok && ((own >> j) & 1u)) {
          if (isfinite(z[j])) key = argmax_key(z[j], f);
          else flag_status(p.status, DVI_DEV_NONFINITE);
        }
        key = warp_max_u64(key);
        if (lane == 0) es.redk[warp][j] = key;
      }
      named_bar(1, kTileRows);
      if (row < kChunk && ((own >> row) & 1u)) {
        unsigned long long k0 = es.redk[0][row], k1 = es.redk[1][row];
        unsigned long long k2 = es.redk[2][row], k3 = es.redk[3][row];
        k0 = k0 > k1 ? k0 : k1;
        k2 = k2 > k3 ? k2 : k3;
        atomicMax(p.amax + c0 + row, k0 > k2 ? k0 : k2);
      }
      named_bar(1, kTileRows);
    }
  }
}

// Split-K arrival: returns true in the CTA that must reduce tile `ci`.
__device__ __forceinline__ bool split_arrive(const ProjArgs& p, int ci, int row, EpiSmem& es) {
  __threadfence();
  named_bar(1, kTileRows);
  if (row == 0) {
    const int old = atomicAdd(p.counters + ci, 1);
    es.flag = (old == p.n_splits - 1);
  }
  named_bar(1, kTileRows);
  const bool last = es.flag != 0;
  if (last) {
    __threadfence();
    if (row == 0) p.counters[ci] = 0;
  }
  return last;
}

// Sum of the split partials of one element, in split order; the loads of up
// to eight splits are issued before their sum so their latencies overlap.
__device__ __forceinline__ float sum_splits(const float* base, size_t stride, int n_splits) {
  float a = 0.f;
  for (int s0 = 0; s0 < n_splits; s0 += 8) {
    float t[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) t[u] = (s0 + u < n_splits) ? __ldcg(base + (s0 + u) * stride) : 0.f;
#pragma unroll
    for (int u = 0; u < 8; ++u)
      if (s0 + u < n_splits) a += t[u];
  }
  return a;
}

__device__ __forceinline__ uint32_t tmem_cols(int n) {
  uint32_t c = 32;
  while (c < static_cast<uint32_t>(n)) c <<= 1;
  return c;
}

// Writes one 64-wide K block of the B operand from float32 rows (B_SOFT_F32):
// the hi rows, then n_pad rows further the lo rows.
__device__ __forceinline__ void produce_b_f32(const ProjArgs& p, uint8_t* bs, int kb, int tid) {
  const int nslots = p.n_pad * 8;
  for (int slot = tid; slot < nslots; slot += kTileRows) {
    const int n = slot >> 3, c = slot & 7;
    const int k0 = kb * kKBlock + c * 8;
    uint4 val = make_uint4(0u, 0u, 0u, 0u), lo = val;
    if (n < p.M && k0 < p.K) {
      const float* src = static_cast<const float*>(p.act) + static_cast<size_t>(p.act_row0 + n) * p.ld_act + k0;
      float f[8];
      if (k0 + 8 <= p.K) {
        const float4 a = *reinterpret_cast<const float4*>(src);
        const float4 b = *reinterpret_cast<const float4*>(src + 4);
        f[0] = a.x; f[1] = a.y; f[2] = a.z; f[3] = a.w; f[4] = b.x; f[5] = b.y; f[6] = b.z; f[7] = b.w;
      } else {
#pragma unroll
        for (int e = 0; e < 8; ++e) f[e] = (k0 + e < p.K) ? src[e] : 0.f;
      }
      split_bf16x2(f[0], f[1], val.x, lo.x);
      split_bf16x2(f[2], f[3], val.y, lo.y);
      split_bf16x2(f[4], f[5], val.z, lo.z);
      split_bf16x2(f[6], f[7], val.w, lo.w);
    }
    *reinterpret_cast<uint4*>(bs + n * 128 + ((c ^ (n & 7)) << 4)) = val;
    const int nl = n + p.n_pad;
    *reinterpret_cast<uint4*>(bs + nl * 128 + ((c ^ (nl & 7)) << 4)) = lo;
  }
}

// ------------------------------------------------------------------ tcgen05
// kSplit: the launch splits K over a cluster (n_splits > 1); the unsplit
// instantiation carries no cluster code.
template <bool kSplit>
__global__ void __launch_bounds__(192, 2)
    proj_tc_kernel(const __grid_constant__ CUtensorMap m0, const __grid_constant__ CUtensorMap m1,
                   const __grid_constant__ CUtensorMap m2, const __grid_constant__ CUtensorMap mb,
                   const ProjArgs p, int stages) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  uint8_t* base = smem_raw + (((raw + 1023u) & ~1023u) - raw);
  constexpr int abytes = 16384;
  const int bbytes = 2 * p.n_pad * 128;   // hi rows, then lo rows
  uint8_t* sA = base;
  uint8_t* sB = base + stages * abytes;
  uint64_t* full = reinterpret_cast<uint64_t*>(sB + stages * bbytes);
  uint64_t* empty = full + stages;
  uint64_t* done = empty + stages;
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(done + 1);
  float* rstd = reinterpret_cast<float*>(tmem_holder + 4);
  int* posn = reinterpret_cast<int*>(rstd + kMaxTokens);

  // after `done` the A stages are free: epilogue scratch, then this split's
  // partial tile [n_pad][128] for the cluster reduction
  EpiSmem& es = *reinterpret_cast<EpiSmem*>(sA);
  float* part = reinterpret_cast<float*>(sA + abytes);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int tile = blockIdx.x / p.n_splits, split = blockIdx.x % p.n_splits;
  const int kb0 = split * p.kb_per_split;
  const int nkb = min(p.kb_per_split, p.kb_total - kb0);
  const uint32_t ncols = tmem_cols(2 * p.n_pad);
  const bool soft_b = p.b_mode == B_SOFT_F32;
  const bool gu = p.flavor == EPI_GATEUP;
  const int S = kSplit ? p.n_splits : 1;

  if (threadIdx.x == 0) {
    for (int s = 0; s < stages; ++s) {
      mbar_init(&full[s], soft_b ? 5 : 1);   // TMA arrival (+ one per B-producer warp)
      mbar_init(&empty[s], 1);               // tcgen05.commit
    }
    mbar_init(done, 1);
    mbar_fence_init();
  }
  if (warp == 0) tmem_alloc(tmem_holder, ncols);
  if (warp == 4 && lane == 0) {
    tma_prefetch_desc(&m0);
    if (gu || p.flavor == EPI_QKV) tma_prefetch_desc(&m1);
    if (p.flavor == EPI_QKV) tma_prefetch_desc(&m2);
    if (!soft_b) tma_prefetch_desc(&mb);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  griddep_launch();
  const uint32_t tmem = *tmem_holder;
  bool ok = true;

  if (warp == 4) {
    // ---------------- TMA producer: weight tile (+ activation tile) per stage
    if (lane == 0) {
      const CUtensorMap* map = &m0;
      int y = tile * kTileRows;
      if (p.flavor == EPI_QKV) {
        const int tq = p.rows_q / kTileRows, tk = p.rows_k / kTileRows;
        if (tile >= tq + tk) { map = &m2; y = (tile - tq - tk) * kTileRows; }
        else if (tile >= tq) { map = &m1; y = (tile - tq) * kTileRows; }
      } else if (gu) {
        y = tile * kGuRows;
      }
      const uint64_t pol = l2_evict_first_policy();
      const int nbox = p.n_pad / 16;
      const uint32_t tx = abytes + (soft_b ? 0u : static_cast<uint32_t>(bbytes));
      auto load_a = [&](int i) {
        const int s = i % stages;
        const int x = (kb0 + i) * kKBlock;
        if (gu) {
          tma_load_2d(sA + s * abytes, &m0, x, y, &full[s], pol);
          tma_load_2d(sA + s * abytes + abytes / 2, &m1, x, y, &full[s], pol);
        } else {
          tma_load_2d(sA + s * abytes, map, x, y, &full[s], pol);
        }
      };
      auto load_b = [&](int i) {
        if (soft_b) return;
        const int s = i % stages;
        const int x = (kb0 + i) * kKBlock;
        // the activation map is [plane][rows][cols]: rows past the buffer's
        // are out of bounds (zero fill, no traffic) in either plane
        for (int b = 0; b < nbox; ++b) {
          tma_load_3d(sB + s * bbytes + b * 2048, &mb, x, p.act_row0 + b * 16, 0, &full[s], 0ull);
          tma_load_3d(sB + s * bbytes + (nbox + b) * 2048, &mb, x, p.act_row0 + b * 16, 1, &full[s], 0ull);
        }
      };
      // The first stages' weight tiles do not depend on earlier kernels.
      const int pre = p.prefetch_a ? min(stages, nkb) : 0;
      for (int i = 0; i < pre; ++i) {
        mbar_arrive_expect_tx(&full[i], tx);
        load_a(i);
      }
      griddep_wait();
      for (int i = 0; i < pre; ++i) load_b(i);
      int issued = pre;
      for (int i = pre; i < nkb; ++i) {
        const int s = i % stages;
        const uint32_t ph = (i / stages) & 1;
        if (!mbar_wait(&empty[s], ph ^ 1, p.status)) break;
        mbar_arrive_expect_tx(&full[s], tx);
        load_a(i);
        load_b(i);
        issued = i + 1;
      }
      // Drain: every issued copy has landed before the CTA moves on.
      for (int i = max(0, issued - stages); i < issued; ++i)
        mbar_wait(&full[i % stages], (i / stages) & 1, p.status);
    }
    __syncwarp();
  } else if (warp == 5) {
    // ---------------- MMA issuer
    if (lane == 0) {
      // hi and lo rows are adjacent in the stage: one MMA of N = 2 n_pad
      // covers both while N <= 256, else one MMA each
      const bool fused_lo = 2 * p.n_pad <= 256;
      const uint32_t idesc = idesc_bf16_m128(static_cast<uint32_t>(fused_lo ? 2 * p.n_pad : p.n_pad));
      for (int i = 0; i < nkb; ++i) {
        const int s = i % stages;
        const uint32_t ph = (i / stages) & 1;
        if (!mbar_wait(&full[s], ph, p.status)) break;
        tc_fence_after();
        const uint32_t a = smem_u32(sA + s * abytes);
        const uint32_t b = smem_u32(sB + s * bbytes);
        const uint32_t blo = b + static_cast<uint32_t>(p.n_pad) * 128u;
#pragma unroll
        for (int kk = 0; kk < kKBlock / 16; ++kk) {
          const uint64_t ad = smem_desc_sw128(a + kk * 32);
          tc_mma_bf16(tmem, ad, smem_desc_sw128(b + kk * 32), idesc, (i | kk) != 0);
          if (!fused_lo)
            tc_mma_bf16(tmem + static_cast<uint32_t>(p.n_pad), ad, smem_desc_sw128(blo + kk * 32), idesc,
                        (i | kk) != 0);
        }
        tc_commit(&empty[s]);
      }
      tc_commit(done);
    }
    __syncwarp();
  } else {
    // ---------------- warps 0-3: (B producer for f32 rows), norm scales, TMEM
    const int tid = threadIdx.x;
    griddep_wait();
    if (soft_b) {
      for (int i = 0; i < nkb; ++i) {
        const int s = i % stages;
        const uint32_t ph = (i / stages) & 1;
        if (!mbar_wait(&empty[s], ph ^ 1, p.status)) break;
        produce_b_f32(p, sB + s * bbytes, kb0 + i, tid);
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(&full[s]);
      }
    }
    compute_rstd(p, rstd, posn, tid, kTileRows);
    named_bar(1, kTileRows);
    ok = mbar_wait(done, 0, p.status);
    tc_fence_after();
    const uint32_t lane_base = tmem + ((static_cast<uint32_t>(warp) * 32u) << 16);
    const int nchunks = (p.M + kChunk - 1) / kChunk;
    float v[kChunk];
    if (!kSplit) {
      for (int c = 0; c < nchunks; ++c) {
        float vl[kChunk];
        tmem_ld16(lane_base + c * kChunk, v);
        tmem_ld16(lane_base + p.n_pad + c * kChunk, vl);
#pragma unroll
        for (int j = 0; j < kChunk; ++j) v[j] += vl[j];
        if (ok)
          epilogue_chunk<__nv_bfloat16>(p, tile, tid, c * kChunk, v, rstd, posn, es, valid_cols(p, c * kChunk));
      }
    } else {
      for (int c = 0; c < nchunks; ++c) {
        float vl[kChunk];
        tmem_ld16(lane_base + c * kChunk, v);
        tmem_ld16(lane_base + p.n_pad + c * kChunk, vl);
#pragma unroll
        for (int j = 0; j < kChunk; ++j)
          if (c * kChunk + j < p.M) part[(c * kChunk + j) * kTileRows + tid] = v[j] + vl[j];
      }
    }
    tc_fence_before();
    named_bar(1, kTileRows);
    if (warp == 0) {
      tc_fence_after();
      tmem_dealloc(tmem, ncols);
    }
  }
  if (kSplit) {
    // ---------------- split-K across the cluster: rank r finishes the token
    // columns n with n % S == r, summing every rank's partial in rank order
    // (all of a column's loads from the peers are issued before the sum)
    cluster_arrive_release();
    cluster_wait_acquire();
    if (warp < 4) {
      const int tid = threadIdx.x;
      uint32_t peer[8];
      const uint32_t mine = smem_u32(part) + static_cast<uint32_t>(tid) * 4u;
#pragma unroll
      for (int r = 0; r < 8; ++r) peer[r] = r < S ? mapa_shared(mine, r) : 0u;
      const int nchunks = (p.M + kChunk - 1) / kChunk;
      for (int c = 0; c < nchunks; ++c) {
        uint32_t own = 0;
#pragma unroll
        for (int j = 0; j < kChunk; ++j)
          if (c * kChunk + j < p.M && (c * kChunk + j) % S == split) own |= 1u << j;
        if (!own) continue;
        float v[kChunk];
#pragma unroll
        for (int j = 0; j < kChunk; ++j) {
          v[j] = 0.f;
          if ((own >> j) & 1u) {
            const uint32_t off = static_cast<uint32_t>((c * kChunk + j) * kTileRows) * 4u;
            float t[8];
#pragma unroll
            for (int r = 0; r < 8; ++r) t[r] = r < S ? ld_cluster_f32(peer[r] + off) : 0.f;
            float acc = t[0];
#pragma unroll
            for (int r = 1; r < 8; ++r)
              if (r < S) acc += t[r];
            v[j] = acc;
          }
        }
        epilogue_chunk<__nv_bfloat16>(p, tile, tid, c * kChunk, v, rstd, posn, es, own);
      }
    }
    // every rank keeps its shared memory until all have read it
    cluster_arrive_release();
    cluster_wait_acquire();
  }
}

// ------------------------------------------------------------------ FP32 FMA
__global__ void __launch_bounds__(128) proj_f32_kernel(const ProjArgs p) {
  __shared__ float Ws[kTileRows][kKBlockF32 + 1];
  __shared__ float Bs[kChunk][kKBlockF32];
  __shared__ float rstd[kChunk];
  __shared__ int posn[kChunk];
  __shared__ EpiSmem es;
  griddep_launch();
  griddep_wait();
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int tile = blockIdx.x / p.n_splits, split = blockIdx.x % p.n_splits;
  const int ttile = blockIdx.y, c0 = ttile * kChunk;
  const int kb0 = split * p.kb_per_split;
  const int nkb = min(p.kb_per_split, p.kb_total - kb0);
  const bool gu = p.flavor == EPI_GATEUP;

  // weight row of tile row r (nullptr = zero row)
  const float* w0 = static_cast<const float*>(p.w0);
  int row0 = tile * kTileRows, rows = p.n_out;
  if (p.flavor == EPI_QKV) {
    const int tq = p.rows_q / kTileRows, tk = p.rows_k / kTileRows;
    if (tile >= tq + tk) { w0 = static_cast<const float*>(p.w2); row0 = (tile - tq - tk) * kTileRows; rows = p.rows_v; }
    else if (tile >= tq) { w0 = static_cast<const float*>(p.w1); row0 = (tile - tq) * kTileRows; rows = p.rows_k; }
    else rows = p.rows_q;
  }
  auto wrow = [&](int r) -> const float* {
    if (gu) {
      const int f = tile * kGuRows + (r & (kGuRows - 1));
      if (f >= p.n_out) return nullptr;
      return static_cast<const float*>(r < kGuRows ? p.w0 : p.w1) + static_cast<size_t>(f) * p.K;
    }
    return row0 + r < rows ? w0 + static_cast<size_t>(row0 + r) * p.K : nullptr;
  };
  const float* act = static_cast<const float*>(p.act);
  if (tid < kChunk) {
    float r = 1.f;
    const int n = c0 + tid;
    if (p.ss && n < p.M) {
      float s = 0.f;
      for (int t = 0; t < p.ss_tiles; ++t) s += p.ss[static_cast<size_t>(t) * p.ss_ld + n];
      r = rsqrtf(s / static_cast<float>(p.d_norm) + p.eps);
    }
    rstd[tid] = r;
    if (p.flavor == EPI_QKV && n < p.M) {
      int seq, pos;
      row_seq_pos(p, n, seq, pos);
      posn[tid] = pos;
    }
  }
  __syncthreads();
  float acc[kChunk];
#pragma unroll
  for (int j = 0; j < kChunk; ++j) acc[j] = 0.f;
  for (int i = 0; i < nkb; ++i) {
    const int k = (kb0 + i) * kKBlockF32 + lane;
    for (int q = 0; q < kTileRows / 4; ++q) {
      const int r = warp + 4 * q;
      const float* wr = wrow(r);
      Ws[r][lane] = (wr && k < p.K) ? wr[k] : 0.f;
    }
    for (int e = 0; e < (kChunk * kKBlockF32) / 128; ++e) {
      const int idx = tid + 128 * e;
      const int j = idx / kKBlockF32, kk = idx % kKBlockF32;
      const int n = c0 + j, kg = (kb0 + i) * kKBlockF32 + kk;
      Bs[j][kk] = (n < p.M && kg < p.K) ? act[static_cast<size_t>(p.act_row0 + n) * p.ld_act + kg] : 0.f;
    }
    __syncthreads();
#pragma unroll 8
    for (int kk = 0; kk < kKBlockF32; ++kk) {
      const float w = Ws[tid][kk];
#pragma unroll
      for (int j = 0; j < kChunk; ++j) acc[j] = fmaf(w, Bs[j][kk], acc[j]);
    }
    __syncthreads();
  }
  const int row = tid;
  // epilogue_chunk indexes rstd and positions by token; shift so that
  // rstd[c0 + j] is this tile's
  float* rs = rstd - c0;
  const int* ps = posn - c0;
  if (p.n_splits == 1) {
    epilogue_chunk<float>(p, tile, row, c0, acc, rs, ps, es, valid_cols(p, c0));
    return;
  }
  const size_t reg = static_cast<size_t>(kTileRows) * kChunk;
  const int ci = tile * p.n_ttiles + ttile;
  float* mine = p.part + (static_cast<size_t>(ci) * p.n_splits + split) * reg;
#pragma unroll
  for (int j = 0; j < kChunk; ++j) mine[j * kTileRows + row] = acc[j];
  if (!split_arrive(p, ci, row, es)) return;
  const float* all = p.part + static_cast<size_t>(ci) * p.n_splits * reg;
#pragma unroll
  for (int j = 0; j < kChunk; ++j) acc[j] = sum_splits(all + j * kTileRows + row, reg, p.n_splits);
  epilogue_chunk<float>(p, tile, row, c0, acc, rs, ps, es, valid_cols(p, c0));
}

// ------------------------------------------------------------------ host
// Work per launch: n_tiles output tiles x n_splits K ranges.  bf16: one wave
// of at most two CTAs per SM (the shared-memory ring of four stages admits
// two), splits only while tiles are too few, at most 8 (a portable cluster)
// and at least 4 K blocks each.  f32: balanced waves of the FFMA kernel.
void plan_splits(ProjArgs& a, int n_sms, bool tc) {
  if (a.flavor == EPI_QKV)
    a.n_tiles = a.rows_q / kTileRows + a.rows_k / kTileRows + a.rows_v / kTileRows;
  else if (a.flavor == EPI_GATEUP)
    a.n_tiles = (a.n_out + kGuRows - 1) / kGuRows;
  else
    a.n_tiles = (a.n_out + kTileRows - 1) / kTileRows;
  const int kbw = tc ? kKBlock : kKBlockF32;
  a.kb_total = (a.K + kbw - 1) / kbw;
  if (tc) {
    int s = std::max(1, std::min(8, (2 * n_sms) / std::max(1, a.n_tiles)));
    s = std::max(1, std::min(s, a.kb_total / 4));
    a.kb_per_split = (a.kb_total + s - 1) / s;
    a.n_splits = (a.kb_total + a.kb_per_split - 1) / a.kb_per_split;
    return;
  }
  const int slots = 4 * n_sms;
  int best_s = 1, best_kbps = a.kb_total;
  double best_cost = 1e30;
  for (int s = 1; s <= 32 && s <= a.kb_total; ++s) {
    const int kbps = (a.kb_total + s - 1) / s;
    if (s > 1 && kbps < 2) break;
    const int s_eff = (a.kb_total + kbps - 1) / kbps;
    const long units = static_cast<long>(a.n_tiles) * s_eff;
    const long waves = (units + slots - 1) / slots;
    const double cost = static_cast<double>(waves) * (kbps + 2);
    if (cost < best_cost - 1e-9) { best_cost = cost; best_s = s_eff; best_kbps = kbps; }
  }
  a.n_splits = best_s;
  a.kb_per_split = best_kbps;
}

// Global split-K scratch (f32 path only; bf16 reduces inside the cluster).
size_t proj_partial_floats(const ProjArgs& a, bool tc) {
  if (tc || a.n_splits <= 1) return 0;
  const int ntt = (a.M + kChunk - 1) / kChunk;
  return static_cast<size_t>(a.n_tiles) * ntt * a.n_splits * kTileRows * kChunk;
}

static int tc_stages(int n_pad, size_t* smem_bytes) {
  const int per = 16384 + 2 * n_pad * 128;   // weight tile + hi and lo activation rows
  const int fixed = 1024 /*align*/ + 1024 /*barriers, tmem slot*/ + 8 * kMaxTokens /*rstd, positions*/;
  // two CTAs per SM while the ring keeps at least three stages
  int stages = std::max(2, std::min(4, (112 * 1024 - fixed) / per));
  *smem_bytes = static_cast<size_t>(fixed) + static_cast<size_t>(stages) * per;
  return stages;
}

cudaError_t launch_proj(const ProjArgs& a0, const ProjMaps* maps, cudaStream_t s) {
  cudaError_t e;
  if (a0.dtype == DVI_BF16) {
    static bool attr = false;
    if (!attr) {
      cudaFuncSetAttribute(proj_tc_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024);
      cudaFuncSetAttribute(proj_tc_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024);
      attr = true;
    }
    ProjArgs a = a0;
    // the cluster reduction keeps a [n_pad][128] partial in the A stages
    if (a.n_pad > 64 && a.n_splits > 1) {
      a.n_splits = 1;
      a.kb_per_split = a.kb_total;
    }
    size_t smem = 0;
    const int stages = tc_stages(a.n_pad, &smem);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(a.n_tiles * a.n_splits);
    cfg.blockDim = dim3(192);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute at[2];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    at[1].id = cudaLaunchAttributeClusterDimension;
    at[1].val.clusterDim.x = a.n_splits;
    at[1].val.clusterDim.y = 1;
    at[1].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = a.n_splits > 1 ? 2 : 1;
    e = a.n_splits > 1
            ? cudaLaunchKernelEx(&cfg, proj_tc_kernel<true>, maps->m0, maps->m1, maps->m2, maps->mb, a, stages)
            : cudaLaunchKernelEx(&cfg, proj_tc_kernel<false>, maps->m0, maps->m1, maps->m2, maps->mb, a, stages);
  } else {
    ProjArgs b = a0;
    b.n_ttiles = (a0.M + kChunk - 1) / kChunk;
    e = launch_pdl(proj_f32_kernel, dim3(a0.n_tiles * a0.n_splits, b.n_ttiles), dim3(128), 0, s, b);
  }
  return e != cudaSuccess ? e : cudaGetLastError();
}

static PFN_cuTensorMapEncodeTiled_v12000 encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 encode = nullptr;
  if (!encode) {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) !=
            cudaSuccess ||
        q != cudaDriverEntryPointSuccess || !fn)
      return nullptr;
    encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  }
  return encode;
}

static bool make_map(CUtensorMap* map, const void* ptr, int rows, int cols, int box_rows) {
  auto encode = encoder();
  if (!encode) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(cols) * 2};
  cuuint32_t box[2] = {kKBlock, static_cast<cuuint32_t>(box_rows)};
  cuuint32_t estr[2] = {1, 1};
  const CUresult r = encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box,
                            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

bool make_weight_map(CUtensorMap* map, const void* w, int rows, int cols) {
  return make_map(map, w, rows, cols, kTileRows);
}
bool make_half_weight_map(CUtensorMap* map, const void* w, int rows, int cols) {
  return make_map(map, w, rows, cols, kGuRows);
}
bool make_act_map(CUtensorMap* map, const void* act, int rows, int cols) {
  // two planes (hi, lo) of [rows][cols] bf16, boxes of 16 rows x 64 columns
  auto encode = encoder();
  if (!encode) return false;
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows), 2};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(cols) * 2, static_cast<cuuint64_t>(rows) * cols * 2};
  cuuint32_t box[3] = {kKBlock, 16, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  const CUresult r = encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(act), dims, strides, box,
                            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}
bool make_kv_map(CUtensorMap* map, const void* cache, long long rows, int hd) {
  auto encode = encoder();
  if (!encode) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(hd), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(hd) * 2};
  cuuint32_t box[2] = {64, 64};
  cuuint32_t estr[2] = {1, 1};
  const CUresult r = encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(cache), dims, strides, box,
                            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

}  // namespace dvi
