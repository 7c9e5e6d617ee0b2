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
// for its predecessor.  The drafter head (bf16, few rows) also forms the
// LoRA term's B u in its epilogue warps while the weights stream.
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
//
// Persistent chain (bf16, opt-in): one launch runs several projections of
// a pass in order (a layer's O, gate/up, down and the next layer's QKV).
// Each phase's (tile, K block) sequence is cut into equal contiguous ranges,
// one per CTA (stream-K); a tile covered by several CTAs is summed in K
// order by the CTA holding its first K block, from the others' partials in
// global scratch.  A phase's activation loads wait on a release/acquire
// counter of the previous phase's finished tiles (bounded polls); its weight
// loads do not, so the ring fills across the boundary.  Every CTA must be
// resident at once: the grid is the number of CTAs the SMs hold.
#include <algorithm>
#include <cudaTypedefs.h>

#include "finalize.cuh"

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
      // loads in batches of eight, summed in tile order
      float s = 0.f;
      int t = 0;
      for (; t + 8 <= p.ss_tiles; t += 8) {
        float x[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) x[u] = __ldcg(p.ss + static_cast<size_t>(t + u) * p.ss_ld + n);
#pragma unroll
        for (int u = 0; u < 8; ++u) s += x[u];
      }
      for (; t < p.ss_tiles; ++t) s += __ldcg(p.ss + static_cast<size_t>(t) * p.ss_ld + n);
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
                               const float* rstd, const int* posn, EpiSmem& es, uint32_t own,
                               const float* bu_s = nullptr) {
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
    // sequence of column c0 + j, advanced column by column (no division in
    // the unrolled loop)
    int seq = p.seq0 + c0 / p.rows_per_seq, in_seq = c0 % p.rows_per_seq;
#pragma unroll
    for (int j = 0; j < kChunk; ++j, seq += (++in_seq == p.rows_per_seq), in_seq = in_seq == p.rows_per_seq ? 0 : in_seq) {
      const int n = c0 + j;
      if ((own >> j) & 1u) {
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
        xn = __ldcg(xp) + v[j];
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
      if (p.lora_r <= kBuRank) {
        // the row of A once into registers for every column of the chunk
        float av[kBuRank];
#pragma unroll
        for (int q = 0; q < kBuRank; ++q) av[q] = q < p.lora_r ? arow[q] : 0.f;
        for (int j = 0; j < kChunk; ++j) {
          const int n = c0 + j;
          if ((own >> j) & 1u) {
            const float* bu = (p.lora_bmat ? bu_s : p.lora_bu) + static_cast<size_t>(n) * p.lora_r;
            float acc = 0.f;
#pragma unroll
            for (int q = 0; q < kBuRank; ++q)
              if (q < p.lora_r) acc = fmaf(av[q], bu[q], acc);
            z[j] = fmaf(p.gamma, acc, z[j]);
          }
        }
      } else {
        for (int j = 0; j < kChunk; ++j) {
          const int n = c0 + j;
          if ((own >> j) & 1u) {
            const float* bu = (p.lora_bmat ? bu_s : p.lora_bu) + static_cast<size_t>(n) * p.lora_r;
            float acc = 0.f;
            for (int q = 0; q < p.lora_r; ++q) acc = fmaf(arow[q], bu[q], acc);
            z[j] = fmaf(p.gamma, acc, z[j]);
          }
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
            row = i < p.log_dst_rows ? row / p.log_src_rows * p.log_dst_rows + p.log_dst_off + i : -1;
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
// instantiation carries no cluster code.  kFinNT > 0: a head whose last CTA
// may run a finalize step (row arrays of kFinNT tiles: d <= 128 kFinNT); the
// other instantiations carry none of its code or registers.
template <bool kSplit, int kFinNT = 0>
__global__ void __launch_bounds__(192, 2)
    proj_tc_kernel(const __grid_constant__ CUtensorMap m0, const __grid_constant__ CUtensorMap m1,
                   const __grid_constant__ CUtensorMap m2, const __grid_constant__ CUtensorMap mb,
                   const ProjArgs p, int stages, const __grid_constant__ FinArgs fin) {
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
  float* bu_s = reinterpret_cast<float*>(posn + kMaxTokens);   // [kBuRows][kBuRank] in-kernel B u

  // after `done` every stage is free: epilogue scratch in the first A
  // stage, then this split's partial tile [n_pad][128] (n_pad * 512 bytes,
  // which the remaining A stages and the B stages always hold: at least two
  // stages of 16 KB + n_pad * 256 bytes)
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
      dep_wait(p.dep_wait, p.dep_count, p.status);
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
    if (p.dep_wait) {
      if (tid == 0) dep_wait(p.dep_wait, p.dep_count, p.status);
      named_bar(1, kTileRows);
    } else {
      griddep_wait();
    }
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
    if (p.lora_bmat) {
      // B u of the LoRA term while the weights stream: warp w takes rows
      // q = w, w + 4, ... of B; u = (x * rstd) * g, four features per lane
      // per step, summed per lane in feature order then across the warp
      for (int n = 0; n < p.M; ++n) {
        const float r = rstd[n];
        const float4* x4 = reinterpret_cast<const float4*>(p.bu_x + static_cast<size_t>(n) * p.bu_ldx);
        const float4* g4 = reinterpret_cast<const float4*>(p.bu_g);
        for (int q = warp; q < p.lora_r; q += 4) {
          const float4* br = reinterpret_cast<const float4*>(p.lora_bmat + static_cast<size_t>(q) * p.K);
          float acc = 0.f;
#pragma unroll 4
          for (int c = lane; c < p.K / 4; c += 32) {
            const float4 b = br[c], xx = x4[c], gg = g4[c];
            acc = fmaf(b.x, xx.x * r * gg.x, acc);
            acc = fmaf(b.y, xx.y * r * gg.y, acc);
            acc = fmaf(b.z, xx.z * r * gg.z, acc);
            acc = fmaf(b.w, xx.w * r * gg.w, acc);
          }
          acc = warp_sum(acc);
          if (lane == 0) bu_s[n * p.lora_r + q] = acc;
        }
      }
      named_bar(1, kTileRows);
    }
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
          epilogue_chunk<__nv_bfloat16>(p, tile, tid, c * kChunk, v, rstd, posn, es, valid_cols(p, c * kChunk),
                                        bu_s);
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
    // a head whose last CTA runs the pass's finalize step (the ring is free)
    if constexpr (!kSplit && kFinNT > 0) {
      if (fin.kind != FIN_NONE) head_finalize<kFinNT>(fin, sA + abytes, tid);
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
        // columns n of [c0, c0 + 16) with n = split (mod S)
        const int c0 = c * kChunk, c1 = min(p.M, c0 + kChunk);
        uint32_t own = 0;
        for (int n = c0 + (split - c0 % S + S) % S; n < c1; n += S) own |= 1u << (n - c0);
        if (!own) continue;
        // one compact loop over the owned columns: the sum of every rank's
        // partial (in rank order) replaces this rank's own partial, which
        // only this rank reads for the columns it owns
#pragma unroll 1
        for (int j = 0; j < kChunk; ++j) {
          if (!((own >> j) & 1u)) continue;
          const uint32_t off = static_cast<uint32_t>((c * kChunk + j) * kTileRows) * 4u;
          float t[8];
#pragma unroll
          for (int r = 0; r < 8; ++r) t[r] = r < S ? ld_cluster_f32(peer[r] + off) : 0.f;
          float acc = t[0];
#pragma unroll
          for (int r = 1; r < 8; ++r)
            if (r < S) acc += t[r];
          part[(c * kChunk + j) * kTileRows + tid] = acc;
        }
        float v[kChunk];
#pragma unroll
        for (int j = 0; j < kChunk; ++j) v[j] = ((own >> j) & 1u) ? part[(c * kChunk + j) * kTileRows + tid] : 0.f;
        epilogue_chunk<__nv_bfloat16>(p, tile, tid, c * kChunk, v, rstd, posn, es, own, bu_s);
      }
    }
    // every rank keeps its shared memory until all have read it
    cluster_arrive_release();
    cluster_wait_acquire();
  }
  if (p.dep_signal) {
    // this CTA's outputs (and a head's finalize step) are written; the
    // barrier orders them before thread 0's release
    __syncthreads();
    if (threadIdx.x == 0) dep_signal(p.dep_signal);
  }
}

// ------------------------------------------------------------------ chain
__device__ __forceinline__ int ld_acquire_gpu(const int* ptr) {
  int v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(ptr) : "memory");
  return v;
}
__device__ __forceinline__ void red_release_gpu_add(int* ptr, int v) {
  asm volatile("red.release.gpu.global.add.s32 [%0], %1;" ::"l"(ptr), "r"(v) : "memory");
}
// Orders this thread's generic-proxy global accesses with its later (or
// earlier) TMA accesses.
__device__ __forceinline__ void fence_proxy_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}

// CTAs that take part in a phase of `all` blocks: every one of them gets at
// least one block, so a tile's contributors are consecutive CTAs.
__device__ __forceinline__ int chain_width(long long all, int n_ctas) {
  return static_cast<int>(all < n_ctas ? all : n_ctas);
}
// The CTA's share of one phase: K blocks [k0, k1) of the phase's sequence of
// n_tiles x kb_total (tile-major) blocks.
struct ChainRange {
  long long k0[kChainMax];
  int n[kChainMax];
  int total;
};
__device__ __forceinline__ void chain_range(const ChainArgs& a, int cta, ChainRange& r) {
  r.total = 0;
#pragma unroll
  for (int ph = 0; ph < kChainMax; ++ph) {
    r.k0[ph] = 0;
    r.n[ph] = 0;
    if (ph < a.n_phases) {
      const long long all = static_cast<long long>(a.p[ph].n_tiles) * a.p[ph].kb_total;
      const int g = chain_width(all, a.n_ctas);
      if (cta < g) {
        r.k0[ph] = all * cta / g;
        r.n[ph] = static_cast<int>(all * (cta + 1) / g - r.k0[ph]);
        r.total += r.n[ph];
      }
    }
  }
}
// Sequential walk over the CTA's blocks: phase, tile, K block within the tile.
struct ChainCursor {
  int ph, tile, kb, kbt, left;
};
__device__ __forceinline__ void cursor_settle(const ChainArgs& a, const ChainRange& r, ChainCursor& c) {
  while (c.left == 0 && c.ph + 1 < a.n_phases) {
    ++c.ph;
    c.left = r.n[c.ph];
    c.kbt = a.p[c.ph].kb_total;
    c.tile = static_cast<int>(r.k0[c.ph] / c.kbt);
    c.kb = static_cast<int>(r.k0[c.ph] - static_cast<long long>(c.tile) * c.kbt);
  }
}
__device__ __forceinline__ void cursor_init(const ChainArgs& a, const ChainRange& r, ChainCursor& c) {
  c.ph = -1;
  c.left = 0;
  cursor_settle(a, r, c);
}
__device__ __forceinline__ void cursor_next(const ChainArgs& a, const ChainRange& r, ChainCursor& c) {
  --c.left;
  if (++c.kb == c.kbt) {
    c.kb = 0;
    ++c.tile;
  }
  if (c.left == 0) cursor_settle(a, r, c);
}
// CTA whose range holds block k of a phase with `all` blocks.
__device__ __forceinline__ int chain_owner(long long k, long long all, int n_ctas) {
  const long long g = chain_width(all, n_ctas);
  return static_cast<int>(((k + 1) * g + all - 1) / all) - 1;
}

constexpr uint32_t kChainPollLimit = 1u << 21;   // polls of another CTA's counter before giving up

__global__ void __launch_bounds__(192, 2) proj_chain_kernel(const __grid_constant__ ChainArgs a, int stages) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  uint8_t* base = smem_raw + (((raw + 1023u) & ~1023u) - raw);
  constexpr int abytes = 16384;
  const int n_pad = a.p[0].n_pad;
  const int bbytes = 2 * n_pad * 128;
  uint8_t* sA = base;
  uint8_t* sB = base + stages * abytes;
  uint64_t* full = reinterpret_cast<uint64_t*>(sB + stages * bbytes);
  uint64_t* empty = full + stages;
  uint64_t* accf = empty + stages;   // [2] accumulator b holds a finished segment
  uint64_t* acce = accf + 2;         // [2] accumulator b has been read
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(acce + 2);
  float* rstd = reinterpret_cast<float*>(tmem_holder + 4);
  int* posn = reinterpret_cast<int*>(rstd + kMaxTokens);
  EpiSmem& es = *reinterpret_cast<EpiSmem*>(posn + kMaxTokens);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int cta = blockIdx.x;
  const uint32_t bufcols = tmem_cols(2 * n_pad);
  int* status = a.p[0].status;
  ChainRange rg;
  chain_range(a, cta, rg);

  if (threadIdx.x == 0) {
    for (int s = 0; s < stages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&accf[b], 1);
      mbar_init(&acce[b], 1);
    }
    mbar_fence_init();
  }
  if (warp == 0) tmem_alloc(tmem_holder, 2 * bufcols);
  if (warp == 4 && lane == 0) {
    for (int ph = 0; ph < a.n_phases; ++ph) {
      const int f = a.p[ph].flavor;
      tma_prefetch_desc(&a.maps[ph][0]);
      if (f == EPI_GATEUP || f == EPI_QKV) tma_prefetch_desc(&a.maps[ph][1]);
      if (f == EPI_QKV) tma_prefetch_desc(&a.maps[ph][2]);
      tma_prefetch_desc(&a.maps[ph][3]);
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  griddep_launch();
  const uint32_t tmem = *tmem_holder;

  if (warp == 4) {
    // ---------------- TMA producer.  Weight loads run up to the ring's depth
    // ahead of the activation loads, which wait for the previous phase.
    if (lane == 0 && rg.total > 0) {
      const uint64_t pol = l2_evict_first_policy();
      const uint32_t tx = abytes + static_cast<uint32_t>(bbytes);
      const int nbox = n_pad / 16;
      auto load_a = [&](int j, const ChainCursor& c) {
        const ProjArgs& p = a.p[c.ph];
        const int x = c.kb * kKBlock;
        uint8_t* dst = sA + (j % stages) * abytes;
        uint64_t* bar = &full[j % stages];
        if (p.flavor == EPI_GATEUP) {
          tma_load_2d(dst, &a.maps[c.ph][0], x, c.tile * kGuRows, bar, pol);
          tma_load_2d(dst + abytes / 2, &a.maps[c.ph][1], x, c.tile * kGuRows, bar, pol);
        } else {
          int m = 0, y = c.tile * kTileRows;
          if (p.flavor == EPI_QKV) {
            const int tq = p.rows_q / kTileRows, tk = p.rows_k / kTileRows;
            if (c.tile >= tq + tk) { m = 2; y = (c.tile - tq - tk) * kTileRows; }
            else if (c.tile >= tq) { m = 1; y = (c.tile - tq) * kTileRows; }
          }
          tma_load_2d(dst, &a.maps[c.ph][m], x, y, bar, pol);
        }
      };
      auto load_b = [&](int j, const ChainCursor& c) {
        const int x = c.kb * kKBlock;
        const int row0 = a.p[c.ph].act_row0;
        uint8_t* dst = sB + (j % stages) * bbytes;
        uint64_t* bar = &full[j % stages];
        for (int b = 0; b < nbox; ++b) {
          tma_load_3d(dst + b * 2048, &a.maps[c.ph][3], x, row0 + b * 16, 0, bar, 0ull);
          tma_load_3d(dst + (nbox + b) * 2048, &a.maps[c.ph][3], x, row0 + b * 16, 1, bar, 0ull);
        }
      };
      int ia = 0, ib = 0;
      ChainCursor ca, cb;
      cursor_init(a, rg, ca);
      cursor_init(a, rg, cb);
      for (; ia < min(stages, rg.total); ++ia) {
        mbar_arrive_expect_tx(&full[ia], tx);
        load_a(ia, ca);
        cursor_next(a, rg, ca);
      }
      griddep_wait();
      int ready = 0;          // phases 0..ready may load activations
      uint32_t idle = 0;
      bool ok = true;
      while (ib < rg.total) {
        bool prog = false;
        if (ib < ia) {
          const int ph = cb.ph;
          if (ph > ready && ld_acquire_gpu(a.phase_done + ph - 1) >= a.p[ph - 1].n_tiles) {
            fence_proxy_async_global();
            ready = ph;
          }
          if (ph <= ready) {
            load_b(ib, cb);
            cursor_next(a, rg, cb);
            ++ib;
            prog = true;
          }
        }
        if (ia < rg.total && mbar_test_wait(&empty[ia % stages], ((ia / stages) & 1) ^ 1)) {
          mbar_arrive_expect_tx(&full[ia % stages], tx);
          load_a(ia, ca);
          cursor_next(a, rg, ca);
          ++ia;
          prog = true;
        }
        if (prog) {
          idle = 0;
        } else if (++idle > kChainPollLimit) {
          flag_status(status, DVI_DEV_TIMEOUT);
          ok = false;
          break;
        } else if (idle > 16) {
          __nanosleep(64);
        }
      }
      if (!ok) {
        // copies in flight land within microseconds; wait (bounded) for the
        // stages whose activation loads were issued
        for (int j = max(0, ib - stages); j < ib; ++j) mbar_wait(&full[j % stages], (j / stages) & 1, status);
      }
    }
    __syncwarp();
  } else if (warp == 5) {
    // ---------------- MMA issuer: one accumulator per segment (a run of
    // blocks of one tile), alternating between two TMEM buffers
    if (lane == 0 && rg.total > 0) {
      const bool fused_lo = 2 * n_pad <= 256;
      const uint32_t idesc = idesc_bf16_m128(static_cast<uint32_t>(fused_lo ? 2 * n_pad : n_pad));
      int seg = -1, cur_ph = -1, cur_tile = -1;
      uint32_t acc = tmem;
      ChainCursor cm;
      cursor_init(a, rg, cm);
      for (int j = 0; j < rg.total; ++j, cursor_next(a, rg, cm)) {
        const bool first = cm.ph != cur_ph || cm.tile != cur_tile;
        if (first) {
          if (seg >= 0) tc_commit(&accf[seg & 1]);
          ++seg;
          cur_ph = cm.ph;
          cur_tile = cm.tile;
          if (seg >= 2 && !mbar_wait(&acce[seg & 1], ((seg >> 1) - 1) & 1, status)) break;
          tc_fence_after();
          acc = tmem + static_cast<uint32_t>(seg & 1) * bufcols;
        }
        const int s = j % stages;
        if (!mbar_wait(&full[s], (j / stages) & 1, status)) break;
        tc_fence_after();
        const uint32_t ab = smem_u32(sA + s * abytes);
        const uint32_t bb = smem_u32(sB + s * bbytes);
        const uint32_t blo = bb + static_cast<uint32_t>(n_pad) * 128u;
#pragma unroll
        for (int kk = 0; kk < kKBlock / 16; ++kk) {
          const uint64_t ad = smem_desc_sw128(ab + kk * 32);
          const uint32_t accum = (first && kk == 0) ? 0u : 1u;
          tc_mma_bf16(acc, ad, smem_desc_sw128(bb + kk * 32), idesc, accum);
          if (!fused_lo)
            tc_mma_bf16(acc + static_cast<uint32_t>(n_pad), ad, smem_desc_sw128(blo + kk * 32), idesc, accum);
        }
        tc_commit(&empty[s]);
      }
      if (seg >= 0) tc_commit(&accf[seg & 1]);
    }
    __syncwarp();
  } else {
    // ---------------- warps 0-3: partial tiles, reductions, epilogues
    const int tid = threadIdx.x;
    griddep_wait();
    int seg = 0;
    bool ok = true;
    for (int ph = 0; ph < a.n_phases && ok; ++ph) {
      const ProjArgs& p = a.p[ph];
      const long long all = static_cast<long long>(p.n_tiles) * p.kb_total;
      const int nchunks = (p.M + kChunk - 1) / kChunk;
      const size_t slot = static_cast<size_t>(n_pad) * kTileRows;
      if (rg.n[ph] > 0) {
        // 1/rms of this phase's rows as soon as the previous phase is done
        // (overlapping this phase's weight stream)
        if (ph > 0) {
          if (tid == 0) {
            uint32_t i = 0;
            while (ld_acquire_gpu(a.phase_done + ph - 1) < a.p[ph - 1].n_tiles) {
              if (++i > kChainPollLimit) {
                flag_status(status, DVI_DEV_TIMEOUT);
                break;
              }
              if (i > 16) __nanosleep(64);
            }
          }
          named_bar(1, kTileRows);
          ld_acquire_gpu(a.phase_done + ph - 1);
        }
        compute_rstd(p, rstd, posn, tid, kTileRows);
        named_bar(1, kTileRows);
      }
      auto finish_tile = [&]() {
        __threadfence();
        fence_proxy_async_global();
        named_bar(1, kTileRows);
        if (tid == 0) red_release_gpu_add(a.phase_done + ph, 1);
      };
      long long k = rg.k0[ph];
      const long long kend = k + rg.n[ph];
      while (k < kend) {
        const int tile = static_cast<int>(k / p.kb_total);
        const long long tend = min(kend, static_cast<long long>(tile + 1) * p.kb_total);
        const bool whole = tend - k == p.kb_total;
        const int b = seg & 1;
        ok = mbar_wait(&accf[b], (seg >> 1) & 1, status);
        if (!ok) break;
        tc_fence_after();
        const uint32_t lane_base = tmem + ((static_cast<uint32_t>(warp) * 32u) << 16) + static_cast<uint32_t>(b) * bufcols;
        float v[kChunk], vl[kChunk];
        if (whole) {
          for (int c = 0; c < nchunks; ++c) {
            tmem_ld16(lane_base + c * kChunk, v);
            tmem_ld16(lane_base + n_pad + c * kChunk, vl);
#pragma unroll
            for (int j = 0; j < kChunk; ++j) v[j] += vl[j];
            epilogue_chunk<__nv_bfloat16>(p, tile, tid, c * kChunk, v, rstd, posn, es, valid_cols(p, c * kChunk));
          }
          tc_fence_before();
          named_bar(1, kTileRows);
          if (tid == 0) mbar_arrive(&acce[b]);
          finish_tile();
        } else {
          const long long t0 = static_cast<long long>(tile) * p.kb_total;
          const int first = chain_owner(t0, all, a.n_ctas);
          const int last = chain_owner(t0 + p.kb_total - 1, all, a.n_ctas);
          int* ctr = a.tile_ctr + ph * kChainTiles + tile;
          if (cta != first) {
            // contributor: partial into the slot, then a release increment
            // of the tile's counter; nothing to wait for
            float* mine = a.part + (static_cast<size_t>(tile) + cta) * slot;
            for (int c = 0; c < nchunks; ++c) {
              tmem_ld16(lane_base + c * kChunk, v);
              tmem_ld16(lane_base + n_pad + c * kChunk, vl);
#pragma unroll
              for (int j = 0; j < kChunk; ++j)
                if (c * kChunk + j < p.M) __stcg(mine + (c * kChunk + j) * kTileRows + tid, v[j] + vl[j]);
            }
            tc_fence_before();
            __threadfence();
            named_bar(1, kTileRows);
            if (tid == 0) {
              mbar_arrive(&acce[b]);
              red_release_gpu_add(ctr, 1);
            }
          } else {
            // finisher (the CTA holding the tile's first K block, whose last
            // segment of the phase this is): wait for the other contributors,
            // then sum its own accumulator and their partials in K order
            if (tid == 0) {
              uint32_t i = 0;
              while (ld_acquire_gpu(ctr) < last - first) {
                if (++i > kChainPollLimit) {
                  flag_status(status, DVI_DEV_TIMEOUT);
                  break;
                }
                if (i > 16) __nanosleep(32);
              }
            }
            named_bar(1, kTileRows);
            const float* src = a.part + (static_cast<size_t>(tile) + first) * slot + tid;
            const int nc = last - first + 1;
            for (int c = 0; c < nchunks; ++c) {
              const uint32_t own = valid_cols(p, c * kChunk);
              const float* col = src + static_cast<size_t>(c) * kChunk * kTileRows;
              tmem_ld16(lane_base + c * kChunk, v);
              tmem_ld16(lane_base + n_pad + c * kChunk, vl);
#pragma unroll
              for (int j = 0; j < kChunk; ++j) v[j] += vl[j];
              // the other contributors' partials: four contributors' loads of
              // all 16 columns in flight at a time (columns past M are in
              // the slot and ignored)
              int cc = 1;
              for (; cc + 4 <= nc; cc += 4) {
                float t[4][kChunk];
#pragma unroll
                for (int u = 0; u < 4; ++u)
#pragma unroll
                  for (int j = 0; j < kChunk; ++j) t[u][j] = __ldcg(col + (cc + u) * slot + j * kTileRows);
#pragma unroll
                for (int u = 0; u < 4; ++u)
#pragma unroll
                  for (int j = 0; j < kChunk; ++j) v[j] += t[u][j];
              }
              for (; cc < nc; ++cc) {
                float t[kChunk];
#pragma unroll
                for (int j = 0; j < kChunk; ++j) t[j] = __ldcg(col + cc * slot + j * kTileRows);
#pragma unroll
                for (int j = 0; j < kChunk; ++j) v[j] += t[j];
              }
#pragma unroll
              for (int j = 0; j < kChunk; ++j) v[j] = ((own >> j) & 1u) ? v[j] : 0.f;
              epilogue_chunk<__nv_bfloat16>(p, tile, tid, c * kChunk, v, rstd, posn, es, own);
            }
            tc_fence_before();
            named_bar(1, kTileRows);
            if (tid == 0) {
              mbar_arrive(&acce[b]);
              *ctr = 0;
            }
            finish_tile();
          }
        }
        ++seg;
        k = tend;
      }
    }
  }
  // ---------------- teardown; the last CTA to leave resets the phase counters
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, 2 * bufcols);
  }
  if (threadIdx.x == 0) {
    __threadfence();
    if (atomicAdd(a.exit_ctr, 1) == a.n_ctas - 1) {
      for (int ph = 0; ph < kChainMax; ++ph) a.phase_done[ph] = 0;
      *a.exit_ctr = 0;
      __threadfence();
    }
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
  const int fixed = 1024 /*align*/ + 1024 /*barriers, tmem slot*/ + 8 * kMaxTokens /*rstd, positions*/ +
                    4 * kBuRows * kBuRank /*in-kernel B u*/;
  // two CTAs per SM while the ring keeps at least three stages
  int stages = std::max(2, std::min(4, (112 * 1024 - fixed) / per));
  *smem_bytes = static_cast<size_t>(fixed) + static_cast<size_t>(stages) * per;
  return stages;
}

size_t fin_smem_bytes() { return (sizeof(FinSmem) + 15) / 16 * 16; }

bool head_fin_ok(const ProjArgs& a, size_t stage_bytes, bool* stage) {
  if (a.dtype != DVI_BF16 || a.flavor != EPI_HEAD || a.n_splits != 1) return false;
  size_t smem = 0;
  const int stages = tc_stages(a.n_pad, &smem);
  const size_t ring = static_cast<size_t>(stages) * (16384 + 2 * static_cast<size_t>(a.n_pad) * 128);
  *stage = ring >= 16384 + fin_smem_bytes() + stage_bytes;
  return ring >= 16384 + fin_smem_bytes();
}

cudaError_t launch_proj(const ProjArgs& a0, const ProjMaps* maps, cudaStream_t s, const FinArgs* fin) {
  cudaError_t e;
  FinArgs f{};
  if (fin) f = *fin;
  if (a0.dtype == DVI_BF16) {
    static PerDevice attr;
    attr.once([] {
      cudaFuncSetAttribute(proj_tc_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024);
      cudaFuncSetAttribute(proj_tc_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024);
      cudaFuncSetAttribute(proj_tc_kernel<false, 32>, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024);
      cudaFuncSetAttribute(proj_tc_kernel<false, 64>, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024);
    });
    ProjArgs a = a0;
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
    if (a.n_splits > 1)
      e = cudaLaunchKernelEx(&cfg, proj_tc_kernel<true>, maps->m0, maps->m1, maps->m2, maps->mb, a, stages, f);
    else if (f.kind == FIN_NONE)
      e = cudaLaunchKernelEx(&cfg, proj_tc_kernel<false>, maps->m0, maps->m1, maps->m2, maps->mb, a, stages, f);
    else if (a.K <= 32 * kTileRows)
      e = cudaLaunchKernelEx(&cfg, proj_tc_kernel<false, 32>, maps->m0, maps->m1, maps->m2, maps->mb, a, stages, f);
    else
      e = cudaLaunchKernelEx(&cfg, proj_tc_kernel<false, 64>, maps->m0, maps->m1, maps->m2, maps->mb, a, stages, f);
  } else {
    ProjArgs b = a0;
    b.n_ttiles = (a0.M + kChunk - 1) / kChunk;
    e = launch_pdl(proj_f32_kernel, dim3(a0.n_tiles * a0.n_splits, b.n_ttiles), dim3(128), 0, s, b);
  }
  return e != cudaSuccess ? e : cudaGetLastError();
}

// Chain kernel: ring depth for two CTAs per SM at n_pad.
static int chain_stages(int n_pad, size_t* smem_bytes) {
  const int per = 16384 + 2 * n_pad * 128;
  const int fixed = 1024 /*align*/ + 16 * 8 + 16 /*barriers, tmem slot*/ + 8 * kMaxTokens /*rstd, positions*/ +
                    static_cast<int>(sizeof(EpiSmem));
  const int budget = 113 * 1024;   // two CTAs per SM
  int stages = std::max(2, std::min(6, (budget - fixed) / per));
  *smem_bytes = static_cast<size_t>(fixed) + static_cast<size_t>(stages) * per;
  return stages;
}

static void chain_attr() {
  static PerDevice done;
  done.once([] {
    cudaFuncSetAttribute(proj_chain_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024);
    cudaFuncSetAttribute(proj_chain_kernel, cudaFuncAttributePreferredSharedMemoryCarveout,
                         cudaSharedmemCarveoutMaxShared);
  });
}

int chain_ctas_per_sm(int n_pad) {
  if (n_pad < 16 || n_pad > kChainMaxPad || n_pad % 16) return 0;
  chain_attr();
  size_t smem = 0;
  chain_stages(n_pad, &smem);
  // from the device limits: shared memory (with the per-block reservation)
  // and registers (allocated per warp in units of 256)
  int dev = 0, smem_sm = 0, reserved = 0, regs_sm = 0;
  cudaFuncAttributes fa{};
  if (cudaGetDevice(&dev) != cudaSuccess || cudaFuncGetAttributes(&fa, proj_chain_kernel) != cudaSuccess ||
      cudaDeviceGetAttribute(&smem_sm, cudaDevAttrMaxSharedMemoryPerMultiprocessor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&reserved, cudaDevAttrReservedSharedMemoryPerBlock, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&regs_sm, cudaDevAttrMaxRegistersPerMultiprocessor, dev) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  const size_t per_cta = smem + fa.sharedSizeBytes + static_cast<size_t>(reserved);
  const int by_smem = static_cast<int>(static_cast<size_t>(smem_sm) / per_cta);
  const int regs_warp = (fa.numRegs * 32 + 255) / 256 * 256;
  const int by_regs = regs_sm / (regs_warp * 6);
  return std::max(0, std::min(2, std::min(by_smem, by_regs)));
}

size_t chain_partial_floats(int max_tiles, int n_ctas, int n_pad) {
  return static_cast<size_t>(max_tiles + n_ctas) * n_pad * kTileRows;
}

cudaError_t launch_chain(const ChainArgs& a, cudaStream_t s) {
  chain_attr();
  size_t smem = 0;
  const int stages = chain_stages(a.p[0].n_pad, &smem);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(a.n_ctas);
  cfg.blockDim = dim3(192);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, proj_chain_kernel, a, stages);
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
bool make_weight_map_kblocks(CUtensorMap* map, const void* w, int rows, int cols, int box_rows, int box_kblocks) {
  // W [rows][cols] bf16 seen as [cols / 64][rows][64]: one box is box_kblocks
  // tiles of box_rows x 64 (each tile 128-byte swizzled, tiles consecutive)
  auto encode = encoder();
  if (!encode || cols % kKBlock || box_rows < 1 || box_rows > 256 || box_kblocks < 1 || box_kblocks > 256)
    return false;
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(kKBlock), static_cast<cuuint64_t>(rows),
                        static_cast<cuuint64_t>(cols / kKBlock)};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(cols) * 2, static_cast<cuuint64_t>(kKBlock) * 2};
  cuuint32_t box[3] = {kKBlock, static_cast<cuuint32_t>(box_rows), static_cast<cuuint32_t>(box_kblocks)};
  cuuint32_t estr[3] = {1, 1, 1};
  const CUresult r = encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(w), dims, strides, box,
                            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}
bool make_act_map_box(CUtensorMap* map, const void* act, int rows, int cols, int box_rows) {
  // two planes (hi, lo) of [rows][cols] bf16, boxes of box_rows rows x 64 columns
  auto encode = encoder();
  if (!encode || box_rows < 1 || box_rows > 256) return false;
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows), 2};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(cols) * 2, static_cast<cuuint64_t>(rows) * cols * 2};
  cuuint32_t box[3] = {kKBlock, static_cast<cuuint32_t>(box_rows), 1};
  cuuint32_t estr[3] = {1, 1, 1};
  const CUresult r = encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(act), dims, strides, box,
                            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}
bool make_act_map(CUtensorMap* map, const void* act, int rows, int cols) {
  return make_act_map_box(map, act, rows, cols, 16);
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
