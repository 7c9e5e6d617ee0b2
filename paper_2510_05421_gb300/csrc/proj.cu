// Projection kernels of the split decoder (Sec. 3.1's f_{0->k}, f_{k->L} and
// both heads): Y[tok][f] = sum_k W[f][k] * B[tok][k] for a few token rows.
//
// Decode passes carry 1..256 token rows against weight matrices of up to
// 32000 x 11008, so every launch is a weight stream: each tile of 128 output
// features (the tcgen05 M dimension) is read from HBM exactly once, and the
// token rows sit on the MMA's N dimension ("swap AB").
//
// bf16 (tcgen05): warp 4 streams 128x64 weight tiles by TMA (128-byte
// swizzle) into a ring of shared-memory stages; warps 0-3 write the matching
// B tile (the token rows, RMSNorm-ed on the fly from the f32 residual stream
// or copied from a bf16 activation) in the same swizzled K-major layout;
// warp 5 issues tcgen05.mma (M=128, N=n_pad, K=16) into a TMEM accumulator
// and releases stages with tcgen05.commit.  Warps 0-3 then read TMEM and run
// the fused epilogue.
//
// f32 (FP32 FMA, no TF32): the same decomposition with a shared-memory tiled
// FFMA main loop of 16 token columns per CTA.
//
// K is split over `n_splits` CTAs per tile when there are too few tiles to
// fill the GPU.  Each split stores its partial tile; the last CTA to arrive
// (an atomic counter per tile) sums the partials in split order -- so results
// are deterministic -- and runs the epilogue.  The split plan depends only on
// the weight shape, never on the number of token rows.
#include <algorithm>
#include <cudaTypedefs.h>

#include "common.cuh"
#include "kernels.h"

namespace dvi {

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

// Fused epilogue for 16 token columns [c0, c0+16) of one 128-feature tile.
// Called by the 128 epilogue threads together (row = feature within tile).
template <typename T>
__device__ void epilogue_chunk(const ProjArgs& p, int tile, int row, int c0, const float (&v)[kChunk],
                               const float (&v2)[kChunk], EpiSmem& es) {
  const int warp = row >> 5, lane = row & 31;
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
      if (n < p.M) {
        int seq, pos;
        row_seq_pos(p, n, seq, pos);
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
    float sq[kChunk];
#pragma unroll
    for (int j = 0; j < kChunk; ++j) {
      const int n = c0 + j;
      float xn = 0.f;
      if (n < p.M && f < p.n_out) {
        float* xp = p.x_res + static_cast<size_t>(n) * p.ld_res + f;
        xn = *xp + v[j];
        *xp = xn;
      }
      sq[j] = xn * xn;
    }
#pragma unroll
    for (int j = 0; j < kChunk; ++j) {
      const float s = warp_sum(sq[j]);
      if (lane == 0) es.red[warp][j] = s;
    }
    named_bar(1, kTileRows);
    if (row < kChunk && c0 + row < p.M)
      p.ss_out[static_cast<size_t>(tile) * p.ss_out_ld + c0 + row] =
          (es.red[0][row] + es.red[1][row]) + (es.red[2][row] + es.red[3][row]);
    named_bar(1, kTileRows);
  } else if (p.flavor == EPI_GATEUP) {
    const int f = tile * kTileRows + row;
    if (f < p.n_out) {
#pragma unroll
      for (int j = 0; j < kChunk; ++j) {
        const int n = c0 + j;
        if (n < p.M) {
          const float g = v[j];
          const float h = g / (1.f + expf(-g)) * v2[j];
          DT<T>::st(static_cast<T*>(p.h_out) + static_cast<size_t>(n) * p.ld_h + f, h);
        }
      }
    }
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
        if (n < p.M) {
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
        for (int j = 0; j < kChunk; ++j)
          if (c0 + j < p.M) dst[static_cast<size_t>(c0 + j) * p.ld_logits + f] = z[j];
      }
    }
    if (p.amax) {
#pragma unroll
      for (int j = 0; j < kChunk; ++j) {
        unsigned long long key = 0;
        if (ok && c0 + j < p.M) {
          if (isfinite(z[j])) key = argmax_key(z[j], f);
          else flag_status(p.status, DVI_DEV_NONFINITE);
        }
        key = warp_max_u64(key);
        if (lane == 0) es.redk[warp][j] = key;
      }
      named_bar(1, kTileRows);
      if (row < kChunk && c0 + row < p.M) {
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

__device__ __forceinline__ uint32_t tmem_cols(int n) {
  uint32_t c = 32;
  while (c < static_cast<uint32_t>(n)) c <<= 1;
  return c;
}

// Writes one 64-wide K block of the B operand (token rows) for stage `bs`.
__device__ __forceinline__ void produce_b_tile(const ProjArgs& p, const float* rstd, uint8_t* bs, int kb,
                                               int tid) {
  const int nslots = p.n_pad * 8;
  for (int slot = tid; slot < nslots; slot += kTileRows) {
    const int n = slot >> 3, c = slot & 7;
    const int k0 = kb * kKBlock + c * 8;
    uint4 val = make_uint4(0u, 0u, 0u, 0u);
    if (n < p.M && k0 < p.K) {
      float f[8];
      const bool full8 = (k0 + 8 <= p.K);
      if (p.b_mode == B_COPY) {
        const __nv_bfloat16* src = static_cast<const __nv_bfloat16*>(p.act) + static_cast<size_t>(n) * p.ld_act + k0;
        if (full8) {
          val = *reinterpret_cast<const uint4*>(src);
        } else {
          uint32_t w[4] = {0u, 0u, 0u, 0u};
          for (int e = 0; e < 8 && k0 + e < p.K; ++e) {
            const uint32_t b = __bfloat16_as_ushort(src[e]);
            w[e >> 1] |= (e & 1) ? (b << 16) : b;
          }
          val = make_uint4(w[0], w[1], w[2], w[3]);
        }
      } else {
        const float* src = (p.b_mode == B_NORM ? p.x : static_cast<const float*>(p.act)) +
                           static_cast<size_t>(n) * (p.b_mode == B_NORM ? p.ldx : p.ld_act) + k0;
        if (full8) {
          const float4 a = *reinterpret_cast<const float4*>(src);
          const float4 b = *reinterpret_cast<const float4*>(src + 4);
          f[0] = a.x; f[1] = a.y; f[2] = a.z; f[3] = a.w; f[4] = b.x; f[5] = b.y; f[6] = b.z; f[7] = b.w;
        } else {
#pragma unroll
          for (int e = 0; e < 8; ++e) f[e] = (k0 + e < p.K) ? src[e] : 0.f;
        }
        if (p.b_mode == B_NORM) {
          const float r = rstd[n];
#pragma unroll
          for (int e = 0; e < 8; ++e) f[e] = (k0 + e < p.K) ? f[e] * r * p.gain[k0 + e] : 0.f;
        }
        val = make_uint4(pack_bf16x2(f[0], f[1]), pack_bf16x2(f[2], f[3]), pack_bf16x2(f[4], f[5]),
                         pack_bf16x2(f[6], f[7]));
      }
    }
    *reinterpret_cast<uint4*>(bs + n * 128 + ((c ^ (n & 7)) << 4)) = val;
  }
}

__device__ __forceinline__ void compute_rstd(const ProjArgs& p, float* rstd, int tid) {
  for (int n = tid; n < p.M; n += kTileRows) {
    float s = 0.f;
    for (int t = 0; t < p.ss_tiles; ++t) s += p.ss[static_cast<size_t>(t) * p.ss_ld + n];
    rstd[n] = rsqrtf(s / static_cast<float>(p.d_norm) + p.eps);
  }
}

// ------------------------------------------------------------------ tcgen05
template <bool DUAL>
__global__ void __launch_bounds__(192, 2)
    proj_tc_kernel(const __grid_constant__ CUtensorMap m0, const __grid_constant__ CUtensorMap m1,
                   const __grid_constant__ CUtensorMap m2, const ProjArgs p, int stages) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  uint8_t* base = smem_raw + (((raw + 1023u) & ~1023u) - raw);
  constexpr int abytes = DUAL ? 32768 : 16384;
  const int bbytes = p.n_pad * 128;
  uint8_t* sA = base;
  uint8_t* sB = base + stages * abytes;
  uint64_t* full = reinterpret_cast<uint64_t*>(sB + stages * bbytes);
  uint64_t* empty = full + stages;
  uint64_t* done = empty + stages;
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(done + 1);
  float* rstd = reinterpret_cast<float*>(tmem_holder + 4);
  EpiSmem& es = *reinterpret_cast<EpiSmem*>(sA);   // A stages are free once `done` fired

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int tile = blockIdx.x / p.n_splits, split = blockIdx.x % p.n_splits;
  const int kb0 = split * p.kb_per_split;
  const int nkb = min(p.kb_per_split, p.kb_total - kb0);
  const uint32_t ncols = tmem_cols(p.n_pad * (DUAL ? 2 : 1));

  if (threadIdx.x == 0) {
    for (int s = 0; s < stages; ++s) {
      mbar_init(&full[s], 5);     // TMA expect_tx arrival + one arrival per B-producer warp
      mbar_init(&empty[s], 1);    // tcgen05.commit
    }
    mbar_init(done, 1);
    mbar_fence_init();
  }
  if (warp == 0) tmem_alloc(tmem_holder, ncols);
  if (warp == 4 && lane == 0) {
    tma_prefetch_desc(&m0);
    if (DUAL || p.flavor == EPI_QKV) tma_prefetch_desc(&m1);
    if (p.flavor == EPI_QKV) tma_prefetch_desc(&m2);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_holder;

  if (warp == 4) {
    // ---------------- TMA producer (weights)
    if (lane == 0) {
      const CUtensorMap* map = &m0;
      int y = tile * kTileRows;
      if (p.flavor == EPI_QKV) {
        const int tq = p.rows_q / kTileRows, tk = p.rows_k / kTileRows;
        if (tile >= tq + tk) { map = &m2; y = (tile - tq - tk) * kTileRows; }
        else if (tile >= tq) { map = &m1; y = (tile - tq) * kTileRows; }
      }
      const uint64_t pol = l2_evict_first_policy();
      int issued = 0;
      for (int i = 0; i < nkb; ++i) {
        const int s = i % stages;
        const uint32_t ph = (i / stages) & 1;
        if (!mbar_wait(&empty[s], ph ^ 1, p.status)) break;
        mbar_arrive_expect_tx(&full[s], abytes);
        const int x = (kb0 + i) * kKBlock;
        tma_load_2d(sA + s * abytes, map, x, y, &full[s], pol);
        if (DUAL) tma_load_2d(sA + s * abytes + 16384, &m1, x, y, &full[s], pol);
        issued = i + 1;
      }
      // Drain: every issued copy has landed before this warp exits.
      for (int i = max(0, issued - stages); i < issued; ++i)
        mbar_wait(&full[i % stages], (i / stages) & 1, p.status);
    }
    return;
  }
  if (warp == 5) {
    // ---------------- MMA issuer
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16_m128(static_cast<uint32_t>(p.n_pad));
      for (int i = 0; i < nkb; ++i) {
        const int s = i % stages;
        const uint32_t ph = (i / stages) & 1;
        if (!mbar_wait(&full[s], ph, p.status)) break;
        tc_fence_after();
        const uint32_t a = smem_u32(sA + s * abytes);
        const uint32_t b = smem_u32(sB + s * bbytes);
#pragma unroll
        for (int kk = 0; kk < kKBlock / 16; ++kk) {
          const uint64_t bd = smem_desc_sw128(b + kk * 32);
          const uint32_t acc = (i | kk) != 0;
          tc_mma_bf16(tmem, smem_desc_sw128(a + kk * 32), bd, idesc, acc);
          if (DUAL) tc_mma_bf16(tmem + static_cast<uint32_t>(p.n_pad), smem_desc_sw128(a + 16384 + kk * 32), bd,
                                idesc, acc);
        }
        tc_commit(&empty[s]);
      }
      tc_commit(done);
    }
    return;
  }

  // ---------------- warps 0-3: B producer, then epilogue
  const int tid = threadIdx.x;
  if (p.b_mode == B_NORM) compute_rstd(p, rstd, tid);
  named_bar(1, kTileRows);
  for (int i = 0; i < nkb; ++i) {
    const int s = i % stages;
    const uint32_t ph = (i / stages) & 1;
    if (!mbar_wait(&empty[s], ph ^ 1, p.status)) break;
    produce_b_tile(p, rstd, sB + s * bbytes, kb0 + i, tid);
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) mbar_arrive(&full[s]);
  }

  const bool ok = mbar_wait(done, 0, p.status);
  tc_fence_after();
  const int row = tid;
  const uint32_t lane_base = tmem + ((static_cast<uint32_t>(warp) * 32u) << 16);
  const int nchunks = (p.M + kChunk - 1) / kChunk;
  float v[kChunk], v2[kChunk];
#pragma unroll
  for (int j = 0; j < kChunk; ++j) v2[j] = 0.f;
  using T = __nv_bfloat16;
  if (p.n_splits == 1) {
    for (int c = 0; c < nchunks; ++c) {
      tmem_ld16(lane_base + c * kChunk, v);
      if (DUAL) tmem_ld16(lane_base + p.n_pad + c * kChunk, v2);
      if (ok) epilogue_chunk<T>(p, tile, row, c * kChunk, v, v2, es);
    }
    tc_fence_before();
    named_bar(1, kTileRows);
    if (warp == 0) {
      tc_fence_after();
      tmem_dealloc(tmem, ncols);
    }
    return;
  }
  const size_t reg = static_cast<size_t>(kTileRows) * p.n_pad * (DUAL ? 2 : 1);
  float* mine = p.part + (static_cast<size_t>(tile) * p.n_splits + split) * reg;
  for (int c = 0; c < nchunks; ++c) {
    tmem_ld16(lane_base + c * kChunk, v);
    if (DUAL) tmem_ld16(lane_base + p.n_pad + c * kChunk, v2);
#pragma unroll
    for (int j = 0; j < kChunk; ++j) {
      const int n = c * kChunk + j;
      if (n < p.M) {
        mine[static_cast<size_t>(n) * kTileRows + row] = v[j];
        if (DUAL) mine[static_cast<size_t>(p.n_pad + n) * kTileRows + row] = v2[j];
      }
    }
  }
  tc_fence_before();
  named_bar(1, kTileRows);
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, ncols);
  }
  if (!ok) return;
  if (!split_arrive(p, tile, row, es)) return;
  const float* all = p.part + static_cast<size_t>(tile) * p.n_splits * reg;
  for (int c = 0; c < nchunks; ++c) {
#pragma unroll
    for (int j = 0; j < kChunk; ++j) {
      const int n = c * kChunk + j;
      float a = 0.f, b = 0.f;
      if (n < p.M) {
        for (int s = 0; s < p.n_splits; ++s) {
          a += __ldcg(all + s * reg + static_cast<size_t>(n) * kTileRows + row);
          if (DUAL) b += __ldcg(all + s * reg + static_cast<size_t>(p.n_pad + n) * kTileRows + row);
        }
      }
      v[j] = a;
      v2[j] = b;
    }
    epilogue_chunk<T>(p, tile, row, c * kChunk, v, v2, es);
  }
}

// ------------------------------------------------------------------ FP32 FMA
template <bool DUAL>
__global__ void __launch_bounds__(128) proj_f32_kernel(const ProjArgs p) {
  __shared__ float Ws[DUAL ? 2 : 1][kTileRows][kKBlockF32 + 1];
  __shared__ float Bs[kChunk][kKBlockF32];
  __shared__ float rstd[kChunk];
  __shared__ EpiSmem es;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int tile = blockIdx.x / p.n_splits, split = blockIdx.x % p.n_splits;
  const int ttile = blockIdx.y, c0 = ttile * kChunk;
  const int kb0 = split * p.kb_per_split;
  const int nkb = min(p.kb_per_split, p.kb_total - kb0);

  const float* w0 = static_cast<const float*>(p.w0);
  int row0 = tile * kTileRows, rows = p.n_out;
  if (p.flavor == EPI_QKV) {
    const int tq = p.rows_q / kTileRows, tk = p.rows_k / kTileRows;
    if (tile >= tq + tk) { w0 = static_cast<const float*>(p.w2); row0 = (tile - tq - tk) * kTileRows; rows = p.rows_v; }
    else if (tile >= tq) { w0 = static_cast<const float*>(p.w1); row0 = (tile - tq) * kTileRows; rows = p.rows_k; }
    else rows = p.rows_q;
  }
  const float* w1 = static_cast<const float*>(p.w1);
  if (p.b_mode == B_NORM && tid < kChunk) {
    const int n = c0 + tid;
    float s = 0.f;
    if (n < p.M)
      for (int t = 0; t < p.ss_tiles; ++t) s += p.ss[static_cast<size_t>(t) * p.ss_ld + n];
    rstd[tid] = rsqrtf(s / static_cast<float>(p.d_norm) + p.eps);
  }
  __syncthreads();
  float acc[kChunk], acc2[kChunk];
#pragma unroll
  for (int j = 0; j < kChunk; ++j) { acc[j] = 0.f; acc2[j] = 0.f; }
  for (int i = 0; i < nkb; ++i) {
    const int k = (kb0 + i) * kKBlockF32 + lane;
    for (int q = 0; q < kTileRows / 4; ++q) {
      const int r = warp + 4 * q;
      const int grow = row0 + r;
      const bool in = grow < rows && k < p.K;
      Ws[0][r][lane] = in ? w0[static_cast<size_t>(grow) * p.K + k] : 0.f;
      if (DUAL) Ws[DUAL ? 1 : 0][r][lane] = in ? w1[static_cast<size_t>(grow) * p.K + k] : 0.f;
    }
    for (int e = 0; e < (kChunk * kKBlockF32) / 128; ++e) {
      const int idx = tid + 128 * e;
      const int j = idx / kKBlockF32, kk = idx % kKBlockF32;
      const int n = c0 + j, kg = (kb0 + i) * kKBlockF32 + kk;
      float val = 0.f;
      if (n < p.M && kg < p.K) {
        if (p.b_mode == B_NORM) val = p.x[static_cast<size_t>(n) * p.ldx + kg] * rstd[j] * p.gain[kg];
        else val = static_cast<const float*>(p.act)[static_cast<size_t>(n) * p.ld_act + kg];
      }
      Bs[j][kk] = val;
    }
    __syncthreads();
#pragma unroll 8
    for (int kk = 0; kk < kKBlockF32; ++kk) {
      const float w = Ws[0][tid][kk];
#pragma unroll
      for (int j = 0; j < kChunk; ++j) acc[j] = fmaf(w, Bs[j][kk], acc[j]);
      if (DUAL) {
        const float w2 = Ws[DUAL ? 1 : 0][tid][kk];
#pragma unroll
        for (int j = 0; j < kChunk; ++j) acc2[j] = fmaf(w2, Bs[j][kk], acc2[j]);
      }
    }
    __syncthreads();
  }
  const int row = tid;
  if (p.n_splits == 1) {
    epilogue_chunk<float>(p, tile, row, c0, acc, acc2, es);
    return;
  }
  const size_t reg = static_cast<size_t>(kTileRows) * kChunk * (DUAL ? 2 : 1);
  const int ci = tile * p.n_ttiles + ttile;
  float* mine = p.part + (static_cast<size_t>(ci) * p.n_splits + split) * reg;
#pragma unroll
  for (int j = 0; j < kChunk; ++j) {
    mine[j * kTileRows + row] = acc[j];
    if (DUAL) mine[(kChunk + j) * kTileRows + row] = acc2[j];
  }
  if (!split_arrive(p, ci, row, es)) return;
  const float* all = p.part + static_cast<size_t>(ci) * p.n_splits * reg;
#pragma unroll
  for (int j = 0; j < kChunk; ++j) {
    float a = 0.f, b = 0.f;
    for (int s = 0; s < p.n_splits; ++s) {
      a += __ldcg(all + s * reg + j * kTileRows + row);
      if (DUAL) b += __ldcg(all + s * reg + (kChunk + j) * kTileRows + row);
    }
    acc[j] = a;
    acc2[j] = b;
  }
  epilogue_chunk<float>(p, tile, row, c0, acc, acc2, es);
}

// ------------------------------------------------------------------ host
void plan_splits(ProjArgs& a, int n_sms, bool tc) {
  if (a.flavor == EPI_QKV)
    a.n_tiles = a.rows_q / kTileRows + a.rows_k / kTileRows + a.rows_v / kTileRows;
  else
    a.n_tiles = (a.n_out + kTileRows - 1) / kTileRows;
  const int kbw = tc ? kKBlock : kKBlockF32;
  a.kb_total = (a.K + kbw - 1) / kbw;
  const int slots = (tc ? 2 : 4) * n_sms;
  const int min_kb = tc ? 4 : 2;
  int best_s = 1, best_kbps = a.kb_total;
  double best_cost = 1e30;
  for (int s = 1; s <= 32 && s <= a.kb_total; ++s) {
    const int kbps = (a.kb_total + s - 1) / s;
    if (s > 1 && kbps < min_kb) break;
    const int s_eff = (a.kb_total + kbps - 1) / kbps;
    const long units = static_cast<long>(a.n_tiles) * s_eff;
    const long waves = (units + slots - 1) / slots;
    const double cost = static_cast<double>(waves) * (kbps + 2);
    if (cost < best_cost - 1e-9) { best_cost = cost; best_s = s_eff; best_kbps = kbps; }
  }
  a.n_splits = best_s;
  a.kb_per_split = best_kbps;
}

size_t proj_partial_floats(const ProjArgs& a, bool tc) {
  if (a.n_splits <= 1) return 0;
  const int dual = a.flavor == EPI_GATEUP ? 2 : 1;
  const int ntt = tc ? 1 : (a.M + kChunk - 1) / kChunk;
  const int cols = tc ? a.n_pad : kChunk;
  return static_cast<size_t>(a.n_tiles) * ntt * a.n_splits * kTileRows * cols * dual;
}

static int tc_stages(int n_pad, bool dual, size_t* smem_bytes) {
  const int per = (dual ? 32768 : 16384) + n_pad * 128;
  const int fixed = 1024 /*align*/ + 1024 /*barriers, tmem slot, rstd*/ + 4 * kMaxTokens;
  int stages = (112 * 1024 - fixed) / per;
  if (stages < 3) stages = (220 * 1024 - fixed) / per;
  stages = std::min(stages, 8);
  stages = std::max(stages, 2);
  *smem_bytes = static_cast<size_t>(fixed) + static_cast<size_t>(stages) * per;
  return stages;
}

cudaError_t launch_proj(const ProjArgs& a, const ProjMaps* maps, cudaStream_t s) {
  if (a.dtype == DVI_BF16) {
    const bool dual = a.flavor == EPI_GATEUP;
    size_t smem = 0;
    const int stages = tc_stages(a.n_pad, dual, &smem);
    dim3 grid(a.n_tiles * a.n_splits);
    if (dual) {
      static bool attr = false;
      if (!attr) {
        cudaFuncSetAttribute(proj_tc_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024);
        attr = true;
      }
      proj_tc_kernel<true><<<grid, 192, smem, s>>>(maps->m0, maps->m1, maps->m2, a, stages);
    } else {
      static bool attr = false;
      if (!attr) {
        cudaFuncSetAttribute(proj_tc_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024);
        attr = true;
      }
      proj_tc_kernel<false><<<grid, 192, smem, s>>>(maps->m0, maps->m1, maps->m2, a, stages);
    }
  } else {
    ProjArgs b = a;
    b.n_ttiles = (a.M + kChunk - 1) / kChunk;
    dim3 grid(a.n_tiles * a.n_splits, b.n_ttiles);
    if (a.flavor == EPI_GATEUP) proj_f32_kernel<true><<<grid, 128, 0, s>>>(b);
    else proj_f32_kernel<false><<<grid, 128, 0, s>>>(b);
  }
  return cudaGetLastError();
}

bool make_weight_map(CUtensorMap* map, const void* w, int rows, int cols) {
  static PFN_cuTensorMapEncodeTiled_v12000 encode = nullptr;
  if (!encode) {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) !=
            cudaSuccess ||
        q != cudaDriverEntryPointSuccess || !fn)
      return false;
    encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  }
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(cols) * 2};
  cuuint32_t box[2] = {kKBlock, kTileRows};
  cuuint32_t estr[2] = {1, 1};
  const CUresult r = encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(w), dims, strides, box,
                            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

}  // namespace dvi
