// Prefill projections: Y[tok][f] = sum_k B[tok][k] W[f][k] for a whole
// prompt pass (hundreds to thousands of token rows), where the work is a
// dense contraction and the tensor pipe, not HBM, bounds it.
//
// The decode kernel (proj.cu) puts the weights on the MMA's M side and the
// few token rows on N, so each weight tile is read once per launch.  With a
// long pass that layout would re-read every weight once per 128 tokens of
// the pass; here the roles swap.  A CTA owns a tile of 128 token rows (the
// tcgen05 M dimension) by 256 output features (N):
//
//   A = activation rows, a bf16 pair hi + lo per value (two planes of the
//       activation buffer): two MMAs per K step, D += A_hi W + A_lo W, into
//       one accumulator -- the product carries the rounding of the weights
//       only, and the weight tile serves both halves of the pair;
//   B = 256 weight rows (two 128-row TMA boxes: q/k/v sections, or 128 gate
//       rows followed by the same 128 up rows).
//
// Per 64-wide K block a stage holds A_hi, A_lo (16 KB each) and B (32 KB):
// 64 KB for 2 x 128 x 256 x 64 multiply-adds.  Three stages fill the shared
// memory of one CTA per SM.  CTAs are persistent: CTA c takes tiles c,
// c + grid, ... (token tile fastest, so the CTAs running at one time share
// their weight tiles through L2 and HBM sees each weight about once per
// pass).  The 512 TMEM columns hold two 256-column accumulators, so the
// epilogue of one tile overlaps the MMAs of the next.
//
// Roles (192 threads): warp 4 issues the TMA loads, warp 5 the MMAs, warps
// 0-3 run the epilogue, one token row per thread (TMEM lane = token row):
// the row's 1/rms of the RMSNorm feeding the projection (its gain is folded
// into the activation rows), then the fused epilogue of the decode kernel's
// flavours: RoPE + q rows + K/V cache rows (QKV), residual add + next
// norm's activation rows + per-128-feature sums of squares (O, down),
// SiLU(gate) * up (gate/up).  Every wait is bounded (flag, then wind down).
#include <algorithm>

#include "common.cuh"
#include "kernels.h"

namespace dvi {

namespace {

constexpr int kPfM = 128;                         // token rows per tile (MMA M)
constexpr int kPfN = 256;                         // output features per tile (MMA N)
constexpr int kPfStages = 3;
constexpr int kPfA = kPfM * 128;                  // one plane of the activation tile: 16 KB
constexpr int kPfB = kPfN * 128;                  // weight tile: 32 KB
constexpr int kPfStage = 2 * kPfA + kPfB;         // 64 KB
constexpr int kPfSmem = kPfStages * kPfStage + 1024 /*align*/ + 256 /*barriers, TMEM slot*/;
constexpr uint32_t kPfCols = 2 * kPfN;            // two accumulators

// Weight rows of half h (0, 1) of feature tile nt: which map, which row.
// QKV: the 256 features of the tile run over [q; k; v] (each section a
// multiple of 128 rows); gate/up: half 0 = gate rows, half 1 = the same up
// rows; other flavours: rows nt*256 + h*128 of the one weight.
__device__ __forceinline__ int pf_half_row(const ProjArgs& p, int nt, int h, int& map) {
  if (p.flavor == EPI_GATEUP) {
    map = h;
    return nt * kTileRows;
  }
  const int f = nt * kPfN + h * kTileRows;
  if (p.flavor == EPI_QKV) {
    if (f < p.rows_q) { map = 0; return f; }
    if (f < p.rows_q + p.rows_k) { map = 1; return f - p.rows_q; }
    map = 2;
    return f - p.rows_q - p.rows_k;   // past rows_v: zero fill
  }
  map = 0;
  return f;
}

// Sixteen f32 values as hi and lo bf16 planes (8 values per 16-byte store).
__device__ __forceinline__ void st_act16(__nv_bfloat16* dst, size_t plane, const float (&v)[16]) {
  uint32_t hi[8], lo[8];
#pragma unroll
  for (int e = 0; e < 8; ++e) split_bf16x2(v[2 * e], v[2 * e + 1], hi[e], lo[e]);
  uint4* h4 = reinterpret_cast<uint4*>(dst);
  uint4* l4 = reinterpret_cast<uint4*>(dst + plane);
  h4[0] = make_uint4(hi[0], hi[1], hi[2], hi[3]);
  h4[1] = make_uint4(hi[4], hi[5], hi[6], hi[7]);
  l4[0] = make_uint4(lo[0], lo[1], lo[2], lo[3]);
  l4[1] = make_uint4(lo[4], lo[5], lo[6], lo[7]);
}

// Sequence and cache position of pass row n.
__device__ __forceinline__ void pf_row_pos(const ProjArgs& p, int n, int& seq, int& pos) {
  seq = p.seq0 + n / p.rows_per_seq;
  pos = p.lens[seq] + p.pos_off + n % p.rows_per_seq;
}

// QKV: RoPE (rotate-half pairs dim and dim + hd/2 of one head, both in the
// tile since sections and heads are 128-aligned), q rows in f32, k and v
// rows into the cache at the row's position.
__device__ __forceinline__ void pf_epi_qkv(const ProjArgs& p, uint32_t acc, int nt, int n, bool live, float rstd) {
  const int hd = p.head_dim, half = hd >> 1;
  int seq = 0, pos = 0;
  if (live) pf_row_pos(p, n, seq, pos);
  const bool pos_ok = pos >= 0 && pos < p.max_len;
  if (live && !pos_ok) flag_status(p.status, DVI_DEV_KV_FULL);
  const bool st = live && pos_ok;
  for (int h = 0; h < 2; ++h) {
    const int f0 = nt * kPfN + h * kTileRows;
    int sec, fl;
    if (f0 < p.rows_q) { sec = 0; fl = f0; }
    else if (f0 < p.rows_q + p.rows_k) { sec = 1; fl = f0 - p.rows_q; }
    else if (f0 < p.rows_q + p.rows_k + p.rows_v) { sec = 2; fl = f0 - p.rows_q - p.rows_k; }
    else break;
    for (int hh = 0; hh < kTileRows / hd; ++hh) {
      const int c0 = h * kTileRows + hh * hd;
      const int head = (fl + hh * hd) / hd;
      for (int j = 0; j < half; j += 16) {
        float a[16], b[16];
        tmem_ld16(acc + static_cast<uint32_t>(c0 + j), a);
        tmem_ld16(acc + static_cast<uint32_t>(c0 + half + j), b);
        if (!st) continue;
#pragma unroll
        for (int e = 0; e < 16; ++e) {
          a[e] *= rstd;
          b[e] *= rstd;
        }
        if (sec < 2) {
          const float2* cs = p.rope + static_cast<size_t>(pos) * half + j;
#pragma unroll
          for (int e = 0; e < 16; ++e) {
            const float2 r = cs[e];
            const float x1 = a[e] * r.x - b[e] * r.y;
            const float x2 = b[e] * r.x + a[e] * r.y;
            a[e] = x1;
            b[e] = x2;
          }
        }
        if (sec == 0) {
          float4* q0 = reinterpret_cast<float4*>(p.q_out + static_cast<size_t>(n) * p.ld_q + head * hd + j);
          float4* q1 = reinterpret_cast<float4*>(p.q_out + static_cast<size_t>(n) * p.ld_q + head * hd + half + j);
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            q0[e] = make_float4(a[4 * e], a[4 * e + 1], a[4 * e + 2], a[4 * e + 3]);
            q1[e] = make_float4(b[4 * e], b[4 * e + 1], b[4 * e + 2], b[4 * e + 3]);
          }
        } else {
          __nv_bfloat16* c = static_cast<__nv_bfloat16*>(sec == 1 ? p.kc : p.vc) +
                             ((static_cast<size_t>(seq) * p.n_kv_heads + head) * p.max_len + pos) * hd;
          uint32_t pa[8], pb[8];
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            pa[e] = pack_bf16x2(a[2 * e], a[2 * e + 1]);
            pb[e] = pack_bf16x2(b[2 * e], b[2 * e + 1]);
          }
          uint4* c0p = reinterpret_cast<uint4*>(c + j);
          uint4* c1p = reinterpret_cast<uint4*>(c + half + j);
          c0p[0] = make_uint4(pa[0], pa[1], pa[2], pa[3]);
          c0p[1] = make_uint4(pa[4], pa[5], pa[6], pa[7]);
          c1p[0] = make_uint4(pb[0], pb[1], pb[2], pb[3]);
          c1p[1] = make_uint4(pb[4], pb[5], pb[6], pb[7]);
        }
      }
    }
  }
}

// O and down: x += y, the next norm's activation rows x * g (hi/lo), and
// the sums of squares of the new x per 128 features (in feature order).
__device__ __forceinline__ void pf_epi_resid(const ProjArgs& p, uint32_t acc, int nt, int n, bool live) {
  for (int h = 0; h < 2; ++h) {
    const int f0 = nt * kPfN + h * kTileRows;
    if (f0 >= p.n_out) break;
    float ssq = 0.f;
    for (int j = 0; j < kTileRows; j += 16) {
      float v[16];
      tmem_ld16(acc + static_cast<uint32_t>(h * kTileRows + j), v);
      if (!live) continue;
      const int f = f0 + j;
      float4* xp = reinterpret_cast<float4*>(p.x_res + static_cast<size_t>(n) * p.ld_res + f);
      float x[16];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float4 t = __ldcg(xp + e);
        x[4 * e] = t.x + v[4 * e];
        x[4 * e + 1] = t.y + v[4 * e + 1];
        x[4 * e + 2] = t.z + v[4 * e + 2];
        x[4 * e + 3] = t.w + v[4 * e + 3];
      }
#pragma unroll
      for (int e = 0; e < 4; ++e) xp[e] = make_float4(x[4 * e], x[4 * e + 1], x[4 * e + 2], x[4 * e + 3]);
#pragma unroll
      for (int e = 0; e < 16; ++e) ssq += x[e] * x[e];
      if (p.xg_out) {
        const float4* g4 = reinterpret_cast<const float4*>(p.g_next + f);
        float y[16];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float4 g = g4[e];
          y[4 * e] = x[4 * e] * g.x;
          y[4 * e + 1] = x[4 * e + 1] * g.y;
          y[4 * e + 2] = x[4 * e + 2] * g.z;
          y[4 * e + 3] = x[4 * e + 3] * g.w;
        }
        st_act16(static_cast<__nv_bfloat16*>(p.xg_out) + static_cast<size_t>(n) * p.ld_xg + f, p.xg_plane, y);
      }
    }
    if (live) p.ss_out[static_cast<size_t>(f0 / kTileRows) * p.ss_out_ld + n] = ssq;
  }
}

// gate/up: columns [0, 128) are the gate rows, [128, 256) the up rows of the
// same 128 features; h = SiLU(gate) * up.
__device__ __forceinline__ void pf_epi_gateup(const ProjArgs& p, uint32_t acc, int nt, int n, bool live,
                                              float rstd) {
  const int f0 = nt * kTileRows;
  for (int j = 0; j < kTileRows; j += 16) {
    float g[16], u[16];
    tmem_ld16(acc + static_cast<uint32_t>(j), g);
    tmem_ld16(acc + static_cast<uint32_t>(kTileRows + j), u);
    const int f = f0 + j;
    if (!live || f >= p.n_out) continue;
    float hv[16];
#pragma unroll
    for (int e = 0; e < 16; ++e) {
      const float gt = g[e] * rstd;
      hv[e] = gt / (1.f + expf(-gt)) * (u[e] * rstd);
    }
    __nv_bfloat16* dst = static_cast<__nv_bfloat16*>(p.h_out) + static_cast<size_t>(n) * p.ld_h + f;
    if (f + 16 <= p.n_out) {
      st_act16(dst, p.h_plane, hv);
    } else {
      for (int e = 0; f + e < p.n_out; ++e) Act<__nv_bfloat16>::st(dst + e, p.h_plane, hv[e]);
    }
  }
}

}  // namespace

__global__ void __launch_bounds__(192, 1)
    proj_pf_kernel(const __grid_constant__ CUtensorMap ma, const __grid_constant__ CUtensorMap mw0,
                   const __grid_constant__ CUtensorMap mw1, const __grid_constant__ CUtensorMap mw2,
                   const ProjArgs p, int n_mtiles, int n_ntiles) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  uint8_t* ring = smem_raw + (((raw + 1023u) & ~1023u) - raw);
  uint64_t* full = reinterpret_cast<uint64_t*>(ring + kPfStages * kPfStage);
  uint64_t* empty = full + kPfStages;
  uint64_t* accf = empty + kPfStages;   // [2] accumulator b holds a finished tile
  uint64_t* acce = accf + 2;            // [2] accumulator b has been read
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(acce + 2);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n_tiles = n_mtiles * n_ntiles;
  const int nkb = p.kb_total;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kPfStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&accf[b], 1);
      mbar_init(&acce[b], 4);
    }
    mbar_fence_init();
  }
  if (warp == 0) tmem_alloc(tmem_holder, kPfCols);
  if (warp == 4 && lane == 0) {
    tma_prefetch_desc(&ma);
    tma_prefetch_desc(&mw0);
    if (p.flavor == EPI_GATEUP || p.flavor == EPI_QKV) tma_prefetch_desc(&mw1);
    if (p.flavor == EPI_QKV) tma_prefetch_desc(&mw2);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  griddep_launch();
  const uint32_t tmem = *tmem_holder;

  if (warp == 4) {
    // ---------------- TMA producer
    if (lane == 0) {
      const uint64_t pol = 0ull;   // default L2 policy: weights are re-read by the other token tiles
      auto wmap = [&](int m) { return m == 0 ? &mw0 : (m == 1 ? &mw1 : &mw2); };
      auto load_w = [&](int nt, int kb, int s) {
        for (int h = 0; h < 2; ++h) {
          int m = 0;
          const int y = pf_half_row(p, nt, h, m);
          tma_load_2d(ring + s * kPfStage + 2 * kPfA + h * (kPfB / 2), wmap(m), kb * kKBlock, y, &full[s], pol);
        }
      };
      auto load_a = [&](int mt, int kb, int s) {
        tma_load_3d(ring + s * kPfStage, &ma, kb * kKBlock, p.act_row0 + mt * kPfM, 0, &full[s], 0ull);
        tma_load_3d(ring + s * kPfStage + kPfA, &ma, kb * kKBlock, p.act_row0 + mt * kPfM, 1, &full[s], 0ull);
      };
      // The first tile's first weight blocks do not depend on earlier kernels.
      int it = 0, issued = 0;
      bool ok = true;
      const int t0 = blockIdx.x;
      const int pre = t0 < n_tiles ? min(kPfStages, nkb) : 0;
      for (int i = 0; i < pre; ++i) {
        mbar_arrive_expect_tx(&full[i], kPfStage);
        load_w(t0 / n_mtiles, i, i);
      }
      griddep_wait();
      for (int i = 0; i < pre; ++i) load_a(t0 % n_mtiles, i, i);
      it = issued = pre;
      for (int t = t0; t < n_tiles && ok; t += gridDim.x) {
        const int mt = t % n_mtiles, nt = t / n_mtiles;
        for (int kb = (t == t0 ? pre : 0); kb < nkb; ++kb, ++it) {
          const int s = it % kPfStages;
          if (!mbar_wait(&empty[s], ((it / kPfStages) & 1) ^ 1, p.status)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&full[s], kPfStage);
          load_w(nt, kb, s);
          load_a(mt, kb, s);
          issued = it + 1;
        }
      }
      // every issued copy has landed before the CTA moves on
      for (int i = max(0, issued - kPfStages); i < issued; ++i)
        mbar_wait(&full[i % kPfStages], (i / kPfStages) & 1, p.status);
    }
    __syncwarp();
  } else if (warp == 5) {
    // ---------------- MMA issuer: D += A_hi W + A_lo W per K step
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16_m128(kPfN);
      int it = 0, j = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < n_tiles && ok; t += gridDim.x, ++j) {
        const int b = j & 1;
        if (!mbar_wait(&acce[b], ((j >> 1) & 1) ^ 1, p.status)) break;
        tc_fence_after();
        const uint32_t d = tmem + static_cast<uint32_t>(b * kPfN);
        for (int kb = 0; kb < nkb; ++kb, ++it) {
          const int s = it % kPfStages;
          if (!mbar_wait(&full[s], (it / kPfStages) & 1, p.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t ahi = smem_u32(ring + s * kPfStage);
          const uint32_t alo = ahi + kPfA;
          const uint32_t bw = ahi + 2 * kPfA;
#pragma unroll
          for (int kk = 0; kk < kKBlock / 16; ++kk) {
            const uint64_t bd = smem_desc_sw128(bw + kk * 32);
            tc_mma_bf16(d, smem_desc_sw128(ahi + kk * 32), bd, idesc, (kb | kk) != 0);
            tc_mma_bf16(d, smem_desc_sw128(alo + kk * 32), bd, idesc, 1u);
          }
          tc_commit(&empty[s]);
        }
        // also after a failed wait, so the epilogue's wait ends and every
        // MMA issued has completed before the TMEM is freed
        tc_commit(&accf[b]);
      }
    }
    __syncwarp();
  } else {
    // ---------------- epilogue: warp w reads TMEM lanes (token rows) 32w..32w+31
    griddep_wait();
    const int tid = threadIdx.x;
    int j = 0;
    for (int t = blockIdx.x; t < n_tiles; t += gridDim.x, ++j) {
      const int b = j & 1;
      const int mt = t % n_mtiles, nt = t / n_mtiles;
      const int n = mt * kPfM + tid;
      const bool live = n < p.M;
      // the row's 1/rms (before the wait: it reads only earlier kernels' output)
      float rstd = 1.f;
      if (p.ss && live) {
        float sq = 0.f;
        for (int q = 0; q < p.ss_tiles; ++q) sq += __ldcg(p.ss + static_cast<size_t>(q) * p.ss_ld + n);
        rstd = rsqrtf(sq / static_cast<float>(p.d_norm) + p.eps);
      }
      if (!mbar_wait(&accf[b], (j >> 1) & 1, p.status)) break;
      tc_fence_after();
      const uint32_t acc = tmem + (static_cast<uint32_t>(warp * 32) << 16) + static_cast<uint32_t>(b * kPfN);
      if (p.flavor == EPI_QKV) pf_epi_qkv(p, acc, nt, n, live, rstd);
      else if (p.flavor == EPI_GATEUP) pf_epi_gateup(p, acc, nt, n, live, rstd);
      else pf_epi_resid(p, acc, nt, n, live);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&acce[b]);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, kPfCols);
  }
}


cudaError_t launch_proj_pf(const ProjArgs& a0, const PfMaps& m, int n_sms, cudaStream_t s) {
  static PerDevice attr;
  attr.once([] { cudaFuncSetAttribute(proj_pf_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kPfSmem); });
  ProjArgs a = a0;
  a.kb_total = (a.K + kKBlock - 1) / kKBlock;
  int n_ntiles;
  if (a.flavor == EPI_QKV) n_ntiles = (a.rows_q + a.rows_k + a.rows_v + kPfN - 1) / kPfN;
  else if (a.flavor == EPI_GATEUP) n_ntiles = (a.n_out + kTileRows - 1) / kTileRows;
  else if (a.flavor == EPI_RESID) n_ntiles = (a.n_out + kPfN - 1) / kPfN;
  else return cudaErrorInvalidValue;
  const int n_mtiles = (a.M + kPfM - 1) / kPfM;
  const int n_tiles = n_mtiles * n_ntiles;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(std::max(1, std::min(n_tiles, n_sms)));
  cfg.blockDim = dim3(192);
  cfg.dynamicSmemBytes = kPfSmem;
  cfg.stream = s;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, proj_pf_kernel, m.act, m.w0, m.w1, m.w2, a, n_mtiles, n_ntiles);
  return e != cudaSuccess ? e : cudaGetLastError();
}

}  // namespace dvi
