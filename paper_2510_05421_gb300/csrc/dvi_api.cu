// C-ABI of the DVI library (include/dvi.h): context, workspace layout and the
// order in which the kernels of each call are enqueued.
//
//  prefill              chunks of the prompt through layers 1..L, verifier head
//                       on the last row -> first committed token (Sec. 3.1)
//  draft_verify_commit  K draft passes (layers 1..k + drafter head), one verify
//                       pass (layers k+1..L on the K rows + LM head), accept /
//                       commit / rollback / log (Sec. 3.3); captured once into
//                       a CUDA graph and replayed (all state is device-side)
//  update_drafter       the KL->RL update of the drafter head (Sec. 3.4)
//  ar_step              greedy AR step of the full model (Sec. 4.1 baseline)
#include <cmath>
#include <cstdio>
#include <cstring>
#include <limits>
#include <string>
#include <vector>

#include "common.cuh"
#include "kernels.h"

using namespace dvi;

namespace {

struct LayerMaps {
  ProjMaps qkv, o, gu, down;
  CUtensorMap gate128, up128;   // gate / up with 128-row boxes (prefill kernel)
};

// One pass of token rows through layers: the f32 residual stream x, its
// per-tile sums of squares ss, and xg = x * g (the next projection's
// activation rows in the model dtype) with its TMA descriptor.
struct Pass {
  float* x;
  float* ss;
  int ss_ld;
  int M;
  int rows_per_seq;
  int seq0;
  int n_seqs;
  int pos_off;
  void* xg;
  const CUtensorMap* xg_map;
  bool pf = false;   // a bf16 prompt pass: projections on the prefill kernel
};

struct Plan {
  int n_tiles, n_splits, kb_total, kb_per_split;
};

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

}  // namespace

struct dvi_ctx {
  dvi_model_config cfg;
  dvi_runtime_config rt;
  dvi_weights w;
  std::vector<dvi_layer_weights> layers;
  cudaStream_t stream = nullptr;
  int n_sms = 152;
  bool tc = false;
  size_t esz = 4;
  int L, d, Hq, Hkv, hd, F, V, k, r, B, K, max_len, cap_steps, cap_rows, chunk, M_max, nq, nkv;
  int pf_rows;   // rows of the prompt-pass buffers: chunk, rounded up to 128 for bf16
  int Kv;   // verify rows per sequence: K, or K + 1 with the bonus row
  // device state
  int *lens, *pending, *draft_ids, *status, *log_step, *log_meta;
  long long* counters;
  float* dev_state;
  int* upd_ctr;   // [4 + cap_rows] the update kernels' counters and grid barrier
  int* fin_ctr;   // arrivals of a head projection's CTAs (finalize in its last CTA)
  // chained launches of a bf16 decode pass: one completion counter per
  // launch, cleared by a memset at the pass's start
  int* dep_ctr = nullptr;
  int n_dep_ctr = 0;
  bool dep_on = false;
  int dep_slot = 0;
  int* dep_prev = nullptr;   // counter of the previous launch, if it signals
  int dep_prev_count = 0;    // that launch's CTAs
  float *x_dr, *ss_dr, *x_ver, *ss_ver, *x_pf, *ss_pf, *q, *bu;
  void *xg_dr, *xg_ver, *xg_pf, *attn_o, *ffn_h;
  unsigned long long* amax;
  void *kcache, *vcache;
  float2* rope;
  float* part;
  size_t part_floats;
  int* proj_counters;
  int n_proj_counters;
  float* attn_part;
  size_t attn_part_floats;
  int* attn_ctr;
  int n_attn_ctr;
  int attn_split_len, attn_nsplits;
  int dec_nsplits;                  // bf16 decode attention: splits (one cluster) per KV head
  int chain_ctas = 0;               // persistent projection chain: grid size (0: not used)
  // draft-phase megakernel (runtime option megakernel): the static part of
  // its arguments, its scratch, and whether it runs (bf16, eligible shapes,
  // one CTA per SM resident)
  bool mk_sized = false;
  bool mk_on = false;
  MkArgs mk{};
  size_t mk_sync_bytes = 0;
  void* mk_sync = nullptr;   // argmax keys, then the completion counters and abort flag
  CUtensorMap* mk_maps_dev = nullptr;   // the kernel's weight descriptors (workspace)
  std::vector<CUtensorMap> mk_maps;     // their host copy (source of the upload)
  float* chain_part = nullptr;
  size_t chain_part_floats = 0;
  int* chain_ctr = nullptr;
  void* log_u;
  float* log_logits;
  float *Z, *rowstat, *stat_part, *coef, *ub, *ga, *ga_part;
  float *m_a, *v_a, *m_b, *v_b, *grad_a, *grad_b;
  // full-head mode (head_mode 1): f32 master of W^S (bf16 only), Adam
  // moments, per-row logit gradients G, the optional gradient copy
  float *w_master = nullptr, *m_w = nullptr, *v_w = nullptr, *G = nullptr, *grad_w = nullptr;
  int *out_ids, *n_committed, *n_accepted, *ar_out;
  size_t ws_bytes;
  void* ws;
  // plans and TMA descriptors
  Plan p_qkv, p_o, p_gu, p_down, p_head;
  std::vector<LayerMaps> maps;
  ProjMaps head_v, head_s;
  // TMA descriptors of the activation buffers (bf16 model)
  CUtensorMap map_xg_dr, map_xg_ver, map_xg_pf, map_attn_o, map_ffn_h, map_log_u;
  // the prompt-pass activation buffers with 128-row boxes (prefill kernel)
  CUtensorMap map_pf_xg, map_pf_attn_o, map_pf_ffn_h;
  CUtensorMap map_kc, map_vc;   // K / V caches as [L*B*H_kv*max_len][hd]
  int log_enabled = 1;
  // graphs of one decode step: the K draft passes, then the verify pass
  cudaGraphExec_t draft_exec = nullptr, verify_exec = nullptr;
  cudaGraphExec_t ar_exec = nullptr;   // one greedy AR step of the full model
  int step_calls = 0, ar_calls = 0;
  long long draft_launches = 0, verify_launches = 0, ar_launches = 0;
  long long launches = 0;
  // optional per-phase timing (0 draft, 1 verify, 2 update): event pairs
  int timing = 0;
  std::vector<cudaEvent_t> ev_pool;
  std::vector<std::pair<int, std::pair<cudaEvent_t, cudaEvent_t>>> ev_marks;
  std::string err;
};

namespace {

dvi_status fail(dvi_ctx* c, dvi_status s, const char* msg) {
  if (c) c->err = msg;
  return s;
}

#define DVI_CUDA(call)                                                                 \
  do {                                                                                 \
    cudaError_t e_ = (call);                                                           \
    if (e_ != cudaSuccess) {                                                           \
      ctx->err = std::string(#call) + ": " + cudaGetErrorString(e_);                   \
      return DVI_ERR_CUDA;                                                             \
    }                                                                                  \
  } while (0)

bool valid_config(const dvi_model_config* c, const dvi_runtime_config* rt, std::string* why) {
  auto bad = [&](const char* m) { if (why) *why = m; return false; };
  if (!c || !rt) return bad("null config");
  if (c->dtype != DVI_F32 && c->dtype != DVI_BF16) return bad("dtype must be DVI_F32 or DVI_BF16");
  if (c->n_layers < 1 || c->d_model < 128 || c->d_model % 128) return bad("d_model must be a positive multiple of 128");
  if (c->n_heads < 1 || c->n_kv_heads < 1 || c->n_heads % c->n_kv_heads) return bad("n_kv_heads must divide n_heads");
  if (c->head_dim != 64 && c->head_dim != 128) return bad("head_dim must be 64 or 128");
  if ((c->n_heads * c->head_dim) % 128 || (c->n_kv_heads * c->head_dim) % 128)
    return bad("H*head_dim must be multiples of 128");
  if (c->n_heads / c->n_kv_heads > kAttnQ) return bad("GQA group larger than 16");
  if (c->d_ffn < 1 || c->vocab < 2) return bad("bad d_ffn / vocab");
  if (c->dtype == DVI_BF16 && c->d_ffn % 8) return bad("bf16 needs d_ffn % 8 == 0");
  if (c->split_k < 1 || c->split_k > c->n_layers) return bad("split_k must be in [1, n_layers]");
  if (c->lora_rank < 0 || c->lora_rank > 64) return bad("lora_rank must be in [0, 64]");
  if (!(c->rms_eps > 0.f) || !(c->rope_theta > 0.f)) return bad("bad rms_eps / rope_theta");
  if (rt->batch < 1 || rt->batch > 64) return bad("batch must be in [1, 64]");
  if (rt->k_spec < 1 || rt->k_spec > 16) return bad("k_spec must be in [1, 16]");
  if (rt->bonus != 0 && rt->bonus != 1) return bad("bonus must be 0 or 1");
  if (rt->persistent != 0 && rt->persistent != 1) return bad("persistent must be 0 or 1");
  if (rt->chain_counters != 0 && rt->chain_counters != 1) return bad("chain_counters must be 0 or 1");
  if (rt->megakernel != 0 && rt->megakernel != 1) return bad("megakernel must be 0 or 1");
  if (rt->k_spec + rt->bonus > 16) return bad("k_spec + bonus must be <= 16");
  if (rt->max_seq_len < rt->k_spec + 2) return bad("max_seq_len too small");
  if (rt->log_steps < 1 || rt->log_steps * rt->batch * rt->k_spec > kMaxTokens)
    return bad("log_steps * batch * k_spec must be in [1, 256]");
  if (rt->head_mode != 0 && rt->head_mode != 1) return bad("head_mode must be 0 (LoRA) or 1 (full W^S)");
  if (rt->max_prefill_chunk && (rt->max_prefill_chunk < 16 || rt->max_prefill_chunk % 16 ||
                                 rt->max_prefill_chunk > (c->dtype == DVI_BF16 ? kMaxPrefillChunk : 128)))
    return bad("max_prefill_chunk must be a multiple of 16 in 16..4096 (bf16) or 16..128 (f32)");
  if (rt->batch * (rt->k_spec + rt->bonus) > kMaxTokens) return bad("batch * (k_spec + bonus) > 256");
  return true;
}

// The one place the workspace layout is defined: walks the buffers in order,
// either measuring (base == nullptr) or assigning pointers.
size_t layout(dvi_ctx* c, char* base) {
  size_t off = 0;
  auto take = [&](size_t bytes) -> char* {
    off = align_up(off, 256);
    char* p = base ? base + off : nullptr;
    off += bytes;
    return p;
  };
  const size_t e = c->esz;
  const int B = c->B, K = c->K, d = c->d, V = c->V, r = c->r;
  const int st = d / kTileRows;
  c->lens = reinterpret_cast<int*>(take(sizeof(int) * B));
  c->pending = reinterpret_cast<int*>(take(sizeof(int) * B));
  c->draft_ids = reinterpret_cast<int*>(take(sizeof(int) * B * (K + 1)));
  c->status = reinterpret_cast<int*>(take(sizeof(int) * 4));
  c->log_step = reinterpret_cast<int*>(take(sizeof(int) * 4));
  c->log_meta = reinterpret_cast<int*>(take(sizeof(int) * 6 * c->cap_rows));
  c->counters = reinterpret_cast<long long*>(take(sizeof(long long) * 8));
  c->dev_state = reinterpret_cast<float*>(take(sizeof(float) * 16));
  c->upd_ctr = reinterpret_cast<int*>(take(sizeof(int) * (4 + c->cap_rows)));
  c->fin_ctr = reinterpret_cast<int*>(take(sizeof(int) * 4));
  c->dep_ctr = reinterpret_cast<int*>(take(sizeof(int) * c->n_dep_ctr));
  c->x_dr = reinterpret_cast<float*>(take(sizeof(float) * B * d));
  c->ss_dr = reinterpret_cast<float*>(take(sizeof(float) * st * B));
  c->x_ver = reinterpret_cast<float*>(take(sizeof(float) * B * c->Kv * d));
  c->ss_ver = reinterpret_cast<float*>(take(sizeof(float) * st * B * c->Kv));
  c->x_pf = reinterpret_cast<float*>(take(sizeof(float) * c->pf_rows * d));
  c->ss_pf = reinterpret_cast<float*>(take(sizeof(float) * st * c->pf_rows));
  // activation rows feeding matrix products: bf16 keeps a hi and a lo plane
  const size_t pl = c->tc ? 2 : 1;
  c->xg_dr = take(pl * e * B * d);
  c->xg_ver = take(pl * e * B * c->Kv * d);
  c->xg_pf = take(pl * e * c->pf_rows * d);
  c->q = reinterpret_cast<float*>(take(sizeof(float) * c->M_max * c->nq));
  c->bu = reinterpret_cast<float*>(take(sizeof(float) * c->M_max * (r > 0 ? r : 1)));
  c->attn_o = take(pl * e * c->M_max * c->nq);
  c->ffn_h = take(pl * e * c->M_max * c->F);
  c->amax = reinterpret_cast<unsigned long long*>(take(sizeof(unsigned long long) * c->M_max));
  const size_t kv = static_cast<size_t>(c->L) * B * c->Hkv * c->max_len * c->hd;
  c->kcache = take(e * kv);
  c->vcache = take(e * kv);
  c->rope = reinterpret_cast<float2*>(take(sizeof(float2) * static_cast<size_t>(c->max_len) * (c->hd / 2)));
  c->part = reinterpret_cast<float*>(take(sizeof(float) * c->part_floats));
  c->proj_counters = reinterpret_cast<int*>(take(sizeof(int) * c->n_proj_counters));
  c->attn_part = reinterpret_cast<float*>(take(sizeof(float) * c->attn_part_floats));
  c->attn_ctr = reinterpret_cast<int*>(take(sizeof(int) * c->n_attn_ctr));
  c->chain_part = reinterpret_cast<float*>(take(sizeof(float) * c->chain_part_floats));
  c->chain_ctr = reinterpret_cast<int*>(take(sizeof(int) * (kChainMax + kChainMax * kChainTiles + 4)));
  c->log_u = take(pl * e * c->cap_rows * d);
  c->log_logits = reinterpret_cast<float*>(take(sizeof(float) * static_cast<size_t>(c->cap_rows) * V));
  c->Z = reinterpret_cast<float*>(take(sizeof(float) * static_cast<size_t>(c->cap_rows) * V));
  c->rowstat = reinterpret_cast<float*>(take(sizeof(float) * c->cap_rows * 8));
  c->stat_part = reinterpret_cast<float*>(take(sizeof(float) * c->cap_rows * ((V + 2047) / 2048) * 9));
  c->coef = reinterpret_cast<float*>(take(sizeof(float) * c->cap_rows * 8));
  const int rr = r > 0 ? r : 1;
  c->ub = reinterpret_cast<float*>(take(sizeof(float) * c->cap_rows * rr));
  c->ga = reinterpret_cast<float*>(take(sizeof(float) * c->cap_rows * rr));
  // partials of G A: one per 128-entry vocabulary tile (separate kernels) or
  // one per CTA of the fused update (at most 256)
  const int nvt = std::max((V + 127) / 128, 256);
  c->ga_part = reinterpret_cast<float*>(take(sizeof(float) * static_cast<size_t>(nvt) * c->cap_rows * rr));
  c->m_a = reinterpret_cast<float*>(take(sizeof(float) * static_cast<size_t>(V) * rr));
  c->v_a = reinterpret_cast<float*>(take(sizeof(float) * static_cast<size_t>(V) * rr));
  c->grad_a = reinterpret_cast<float*>(take(sizeof(float) * static_cast<size_t>(V) * rr));
  c->m_b = reinterpret_cast<float*>(take(sizeof(float) * static_cast<size_t>(rr) * d));
  c->v_b = reinterpret_cast<float*>(take(sizeof(float) * static_cast<size_t>(rr) * d));
  c->grad_b = reinterpret_cast<float*>(take(sizeof(float) * static_cast<size_t>(rr) * d));
  if (c->rt.head_mode == 1) {
    const size_t vd = static_cast<size_t>(V) * d;
    c->w_master = c->tc ? reinterpret_cast<float*>(take(sizeof(float) * vd)) : nullptr;
    c->m_w = reinterpret_cast<float*>(take(sizeof(float) * vd));
    c->v_w = reinterpret_cast<float*>(take(sizeof(float) * vd));
    c->grad_w = reinterpret_cast<float*>(take(sizeof(float) * vd));
    c->G = reinterpret_cast<float*>(take(sizeof(float) * static_cast<size_t>(c->cap_rows) * V));
  }
  c->out_ids = reinterpret_cast<int*>(take(sizeof(int) * B * c->Kv));
  c->n_committed = reinterpret_cast<int*>(take(sizeof(int) * B));
  c->n_accepted = reinterpret_cast<int*>(take(sizeof(int) * B));
  c->ar_out = reinterpret_cast<int*>(take(sizeof(int) * B));
  if (c->mk_sized) {
    MkArgs& a = c->mk;
    const size_t nqkv = static_cast<size_t>(c->Hq + 2 * c->Hkv) * c->hd;
    a.xr = reinterpret_cast<float*>(take(sizeof(float) * 2 * B * d));
    a.qkv = reinterpret_cast<float*>(take(sizeof(float) * B * nqkv));
    a.att = reinterpret_cast<float*>(take(sizeof(float) * B * c->Hq * a.P * (c->hd + 2)));
    a.ao = reinterpret_cast<float*>(take(sizeof(float) * B * d));
    a.hbuf = reinterpret_cast<float*>(take(sizeof(float) * B * c->F));
    a.y = reinterpret_cast<float*>(take(sizeof(float) * B * d));
    a.bu_part = reinterpret_cast<float*>(take(sizeof(float) * c->n_sms * B * (r > 0 ? r : 1)));
    c->mk_sync = take(c->mk_sync_bytes);
    c->mk_maps_dev = reinterpret_cast<CUtensorMap*>(take(sizeof(CUtensorMap) * (7 * c->k + 3)));
    a.keys = reinterpret_cast<unsigned long long*>(c->mk_sync);
    a.ctr = c->mk_sync ? reinterpret_cast<int*>(static_cast<char*>(c->mk_sync) +
                                                sizeof(unsigned long long) * c->Kv * B)
                       : nullptr;
  }
  return align_up(off, 256);
}

Plan plan_for(dvi_ctx* c, int flavor, int n_out, int K, int rq, int rk, int rv) {
  ProjArgs a{};
  a.flavor = flavor;
  a.n_out = n_out;
  a.K = K;
  a.rows_q = rq;
  a.rows_k = rk;
  a.rows_v = rv;
  plan_splits(a, c->n_sms, c->tc);
  return Plan{a.n_tiles, a.n_splits, a.kb_total, a.kb_per_split};
}

void size_mk(dvi_ctx* c);

void size_scratch(dvi_ctx* c) {
  const int Ms[2] = {c->M_max, 1};
  size_t part = 0;
  int ctr = 0;
  const Plan* plans[5] = {&c->p_qkv, &c->p_o, &c->p_gu, &c->p_down, &c->p_head};
  const int flav[5] = {EPI_QKV, EPI_RESID, EPI_GATEUP, EPI_RESID, EPI_HEAD};
  for (int i = 0; i < 5; ++i) {
    for (int M : Ms) {
      ProjArgs a{};
      a.flavor = flav[i];
      a.M = M;
      a.n_pad = (M + 15) / 16 * 16;
      a.n_tiles = plans[i]->n_tiles;
      a.n_splits = plans[i]->n_splits;
      part = std::max(part, proj_partial_floats(a, c->tc));
      const int ntt = c->tc ? 1 : (M + kChunk - 1) / kChunk;
      ctr = std::max(ctr, a.n_tiles * ntt);
    }
  }
  // room for dvi_linear on modest shapes: 8 Mi floats of partials
  c->part_floats = std::max(part, static_cast<size_t>(8) << 20);
  c->n_proj_counters = std::max(ctr, 4096);
  // attention: fixed split length from the capacity so row results do not
  // depend on the number of rows; about 4 CTAs per SM at full length.
  const int target = 4 * c->n_sms;
  int splits = std::max(1, target / std::max(1, c->B * c->Hkv));
  int sl = (c->max_len + splits - 1) / splits;
  sl = std::max(kAttnBlk, (sl + kAttnBlk - 1) / kAttnBlk * kAttnBlk);
  c->attn_split_len = sl;
  c->attn_nsplits = (c->max_len + sl - 1) / sl;
  // bf16 decode: the splits of a KV head form one cluster of at most 8; each
  // split takes an even share of every row's own positions
  c->dec_nsplits = std::max(1, std::min(8, target / std::max(1, c->B * c->Hkv)));
  AttnArgs at{};
  at.n_heads = c->Hq;
  at.n_kv_heads = c->Hkv;
  at.head_dim = c->hd;
  at.n_splits_max = c->attn_nsplits;
  size_t ap = 0;
  int ac = 0;
  const int rps[3] = {c->K, 1, c->chunk};
  const int nse[3] = {c->B, c->B, 1};
  for (int i = 0; i < 3; ++i) {
    at.rows_per_seq = rps[i];
    at.n_seqs = nse[i];
    ap = std::max(ap, attn_partial_floats(at));
    ac = std::max(ac, attn_counters(at));
  }
  // the bf16 tensor-core attention (GQA groups up to 8) combines its splits
  // through distributed shared memory and needs no global scratch
  const bool cluster_attn = c->tc && c->Hq / c->Hkv <= 8;
  c->attn_part_floats = cluster_attn ? 0 : ap;
  c->n_attn_ctr = cluster_attn ? 1 : ac;
  // persistent projection chain (runtime option; bf16 passes of up to
  // kChainMaxPad rows): as many CTAs as the SMs keep resident at every n_pad
  c->chain_ctas = 0;
  c->chain_part_floats = 0;
  if (c->tc && c->rt.persistent) {
    int per_sm = 2;
    for (int np = 16; np <= kChainMaxPad; np += 16) per_sm = std::min(per_sm, chain_ctas_per_sm(np));
    const int max_tiles =
        std::max(std::max(c->p_qkv.n_tiles, c->p_o.n_tiles), std::max(c->p_gu.n_tiles, c->p_down.n_tiles));
    if (per_sm > 0 && max_tiles <= kChainTiles) {
      c->chain_ctas = per_sm * c->n_sms;
      c->chain_part_floats = chain_partial_floats(max_tiles, c->chain_ctas, kChainMaxPad);
    }
  }
  size_mk(c);
}

// The draft-phase megakernel's static arguments and scratch (runtime option
// megakernel): bf16, at most kMkMaxRows sequences, k <= kMkMaxLayers shallow
// layers, GQA groups of 1, 2, 4 or 8 (8 only at head_dim 64), d a multiple of
// 128, d_ffn of 64, a cache of fewer than 2^31 - 65536 rows (its KV boxes
// take a 32-bit row, and a range's last chunk may start past max_seq_len
// when the cache is full), and a ring of at least four 16 KB stages beside
// the kernel's other
// shared memory.  No context bound: its attention streams each unit's range
// at the ring's pace (measured ahead of the per-kernel draft path from 1K to
// 16K positions).
void size_mk(dvi_ctx* c) {
  c->mk_sized = false;
  if (!c->tc || !c->rt.megakernel || c->B > kMkMaxRows || c->k > kMkMaxLayers || c->Hq / c->Hkv > kMkMaxGroup ||
      c->d % 128 || c->F % 64 || (c->hd != 64 && c->hd != 128) || c->B * c->Hkv > c->n_sms ||
      (c->Hq / c->Hkv != 1 && c->Hq / c->Hkv != 2 && c->Hq / c->Hkv != 4 && c->Hq / c->Hkv != 8) ||
      (c->hd == 128 && c->Hq / c->Hkv == 8) ||
      static_cast<long long>(c->L) * c->B * c->Hkv * c->max_len + 65536 > std::numeric_limits<int>::max())
    return;
  MkArgs& a = c->mk;
  a = MkArgs{};
  a.B = c->B;
  a.k = c->k;
  a.d = c->d;
  a.Hq = c->Hq;
  a.Hkv = c->Hkv;
  a.hd = c->hd;
  a.F = c->F;
  a.V = c->V;
  a.max_len = c->max_len;
  a.K = c->K;
  a.Kv = c->Kv;
  a.r = c->r;
  a.eps = c->cfg.rms_eps;
  a.gamma = c->cfg.lora_gamma;
  a.P = std::max(1, std::min(16, c->n_sms / (c->B * c->Hkv)));
  a.mode = MK_DRAFT;
  a.rows_max = mk_rows_max(a, c->n_sms);
  a.n_bound = mk_bounds(a);
  MkArgs ar = a;
  ar.mode = MK_AR;
  a.n_bound = std::max(a.n_bound, mk_bounds(ar));
  a.n_stages = 0;
  for (int ns = 12; ns >= 4 && !a.n_stages; --ns)
    if (mk_smem_bytes(a, ns) <= 227 * 1024) a.n_stages = ns;
  if (!a.n_stages) return;
  c->mk_sync_bytes = sizeof(unsigned long long) * c->Kv * c->B + sizeof(int) * (a.n_bound + 1);
  c->mk_sized = true;
}

bool init_dims(dvi_ctx* c, const dvi_model_config* cfg, const dvi_runtime_config* rt) {
  c->cfg = *cfg;
  c->rt = *rt;
  c->L = cfg->n_layers;
  c->d = cfg->d_model;
  c->Hq = cfg->n_heads;
  c->Hkv = cfg->n_kv_heads;
  c->hd = cfg->head_dim;
  c->F = cfg->d_ffn;
  c->V = cfg->vocab;
  c->k = cfg->split_k;
  c->r = cfg->lora_rank;
  c->B = rt->batch;
  c->K = rt->k_spec;
  c->max_len = rt->max_seq_len;
  c->cap_steps = rt->log_steps;
  c->cap_rows = rt->log_steps * rt->batch * rt->k_spec;
  c->chunk = rt->max_prefill_chunk ? rt->max_prefill_chunk : (cfg->dtype == DVI_BF16 ? 1024 : 128);
  c->pf_rows = cfg->dtype == DVI_BF16 ? (c->chunk + 127) / 128 * 128 : c->chunk;
  c->Kv = c->K + (rt->bonus ? 1 : 0);
  c->M_max = std::max(std::max(c->B * c->Kv, c->pf_rows), std::max(c->cap_rows, c->B));
  // launches of the longest decode pass: the draft phase (Kv passes of k
  // layers and a head), the verify pass, or an AR step
  c->n_dep_ctr = std::max(c->Kv * (5 * c->k + 3), 5 * c->L + 3) + 8;
  c->nq = c->Hq * c->hd;
  c->nkv = c->Hkv * c->hd;
  c->tc = cfg->dtype == DVI_BF16;
  c->esz = c->tc ? 2 : 4;
  int dev = 0;
  if (cudaGetDevice(&dev) == cudaSuccess) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess && n > 0) c->n_sms = n;
  }
  c->p_qkv = plan_for(c, EPI_QKV, 0, c->d, c->nq, c->nkv, c->nkv);
  c->p_o = plan_for(c, EPI_RESID, c->d, c->nq, 0, 0, 0);
  c->p_gu = plan_for(c, EPI_GATEUP, c->F, c->d, 0, 0, 0);
  c->p_down = plan_for(c, EPI_RESID, c->d, c->F, 0, 0, 0);
  c->p_head = plan_for(c, EPI_HEAD, c->V, c->d, 0, 0, 0);
  size_scratch(c);
  return true;
}

ProjArgs base_args(dvi_ctx* c, int flavor, const Plan& pl, const Pass& ps) {
  ProjArgs a{};
  a.flavor = flavor;
  a.dtype = c->cfg.dtype;
  a.M = ps.M;
  a.n_pad = (ps.M + 15) / 16 * 16;
  a.n_tiles = pl.n_tiles;
  a.n_splits = pl.n_splits;
  a.kb_total = pl.kb_total;
  a.kb_per_split = pl.kb_per_split;
  a.n_ttiles = 1;
  a.lens = c->lens;
  a.rows_per_seq = ps.rows_per_seq;
  a.seq0 = ps.seq0;
  a.pos_off = ps.pos_off;
  a.part = c->part;
  a.counters = c->proj_counters;
  a.status = c->status;
  a.eps = c->cfg.rms_eps;
  a.d_norm = c->d;
  a.ss_tiles = c->d / kTileRows;
  a.prefetch_a = 1;
  a.b_mode = B_ACT;
  return a;
}

size_t layer_kv_offset(dvi_ctx* c, int l) {
  return static_cast<size_t>(l) * c->B * c->Hkv * c->max_len * c->hd * c->esz;
}

ProjMaps with_act(const ProjMaps& w, const CUtensorMap* act) {
  ProjMaps m = w;
  if (act) m.mb = *act;
  return m;
}

// Rows of an activation buffer: with bf16 its lo plane starts that many rows
// after its hi plane.
int act_rows(const dvi_ctx* c, const void* buf) {
  if (buf == c->xg_dr) return c->B;
  if (buf == c->xg_ver) return c->B * c->Kv;
  if (buf == c->xg_pf) return c->pf_rows;
  if (buf == c->attn_o || buf == c->ffn_h) return c->M_max;
  if (buf == c->log_u) return c->cap_rows;
  return 0;
}
size_t act_plane(const dvi_ctx* c, const void* buf, int ld) {
  return c->tc ? static_cast<size_t>(act_rows(c, buf)) * ld : 0;
}

// launch_proj with the plane strides of the context's activation buffers.
cudaError_t launch_proj_ctx(const dvi_ctx* c, ProjArgs a, const ProjMaps* m, cudaStream_t s,
                            const FinArgs* fin = nullptr) {
  if (a.xg_out) a.xg_plane = act_plane(c, a.xg_out, a.ld_xg);
  if (a.h_out) a.h_plane = act_plane(c, a.h_out, a.ld_h);
  return launch_proj(a, m, s, fin);
}

struct ProjLaunch {
  ProjArgs a;
  ProjMaps m;
};

// Completion-counter chaining of a bf16 decode pass (runtime option
// chain_counters; common.cuh): clears the pass's counters and turns chaining
// on; bf16 only, and not with the persistent projection chain.
cudaError_t dep_begin(dvi_ctx* c) {
  c->dep_on = false;
  c->dep_prev = nullptr;
  if (!c->tc || c->chain_ctas > 0 || !c->rt.chain_counters) return cudaSuccess;
  const cudaError_t e = cudaMemsetAsync(c->dep_ctr, 0, sizeof(int) * c->n_dep_ctr, c->stream);
  if (e != cudaSuccess) return e;
  c->dep_on = true;
  c->dep_slot = 0;
  return cudaSuccess;
}
void dep_end(dvi_ctx* c) {
  c->dep_on = false;
  c->dep_prev = nullptr;
}
// A launch of `grid` CTAs joins the chain: it waits for the previous
// launch's counter (if that one signals) and signals its own.
template <typename A>
void dep_link(dvi_ctx* c, A& a, int grid) {
  a.dep_wait = nullptr;
  a.dep_signal = nullptr;
  if (!c->dep_on) return;
  a.dep_wait = c->dep_prev;
  a.dep_count = c->dep_prev_count;
  if (c->dep_slot < c->n_dep_ctr) {
    a.dep_signal = c->dep_ctr + c->dep_slot++;
    c->dep_prev = a.dep_signal;
    c->dep_prev_count = grid;
  } else {
    c->dep_prev = nullptr;
  }
}
// A launch outside the chain (it waits for its predecessor's grid): the
// next launch waits for it the same way.
void dep_break(dvi_ctx* c) { c->dep_prev = nullptr; }
// Chaining for the launches enqueued while it lives.
struct DepScope {
  dvi_ctx* c;
  explicit DepScope(dvi_ctx* ctx) : c(ctx) {}
  ~DepScope() { dep_end(c); }
};

// q, k, v of RMSNorm(x) (gain folded into xg, 1/rms in the epilogue), RoPE,
// k/v rows into the cache
ProjLaunch qkv_launch(dvi_ctx* ctx, int l, const Pass& ps) {
  const dvi_layer_weights& lw = ctx->layers[l];
  ProjLaunch r{};
  ProjArgs& a = r.a;
  a = base_args(ctx, EPI_QKV, ctx->p_qkv, ps);
  a.act = ps.xg;
  a.ld_act = ctx->d;
  a.ss = ps.ss;
  a.ss_ld = ps.ss_ld;
  a.K = ctx->d;
  a.rows_q = ctx->nq;
  a.rows_k = ctx->nkv;
  a.rows_v = ctx->nkv;
  a.n_out = ctx->nq;
  a.w0 = lw.wq;
  a.w1 = lw.wk;
  a.w2 = lw.wv;
  a.q_out = ctx->q;
  a.ld_q = ctx->nq;
  a.kc = static_cast<char*>(ctx->kcache) + layer_kv_offset(ctx, l);
  a.vc = static_cast<char*>(ctx->vcache) + layer_kv_offset(ctx, l);
  a.max_len = ctx->max_len;
  a.head_dim = ctx->hd;
  a.n_kv_heads = ctx->Hkv;
  a.rope = ctx->rope;
  if (ctx->tc) r.m = with_act(ctx->maps[l].qkv, ps.xg_map);
  return r;
}

// block-causal multi-query attention of layer l
AttnArgs attn_args(dvi_ctx* ctx, int l, const Pass& ps) {
  AttnArgs t{};
  t.q = ctx->q;
  t.ld_q = ctx->nq;
  t.kc = static_cast<char*>(ctx->kcache) + layer_kv_offset(ctx, l);
  t.vc = static_cast<char*>(ctx->vcache) + layer_kv_offset(ctx, l);
  t.o = ctx->attn_o;
  t.ld_o = ctx->nq;
  t.o_dtype = ctx->cfg.dtype;
  t.dtype = ctx->cfg.dtype;
  t.n_heads = ctx->Hq;
  t.n_kv_heads = ctx->Hkv;
  t.head_dim = ctx->hd;
  t.max_len = ctx->max_len;
  t.lens = ctx->lens;
  t.rows_per_seq = ps.rows_per_seq;
  t.seq0 = ps.seq0;
  t.n_seqs = ps.n_seqs;
  t.pos_off = ps.pos_off;
  const bool dec_cluster = ctx->tc && ctx->Hq / ctx->Hkv <= 8;   // the tensor-core kernel
  t.split_len = dec_cluster ? 0 : ctx->attn_split_len;
  // a prompt pass has query rows enough to fill the GPU without splitting
  // the positions: one CTA walks its rows' whole prefix
  t.n_splits_max = dec_cluster ? (ps.pf ? 1 : ctx->dec_nsplits) : ctx->attn_nsplits;
  t.prefill = ps.pf && dec_cluster ? 1 : 0;
  t.part = ctx->attn_part;
  t.counters = ctx->attn_ctr;
  t.status = ctx->status;
  t.scale = 1.f / sqrtf(static_cast<float>(ctx->hd));
  t.kv_row0 = static_cast<long long>(l) * ctx->B * ctx->Hkv * ctx->max_len;
  t.kmap = &ctx->map_kc;
  t.vmap = &ctx->map_vc;
  t.o_plane = act_plane(ctx, ctx->attn_o, ctx->nq);
  return t;
}

// x += W_o . attn, then xg = x * ffn_norm for the FFN
ProjLaunch o_launch(dvi_ctx* ctx, int l, const Pass& ps) {
  const dvi_layer_weights& lw = ctx->layers[l];
  ProjLaunch r{};
  ProjArgs& a = r.a;
  a = base_args(ctx, EPI_RESID, ctx->p_o, ps);
  a.act = ctx->attn_o;
  a.ld_act = ctx->nq;
  a.K = ctx->nq;
  a.n_out = ctx->d;
  a.w0 = lw.wo;
  a.x_res = ps.x;
  a.ld_res = ctx->d;
  a.ss_out = ps.ss;
  a.ss_out_ld = ps.ss_ld;
  a.g_next = static_cast<const float*>(lw.ffn_norm);
  a.xg_out = ps.xg;
  a.ld_xg = ctx->d;
  if (ctx->tc) r.m = with_act(ctx->maps[l].o, &ctx->map_attn_o);
  return r;
}

// h = SiLU(W_gate n) * (W_up n) with n = RMSNorm(x)
ProjLaunch gu_launch(dvi_ctx* ctx, int l, const Pass& ps) {
  const dvi_layer_weights& lw = ctx->layers[l];
  ProjLaunch r{};
  ProjArgs& a = r.a;
  a = base_args(ctx, EPI_GATEUP, ctx->p_gu, ps);
  a.act = ps.xg;
  a.ld_act = ctx->d;
  a.ss = ps.ss;
  a.ss_ld = ps.ss_ld;
  a.K = ctx->d;
  a.n_out = ctx->F;
  a.w0 = lw.w_gate;
  a.w1 = lw.w_up;
  a.h_out = ctx->ffn_h;
  a.ld_h = ctx->F;
  if (ctx->tc) r.m = with_act(ctx->maps[l].gu, ps.xg_map);
  return r;
}

// x += W_down . h, then xg = x * g_last (the gain of the norm after the layer)
ProjLaunch down_launch(dvi_ctx* ctx, int l, const Pass& ps, const float* g_last) {
  const dvi_layer_weights& lw = ctx->layers[l];
  ProjLaunch r{};
  ProjArgs& a = r.a;
  a = base_args(ctx, EPI_RESID, ctx->p_down, ps);
  a.act = ctx->ffn_h;
  a.ld_act = ctx->F;
  a.K = ctx->F;
  a.n_out = ctx->d;
  a.w0 = lw.w_down;
  a.x_res = ps.x;
  a.ld_res = ctx->d;
  a.ss_out = ps.ss;
  a.ss_out_ld = ps.ss_ld;
  a.g_next = g_last;
  a.xg_out = ps.xg;
  a.ld_xg = ctx->d;
  if (ctx->tc) r.m = with_act(ctx->maps[l].down, &ctx->map_ffn_h);
  return r;
}

dvi_status run_proj(dvi_ctx* ctx, const ProjLaunch& pl) {
  ProjArgs a = pl.a;
  if (ctx->tc) dep_link(ctx, a, a.n_tiles * a.n_splits);
  else dep_break(ctx);
  DVI_CUDA(launch_proj_ctx(ctx, a, ctx->tc ? &pl.m : nullptr, ctx->stream));
  ++ctx->launches;
  return DVI_OK;
}

// Projections gathered for one persistent chain launch.
struct ChainBuilder {
  ChainArgs a;
};

void chain_reset(dvi_ctx* ctx, ChainBuilder& cb) {
  memset(&cb.a, 0, sizeof(cb.a));
  cb.a.n_ctas = ctx->chain_ctas;
  cb.a.phase_done = ctx->chain_ctr;
  cb.a.tile_ctr = ctx->chain_ctr + kChainMax;
  cb.a.exit_ctr = ctx->chain_ctr + kChainMax + kChainMax * kChainTiles;
  cb.a.part = ctx->chain_part;
}

void chain_add(dvi_ctx* ctx, ChainBuilder& cb, const ProjLaunch& pl) {
  ProjArgs a = pl.a;
  if (a.xg_out) a.xg_plane = act_plane(ctx, a.xg_out, a.ld_xg);
  if (a.h_out) a.h_plane = act_plane(ctx, a.h_out, a.ld_h);
  const int n = cb.a.n_phases++;
  cb.a.p[n] = a;
  cb.a.maps[n][0] = pl.m.m0;
  cb.a.maps[n][1] = pl.m.m1;
  cb.a.maps[n][2] = pl.m.m2;
  cb.a.maps[n][3] = pl.m.mb;
}

dvi_status chain_flush(dvi_ctx* ctx, ChainBuilder& cb) {
  if (cb.a.n_phases == 0) return DVI_OK;
  DVI_CUDA(launch_chain(cb.a, ctx->stream));
  ++ctx->launches;
  chain_reset(ctx, cb);
  return DVI_OK;
}

// The persistent chain serves bf16 passes of up to kChainMaxPad rows.
bool use_chain(const dvi_ctx* ctx, const Pass& ps) {
  return ctx->tc && !ps.pf && ctx->chain_ctas > 0 && (ps.M + 15) / 16 * 16 <= kChainMaxPad;
}

// One decoder layer on the pass's rows, one kernel per projection.  `g_last`
// is the gain of whatever consumes the pass's residual after this layer (the
// next layer's attention norm, or the final norm before a head).
// A projection of a bf16 prompt pass on the prefill kernel, with the
// activation buffer's 128-row map and the weights' 128-row maps.
dvi_status run_proj_pf(dvi_ctx* ctx, const ProjLaunch& pl, const CUtensorMap& act, const CUtensorMap& w0,
                       const CUtensorMap* w1 = nullptr, const CUtensorMap* w2 = nullptr) {
  ProjArgs a = pl.a;
  if (a.xg_out) a.xg_plane = act_plane(ctx, a.xg_out, a.ld_xg);
  if (a.h_out) a.h_plane = act_plane(ctx, a.h_out, a.ld_h);
  PfMaps m;
  m.act = act;
  m.w0 = w0;
  m.w1 = w1 ? *w1 : w0;
  m.w2 = w2 ? *w2 : w0;
  DVI_CUDA(launch_proj_pf(a, m, ctx->n_sms, ctx->stream));
  ++ctx->launches;
  return DVI_OK;
}

// One layer of a bf16 prompt pass: QKV, gate/up, O and down on the prefill
// kernel, the attention on the decode attention kernel.
dvi_status enqueue_layer_pf(dvi_ctx* ctx, int l, const Pass& ps, const float* g_last) {
  const LayerMaps& m = ctx->maps[l];
  dvi_status st;
  if ((st = run_proj_pf(ctx, qkv_launch(ctx, l, ps), ctx->map_pf_xg, m.qkv.m0, &m.qkv.m1, &m.qkv.m2)) != DVI_OK)
    return st;
  DVI_CUDA(launch_attn(attn_args(ctx, l, ps), ctx->stream));
  ++ctx->launches;
  if ((st = run_proj_pf(ctx, o_launch(ctx, l, ps), ctx->map_pf_attn_o, m.o.m0)) != DVI_OK) return st;
  if ((st = run_proj_pf(ctx, gu_launch(ctx, l, ps), ctx->map_pf_xg, m.gate128, &m.up128)) != DVI_OK) return st;
  return run_proj_pf(ctx, down_launch(ctx, l, ps, g_last), ctx->map_pf_ffn_h, m.down.m0);
}

dvi_status enqueue_layer(dvi_ctx* ctx, int l, const Pass& ps, const float* g_last) {
  if (ps.pf) return enqueue_layer_pf(ctx, l, ps, g_last);
  dvi_status st;
  if ((st = run_proj(ctx, qkv_launch(ctx, l, ps))) != DVI_OK) return st;
  AttnArgs at = attn_args(ctx, l, ps);
  if (ctx->tc && attn_chainable(at)) dep_link(ctx, at, attn_grid_ctas(at));
  else dep_break(ctx);
  DVI_CUDA(launch_attn(at, ctx->stream));
  ++ctx->launches;
  if ((st = run_proj(ctx, o_launch(ctx, l, ps))) != DVI_OK) return st;
  if ((st = run_proj(ctx, gu_launch(ctx, l, ps))) != DVI_OK) return st;
  return run_proj(ctx, down_launch(ctx, l, ps, g_last));
}

// Gain of the RMSNorm that reads the residual after layer l-1: layer l's
// attention norm, or the final norm after the last layer.
const float* norm_gain_before(dvi_ctx* ctx, int l) {
  return l < ctx->L ? static_cast<const float*>(ctx->layers[l].attn_norm)
                    : static_cast<const float*>(ctx->w.final_norm);
}

// Layers lo..hi-1; after the last one xg holds x * final_norm for a head.
// With the chain: QKV(lo), then per layer the attention kernel and one chain
// of O, gate/up, down and the next layer's QKV.
dvi_status enqueue_layers(dvi_ctx* ctx, int lo, int hi, const Pass& ps) {
  if (!use_chain(ctx, ps)) {
    for (int l = lo; l < hi; ++l) {
      const float* g_last = l + 1 < hi ? norm_gain_before(ctx, l + 1) : static_cast<const float*>(ctx->w.final_norm);
      dvi_status st = enqueue_layer(ctx, l, ps, g_last);
      if (st != DVI_OK) return st;
    }
    return DVI_OK;
  }
  ChainBuilder cb;
  chain_reset(ctx, cb);
  dvi_status st;
  for (int l = lo; l < hi; ++l) {
    if (l == lo) chain_add(ctx, cb, qkv_launch(ctx, l, ps));
    if ((st = chain_flush(ctx, cb)) != DVI_OK) return st;
    DVI_CUDA(launch_attn(attn_args(ctx, l, ps), ctx->stream));
    ++ctx->launches;
    const float* g_last = l + 1 < hi ? norm_gain_before(ctx, l + 1) : static_cast<const float*>(ctx->w.final_norm);
    chain_add(ctx, cb, o_launch(ctx, l, ps));
    chain_add(ctx, cb, gu_launch(ctx, l, ps));
    chain_add(ctx, cb, down_launch(ctx, l, ps, g_last));
    if (l + 1 < hi) chain_add(ctx, cb, qkv_launch(ctx, l + 1, ps));
  }
  return chain_flush(ctx, cb);
}

StepState step_state(dvi_ctx* c) {
  StepState st{};
  st.B = c->B;
  st.K = c->K;
  st.Kv = c->Kv;
  st.bonus = c->Kv > c->K ? 1 : 0;
  st.d = c->d;
  st.vocab = c->V;
  st.max_len = c->max_len;
  st.dtype = c->cfg.dtype;
  st.lens = c->lens;
  st.pending = c->pending;
  st.draft_ids = c->draft_ids;
  st.x_dr = c->x_dr;
  st.ss_dr = c->ss_dr;
  st.ss_dr_ld = c->B;
  st.g0 = norm_gain_before(c, 0);
  st.xg_dr = c->xg_dr;
  st.xg_dr_plane = act_plane(c, c->xg_dr, c->d);
  st.embed = c->w.embed;
  st.amax = c->amax;
  st.out_ids = c->out_ids;
  st.n_committed = c->n_committed;
  st.n_accepted = c->n_accepted;
  st.log_meta = c->log_meta;
  st.log_step = c->log_step;
  st.log_cap_steps = c->cap_steps;
  st.log_enabled = c->log_enabled;
  st.counters = c->counters;
  st.status = c->status;
  return st;
}

// Head projection over `rows` activation rows xg (x * final_norm) starting
// at row `row0` of `act`; 1/rms from `ss`.  W^S (+ LoRA) when `draft`.
// With `bu_inline` (bf16 drafter head) the kernel computes B u itself from
// the draft residual rows instead of reading it from `bu`.
// With `fin` (kind set), the head's last CTA runs that finalize step when the
// head launch can (bf16, unsplit); *fin_done tells the caller whether it did.
dvi_status enqueue_head(dvi_ctx* ctx, bool draft, int rows, int logits_mode, const void* act,
                        const CUtensorMap* act_map, int row0, const float* ss, int ss_ld, bool bu_inline = false,
                        int draft_pass = 0, FinArgs* fin = nullptr, bool* fin_done = nullptr) {
  Pass ps{nullptr, nullptr, 0, rows, 1, 0, 1, 0, nullptr, nullptr};
  ProjArgs a = base_args(ctx, EPI_HEAD, ctx->p_head, ps);
  a.act = act;
  a.ld_act = ctx->d;
  a.act_row0 = row0;
  a.ss = ss;
  a.ss_ld = ss_ld;
  a.K = ctx->d;
  a.n_out = ctx->V;
  a.w0 = draft ? ctx->w.draft_head : ctx->w.lm_head;
  a.amax = ctx->amax;
  if (draft && ctx->r > 0) {
    a.lora_a = ctx->w.lora_a;
    a.lora_bu = ctx->bu;
    a.lora_r = ctx->r;
    a.gamma = ctx->cfg.lora_gamma;
    if (bu_inline) {
      a.lora_bmat = ctx->w.lora_b;
      a.bu_x = ctx->x_dr;
      a.bu_ldx = ctx->d;
      a.bu_g = static_cast<const float*>(ctx->w.final_norm);
    }
  }
  if (logits_mode == 2) {
    a.logits_mode = 2;
    a.ld_logits = ctx->V;
    a.log_step = ctx->log_step;
    a.log_cap_steps = ctx->cap_steps;
    a.log_rows_per_step = ctx->B * ctx->K;
    if (draft) {
      // the drafter's logits of pass j are z of tuple j + 1: the update
      // reads them instead of recomputing them (A, B and W^S only change at
      // an update, which empties the buffer)
      a.logits_out = ctx->Z;
      a.log_src_rows = 1;         // one row per sequence; slot b * K + j
      a.log_dst_rows = ctx->K;
      a.log_dst_off = draft_pass;
    } else {
      a.logits_out = ctx->log_logits;
      a.log_src_rows = ctx->Kv;   // verify rows per sequence; the log keeps the first K
      a.log_dst_rows = ctx->K;
    }
  }
  ProjMaps pm{};
  if (ctx->tc) pm = with_act(draft ? ctx->head_s : ctx->head_v, act_map);
  bool fused = false;
  if (fin && fin_done) {
    bool stage = false;
    const size_t stage_bytes = fin->kind == FIN_DRAFT ? static_cast<size_t>(ctx->B) * ctx->d * ctx->esz : 0;
    fused = head_fin_ok(a, stage_bytes, &stage);
    fin->stage = stage && fin->kind == FIN_DRAFT ? 1 : 0;
    fin->ctr = ctx->fin_ctr;
    *fin_done = fused;
  }
  if (ctx->tc) dep_link(ctx, a, a.n_tiles * a.n_splits);
  else dep_break(ctx);
  DVI_CUDA(launch_proj_ctx(ctx, a, ctx->tc ? &pm : nullptr, ctx->stream, fused ? fin : nullptr));
  ctx->launches += 1;
  return DVI_OK;
}

// The drafter head can compute B u in-kernel: bf16, a LoRA term of rank
// <= kBuRank, at most kBuRows sequences, and a d the float4 loop covers.
bool bu_inline_ok(const dvi_ctx* ctx) {
  return ctx->tc && ctx->r > 0 && ctx->r <= kBuRank && ctx->B <= kBuRows && ctx->d % 128 == 0;
}

// The draft-phase megakernel: every draft pass with its head (MK_DRAFT,
// h_k of pass j to verify row j) or the shallow layers of an AR step (MK_AR,
// h_k to the AR rows that the deep layers read).  Its argmax keys and
// completion counters are cleared first.
dvi_status enqueue_mk(dvi_ctx* ctx, int mode) {
  MkArgs a = ctx->mk;
  a.mode = mode;
  if (mode == MK_DRAFT) {
    a.x_copy = ctx->x_ver;
    a.copy_row_stride = ctx->Kv;
    a.ss_copy = ctx->ss_ver;
    a.ss_copy_ld = ctx->B * ctx->Kv;
    a.xg_copy = ctx->xg_ver;
    a.xg_copy_plane = act_plane(ctx, ctx->xg_ver, ctx->d);
    a.log_enabled = ctx->log_enabled;
    a.log_u = ctx->log_u;
    a.log_plane = act_plane(ctx, ctx->log_u, ctx->d);
    a.zlog = ctx->log_enabled && ctx->rt.head_mode == 0 ? ctx->Z : nullptr;
  } else {
    a.x_copy = ctx->x_dr;
    a.copy_row_stride = 1;
    a.ss_copy = ctx->ss_dr;
    a.ss_copy_ld = ctx->B;
    a.xg_copy = ctx->xg_dr;
    a.xg_copy_plane = act_plane(ctx, ctx->xg_dr, ctx->d);
    a.log_enabled = 0;
  }
  DVI_CUDA(cudaMemsetAsync(ctx->mk_sync, 0, ctx->mk_sync_bytes, ctx->stream));
  DVI_CUDA(launch_mk(a, ctx->n_sms, ctx->stream));
  ctx->launches += 1;
  return DVI_OK;
}

dvi_status enqueue_draft(dvi_ctx* ctx) {
  if (ctx->mk_on) return enqueue_mk(ctx, MK_DRAFT);
  cudaStream_t s = ctx->stream;
  const StepState st = step_state(ctx);
  dvi_status rc;
  DepScope dep(ctx);
  DVI_CUDA(dep_begin(ctx));
  // passes j = 0..K-1 draft t~_{j+1}; with the bonus row, pass K only hands
  // h_{k,n+K} (of t~_K) to the verify rows
  for (int j = 0; j < ctx->Kv; ++j) {
    const bool drafts = j < ctx->K;
    Pass ps{ctx->x_dr, ctx->ss_dr, ctx->B, ctx->B, 1, 0, ctx->B, j, ctx->xg_dr, &ctx->map_xg_dr};
    if ((rc = enqueue_layers(ctx, 0, ctx->k, ps)) != DVI_OK) return rc;
    // u = RMSNorm_final(h_k) into the replay buffer, B u, and h_k to the verify rows
    HeadPrepArgs h{};
    h.x = ctx->x_dr;
    h.ldx = ctx->d;
    h.rows = ctx->B;
    h.gain = static_cast<const float*>(ctx->w.final_norm);
    h.eps = ctx->cfg.rms_eps;
    h.d = ctx->d;
    h.dtype = ctx->cfg.dtype;
    h.x_copy = ctx->x_ver;
    h.ld_copy = ctx->d;
    h.copy_row_stride = ctx->Kv;
    h.copy_row_off = j;
    h.ss_copy = ctx->ss_ver;
    h.ss_copy_ld = ctx->B * ctx->Kv;
    h.g_copy = norm_gain_before(ctx, ctx->k);
    h.xg_copy = ctx->xg_ver;
    h.xg_copy_plane = act_plane(ctx, ctx->xg_ver, ctx->d);
    h.log_u = ctx->log_u;
    h.log_plane = act_plane(ctx, ctx->log_u, ctx->d);
    h.log_step = ctx->log_step;
    h.log_cap_steps = ctx->cap_steps;
    h.log_rows_per_step = ctx->B * ctx->K;
    h.log_row_stride = ctx->K;
    h.log_row_off = j;
    h.log_enabled = drafts ? ctx->log_enabled : 0;
    // bf16: the head computes B u while its weights stream, and the logged u
    // and the hand-off run in the finalize kernel after it (one launch less)
    const bool fused = drafts && bu_inline_ok(ctx);
    if (ctx->r > 0 && drafts && !fused) {
      h.lora_b = ctx->w.lora_b;
      h.bu = ctx->bu;
      h.r = ctx->r;
    }
    if (!fused) {
      dep_break(ctx);
      DVI_CUDA(launch_head_prep(h, s));
      ctx->launches += 1;
    }
    if (!drafts) continue;
    const int zlog = ctx->log_enabled && ctx->rt.head_mode == 0 ? 2 : 0;   // the drafter's logits of the tuple
    FinArgs fa{};
    fa.kind = FIN_DRAFT;
    fa.j = j;
    fa.prep = fused ? 1 : 0;
    fa.st = st;
    fa.hp = h;
    bool fin_done = false;
    if ((rc = enqueue_head(ctx, true, ctx->B, zlog, ctx->xg_dr, &ctx->map_xg_dr, 0, ctx->ss_dr, ctx->B, fused, j,
                           &fa, &fin_done)) != DVI_OK)
      return rc;
    if (!fin_done) {
      dep_break(ctx);
      DVI_CUDA(launch_finalize_draft(st, j, fused ? &h : nullptr, s));
      ctx->launches += 1;
    }
  }
  return DVI_OK;
}

dvi_status enqueue_verify(dvi_ctx* ctx) {
  cudaStream_t s = ctx->stream;
  const StepState st = step_state(ctx);
  dvi_status rc;
  const int M = ctx->B * ctx->Kv;
  DepScope dep(ctx);
  DVI_CUDA(dep_begin(ctx));
  Pass pv{ctx->x_ver, ctx->ss_ver, M, M, ctx->Kv, 0, ctx->B, 0, ctx->xg_ver, &ctx->map_xg_ver};
  if ((rc = enqueue_layers(ctx, ctx->k, ctx->L, pv)) != DVI_OK) return rc;
  FinArgs fa{};
  fa.kind = FIN_VERIFY;
  fa.st = st;
  bool fin_done = false;
  if ((rc = enqueue_head(ctx, false, M, ctx->log_enabled ? 2 : 0, ctx->xg_ver, &ctx->map_xg_ver, 0, ctx->ss_ver, M,
                         false, 0, &fa, &fin_done)) != DVI_OK)
    return rc;
  if (!fin_done) {
    dep_break(ctx);
    DVI_CUDA(launch_finalize_verify(st, s));
    ctx->launches += 1;
  }
  return DVI_OK;
}

void fill_rope_host(int max_len, int hd, float theta, std::vector<float2>& out) {
  const int half = hd / 2;
  out.resize(static_cast<size_t>(max_len) * half);
  for (int p = 0; p < max_len; ++p)
    for (int i = 0; i < half; ++i) {
      const double inv = std::pow(static_cast<double>(theta), -2.0 * i / hd);
      const double ang = static_cast<double>(p) * inv;
      out[static_cast<size_t>(p) * half + i] = make_float2(static_cast<float>(std::cos(ang)),
                                                           static_cast<float>(std::sin(ang)));
    }
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

cudaEvent_t take_event(dvi_ctx* c) {
  if (!c->ev_pool.empty()) {
    cudaEvent_t e = c->ev_pool.back();
    c->ev_pool.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  cudaEventCreate(&e);
  return e;
}

// Records the start of a timed phase; returns the event to close it with.
cudaEvent_t mark_begin(dvi_ctx* c) {
  if (!c->timing) return nullptr;
  cudaEvent_t e = take_event(c);
  cudaEventRecord(e, c->stream);
  return e;
}
void mark_end(dvi_ctx* c, int phase, cudaEvent_t b) {
  if (!c->timing || !b) return;
  cudaEvent_t e = take_event(c);
  cudaEventRecord(e, c->stream);
  c->ev_marks.push_back({phase, {b, e}});
}

// Runs `fn` eagerly, or captures it once into `*exec` and replays it.
template <typename Fn>
dvi_status run_graph(dvi_ctx* ctx, cudaGraphExec_t* exec, long long* nlaunch, bool use_graph, Fn fn) {
  cudaStream_t s = ctx->stream;
  if (!use_graph) return fn();
  if (!*exec) {
    const long long before = ctx->launches;
    cudaGraph_t g = nullptr;
    DVI_CUDA(cudaStreamBeginCapture(s, cudaStreamCaptureModeThreadLocal));
    dvi_status rc = fn();
    cudaError_t ce = cudaStreamEndCapture(s, &g);
    if (rc != DVI_OK) {
      if (g) cudaGraphDestroy(g);
      return rc;
    }
    if (ce != cudaSuccess) return fail(ctx, DVI_ERR_CUDA, cudaGetErrorString(ce));
    ce = cudaGraphInstantiate(exec, g, 0);
    cudaGraphDestroy(g);
    if (ce != cudaSuccess) {
      *exec = nullptr;
      return fail(ctx, DVI_ERR_CUDA, cudaGetErrorString(ce));
    }
    *nlaunch = ctx->launches - before;
    ctx->launches = before;
  }
  DVI_CUDA(cudaGraphLaunch(*exec, s));
  ctx->launches += *nlaunch;
  return DVI_OK;
}

void drop_graphs(dvi_ctx* c) {
  if (c->draft_exec) cudaGraphExecDestroy(c->draft_exec);
  if (c->verify_exec) cudaGraphExecDestroy(c->verify_exec);
  if (c->ar_exec) cudaGraphExecDestroy(c->ar_exec);
  c->draft_exec = c->verify_exec = c->ar_exec = nullptr;
}

}  // namespace

extern "C" {

size_t dvi_workspace_bytes(const dvi_model_config* cfg, const dvi_runtime_config* rt) {
  if (!valid_config(cfg, rt, nullptr)) return 0;
  dvi_ctx c;
  init_dims(&c, cfg, rt);
  return layout(&c, nullptr);
}

dvi_status dvi_create(const dvi_model_config* cfg, const dvi_runtime_config* rt, const dvi_weights* weights,
                      void* workspace, size_t workspace_bytes, dvi_stream stream, dvi_ctx** out) {
  if (!out) return DVI_ERR_INVALID_ARG;
  *out = nullptr;
  std::string why;
  if (!valid_config(cfg, rt, &why)) {
    fprintf(stderr, "dvi_create: %s\n", why.c_str());
    return DVI_ERR_INVALID_ARG;
  }
  if (!weights || !weights->layers || !weights->embed || !weights->final_norm || !weights->lm_head ||
      !weights->draft_head || !workspace)
    return DVI_ERR_INVALID_ARG;
  if (cfg->lora_rank > 0 && (!weights->lora_a || !weights->lora_b)) return DVI_ERR_INVALID_ARG;
  if (rt->head_mode == 1 && (weights->draft_head == weights->lm_head || !aligned16(weights->draft_head))) {
    fprintf(stderr, "dvi_create: head_mode 1 trains draft_head in place: it must not alias lm_head and must be "
                    "16-byte aligned\n");
    return DVI_ERR_INVALID_ARG;
  }
  // B_s and the final-norm gain are read four floats at a time
  if ((cfg->lora_rank > 0 && !aligned16(weights->lora_b)) || !aligned16(weights->final_norm)) {
    fprintf(stderr, "dvi_create: lora_b and final_norm must be 16-byte aligned\n");
    return DVI_ERR_INVALID_ARG;
  }
  // the bf16 prompt passes read the layers' norm gains four floats at a time
  for (int l = 0; l < cfg->n_layers && cfg->dtype == DVI_BF16; ++l)
    if (!aligned16(weights->layers[l].attn_norm) || !aligned16(weights->layers[l].ffn_norm)) {
      fprintf(stderr, "dvi_create: attn_norm and ffn_norm must be 16-byte aligned\n");
      return DVI_ERR_INVALID_ARG;
    }
  if ((reinterpret_cast<uintptr_t>(workspace) & 255u) != 0) return DVI_ERR_INVALID_ARG;
  dvi_ctx* ctx = new dvi_ctx();
  init_dims(ctx, cfg, rt);
  ctx->ws_bytes = layout(ctx, nullptr);
  if (workspace_bytes < ctx->ws_bytes) {
    delete ctx;
    return DVI_ERR_CAPACITY;
  }
  ctx->ws = workspace;
  layout(ctx, static_cast<char*>(workspace));
  ctx->w = *weights;
  ctx->layers.assign(weights->layers, weights->layers + cfg->n_layers);
  ctx->w.layers = ctx->layers.data();
  ctx->stream = reinterpret_cast<cudaStream_t>(stream);
  if (ctx->mk_sized) {
    MkArgs& a = ctx->mk;
    for (int l = 0; l < ctx->k; ++l) {
      const dvi_layer_weights& lw = ctx->layers[l];
      a.layer[l] = MkLayerW{lw.wq, lw.wk, lw.wv, lw.wo, lw.w_gate, lw.w_up, lw.w_down,
                            static_cast<const float*>(lw.attn_norm), static_cast<const float*>(lw.ffn_norm)};
    }
    a.embed = weights->embed;
    a.final_norm = static_cast<const float*>(weights->final_norm);
    a.g_hand = norm_gain_before(ctx, ctx->k);
    a.w_head = weights->draft_head;
    a.lora_a = weights->lora_a;
    a.lora_b = weights->lora_b;
    a.kc = ctx->kcache;
    a.vc = ctx->vcache;
    a.rope = ctx->rope;
    a.lens = ctx->lens;
    a.pending = ctx->pending;
    a.draft_ids = ctx->draft_ids;
    a.log_step = ctx->log_step;
    a.log_cap_steps = ctx->cap_steps;
    a.status = ctx->status;
    // weight descriptors (16 tiles of 8 rows x 64 per box): [k][wq, wk, wv, wo, wg, wu, wd], then W^S,
    // then the K and V caches (16 KB boxes: hd / 64 tiles of 8192 / hd rows x 64)
    ctx->mk_maps.assign(7 * ctx->k + 3, CUtensorMap{});
    bool ok = true;
    for (int l = 0; l < ctx->k && ok; ++l) {
      const dvi_layer_weights& lw = ctx->layers[l];
      CUtensorMap* m = ctx->mk_maps.data() + 7 * l;
      ok = make_weight_map_kblocks(m + 0, lw.wq, ctx->nq, ctx->d, 8, 16) &&
           make_weight_map_kblocks(m + 1, lw.wk, ctx->nkv, ctx->d, 8, 16) &&
           make_weight_map_kblocks(m + 2, lw.wv, ctx->nkv, ctx->d, 8, 16) &&
           make_weight_map_kblocks(m + 3, lw.wo, ctx->d, ctx->nq, 8, 16) &&
           make_weight_map_kblocks(m + 4, lw.w_gate, ctx->F, ctx->d, 8, 16) &&
           make_weight_map_kblocks(m + 5, lw.w_up, ctx->F, ctx->d, 8, 16) &&
           make_weight_map_kblocks(m + 6, lw.w_down, ctx->d, ctx->F, 8, 16);
    }
    ok = ok && make_weight_map_kblocks(ctx->mk_maps.data() + 7 * ctx->k, weights->draft_head, ctx->V, ctx->d, 8, 16);
    const int kv_rows = static_cast<int>(static_cast<long long>(ctx->L) * ctx->B * ctx->Hkv * ctx->max_len);
    const int kv_box = 8192 / ctx->hd;
    ok = ok && make_weight_map_kblocks(ctx->mk_maps.data() + 7 * ctx->k + 1, ctx->kcache, kv_rows, ctx->hd, kv_box,
                                       ctx->hd / 64) &&
         make_weight_map_kblocks(ctx->mk_maps.data() + 7 * ctx->k + 2, ctx->vcache, kv_rows, ctx->hd, kv_box,
                                 ctx->hd / 64);
    a.wmaps = ctx->mk_maps_dev;   // uploaded after the workspace is cleared (below)
    ctx->mk_on = ok && mk_ctas_per_sm(a) >= 1;
  }
  if (ctx->tc) {
    auto mk = [&](CUtensorMap* m, const void* p, int rows, int cols) {
      return aligned16(p) && make_weight_map(m, p, rows, cols);
    };
    bool ok = true;
    ctx->maps.resize(ctx->L);
    for (int l = 0; l < ctx->L && ok; ++l) {
      const dvi_layer_weights& lw = ctx->layers[l];
      LayerMaps& m = ctx->maps[l];
      ok = mk(&m.qkv.m0, lw.wq, ctx->nq, ctx->d) && mk(&m.qkv.m1, lw.wk, ctx->nkv, ctx->d) &&
           mk(&m.qkv.m2, lw.wv, ctx->nkv, ctx->d) && mk(&m.o.m0, lw.wo, ctx->d, ctx->nq) &&
           aligned16(lw.w_gate) && make_half_weight_map(&m.gu.m0, lw.w_gate, ctx->F, ctx->d) &&
           aligned16(lw.w_up) && make_half_weight_map(&m.gu.m1, lw.w_up, ctx->F, ctx->d) &&
           mk(&m.gate128, lw.w_gate, ctx->F, ctx->d) && mk(&m.up128, lw.w_up, ctx->F, ctx->d) &&
           mk(&m.down.m0, lw.w_down, ctx->d, ctx->F);
    }
    ok = ok && mk(&ctx->head_v.m0, weights->lm_head, ctx->V, ctx->d) &&
         mk(&ctx->head_s.m0, weights->draft_head, ctx->V, ctx->d);
    // each map covers both planes of its buffer: [2][R][cols]
    ok = ok && make_act_map(&ctx->map_xg_dr, ctx->xg_dr, ctx->B, ctx->d) &&
         make_act_map(&ctx->map_xg_ver, ctx->xg_ver, ctx->B * ctx->Kv, ctx->d) &&
         make_act_map(&ctx->map_xg_pf, ctx->xg_pf, ctx->pf_rows, ctx->d) &&
         make_act_map_box(&ctx->map_pf_xg, ctx->xg_pf, ctx->pf_rows, ctx->d, kTileRows) &&
         make_act_map_box(&ctx->map_pf_attn_o, ctx->attn_o, ctx->M_max, ctx->nq, kTileRows) &&
         make_act_map_box(&ctx->map_pf_ffn_h, ctx->ffn_h, ctx->M_max, ctx->F, kTileRows) &&
         make_act_map(&ctx->map_attn_o, ctx->attn_o, ctx->M_max, ctx->nq) &&
         make_act_map(&ctx->map_ffn_h, ctx->ffn_h, ctx->M_max, ctx->F) &&
         make_act_map(&ctx->map_log_u, ctx->log_u, ctx->cap_rows, ctx->d);
    const long long kv_rows = static_cast<long long>(ctx->L) * ctx->B * ctx->Hkv * ctx->max_len;
    ok = ok && make_kv_map(&ctx->map_kc, ctx->kcache, kv_rows, ctx->hd) &&
         make_kv_map(&ctx->map_vc, ctx->vcache, kv_rows, ctx->hd);
    if (!ok) {
      fprintf(stderr, "dvi_create: TMA descriptor creation failed (weights must be 16-byte aligned)\n");
      delete ctx;
      return DVI_ERR_INVALID_ARG;
    }
  }
  std::vector<float2> rope;
  fill_rope_host(ctx->max_len, ctx->hd, cfg->rope_theta, rope);
  if (cudaMemsetAsync(workspace, 0, ctx->ws_bytes, ctx->stream) != cudaSuccess ||
      cudaMemcpyAsync(ctx->rope, rope.data(), rope.size() * sizeof(float2), cudaMemcpyHostToDevice, ctx->stream) !=
          cudaSuccess ||
      (ctx->mk_on && cudaMemcpyAsync(ctx->mk_maps_dev, ctx->mk_maps.data(), sizeof(CUtensorMap) * ctx->mk_maps.size(),
                                     cudaMemcpyHostToDevice, ctx->stream) != cudaSuccess) ||
      (ctx->w_master && launch_master_init(weights->draft_head, ctx->w_master,
                                           static_cast<size_t>(ctx->V) * ctx->d, ctx->stream) != cudaSuccess) ||
      cudaStreamSynchronize(ctx->stream) != cudaSuccess) {
    delete ctx;
    return DVI_ERR_CUDA;
  }
  *out = ctx;
  return DVI_OK;
}

dvi_status dvi_prefill(dvi_ctx* ctx, int seq, const int32_t* d_tokens, int n_tokens, int32_t* d_first_token) {
  if (!ctx) return DVI_ERR_INVALID_ARG;
  if (seq < 0 || seq >= ctx->B || !d_tokens || n_tokens < 1)
    return fail(ctx, DVI_ERR_INVALID_ARG, "prefill: bad sequence, tokens or length");
  if (n_tokens + ctx->Kv + 1 > ctx->max_len) return fail(ctx, DVI_ERR_CAPACITY, "prefill: prompt exceeds max_seq_len");
  cudaStream_t s = ctx->stream;
  const StepState st = step_state(ctx);
  DVI_CUDA(launch_reset_seq(st, seq, s));
  ctx->launches += 1;
  int last_rows = 0;
  for (int c0 = 0; c0 < n_tokens; c0 += ctx->chunk) {
    const int rows = std::min(ctx->chunk, n_tokens - c0);
    EmbedArgs e{};
    e.table = ctx->w.embed;
    e.dtype = ctx->cfg.dtype;
    e.d = ctx->d;
    e.vocab = ctx->V;
    e.tokens = d_tokens + c0;
    e.x = ctx->x_pf;
    e.ldx = ctx->d;
    e.ss = ctx->ss_pf;
    e.ss_ld = ctx->pf_rows;
    e.g = norm_gain_before(ctx, 0);
    e.xg = ctx->xg_pf;
    e.xg_plane = act_plane(ctx, ctx->xg_pf, ctx->d);
    e.ldxg = ctx->d;
    e.rows = rows;
    e.status = ctx->status;
    DVI_CUDA(launch_embed(e, s));
    ctx->launches += 1;
    Pass ps{ctx->x_pf, ctx->ss_pf, ctx->pf_rows, rows, rows, seq, 1, c0, ctx->xg_pf, &ctx->map_xg_pf, ctx->tc};
    dvi_status rc = enqueue_layers(ctx, 0, ctx->L, ps);
    if (rc != DVI_OK) return rc;
    last_rows = rows;
  }
  // verifier head on the last prompt row
  dvi_status rc = enqueue_head(ctx, false, 1, 0, ctx->xg_pf, &ctx->map_xg_pf, last_rows - 1,
                               ctx->ss_pf + (last_rows - 1), ctx->pf_rows);
  if (rc != DVI_OK) return rc;
  DVI_CUDA(launch_finalize_prefill(st, seq, n_tokens, d_first_token, s));
  ctx->launches += 2;
  return DVI_OK;
}

dvi_status dvi_draft_verify_commit(dvi_ctx* ctx, int32_t* d_out_ids, int32_t* d_n_committed,
                                   int32_t* d_n_accepted) {
  if (!ctx) return DVI_ERR_INVALID_ARG;
  cudaStream_t s = ctx->stream;
  ctx->step_calls += 1;
  // the first step runs eagerly (it also sets kernel attributes); later
  // steps replay the captured graphs
  const bool g = ctx->rt.use_graphs && ctx->step_calls > 1;
  cudaEvent_t t0 = mark_begin(ctx);
  dvi_status rc = run_graph(ctx, &ctx->draft_exec, &ctx->draft_launches, g, [&] { return enqueue_draft(ctx); });
  if (rc != DVI_OK) return rc;
  mark_end(ctx, 0, t0);
  cudaEvent_t t1 = mark_begin(ctx);
  rc = run_graph(ctx, &ctx->verify_exec, &ctx->verify_launches, g, [&] { return enqueue_verify(ctx); });
  if (rc != DVI_OK) return rc;
  mark_end(ctx, 1, t1);
  if (d_out_ids)
    DVI_CUDA(cudaMemcpyAsync(d_out_ids, ctx->out_ids, sizeof(int) * ctx->B * ctx->Kv, cudaMemcpyDeviceToDevice, s));
  if (d_n_committed)
    DVI_CUDA(cudaMemcpyAsync(d_n_committed, ctx->n_committed, sizeof(int) * ctx->B, cudaMemcpyDeviceToDevice, s));
  if (d_n_accepted)
    DVI_CUDA(cudaMemcpyAsync(d_n_accepted, ctx->n_accepted, sizeof(int) * ctx->B, cudaMemcpyDeviceToDevice, s));
  return DVI_OK;
}

dvi_status dvi_log(dvi_ctx* ctx, int enable) {
  if (!ctx) return DVI_ERR_INVALID_ARG;
  const int e = enable ? 1 : 0;
  if (e != ctx->log_enabled) drop_graphs(ctx);
  ctx->log_enabled = e;
  return DVI_OK;
}

dvi_status dvi_update_drafter(dvi_ctx* ctx, const dvi_update_config* u) {
  if (!ctx || !u) return DVI_ERR_INVALID_ARG;
  if (!(u->tau > 0.f) || u->t_ramp < 0 || u->t_warmup < 0 || u->objective < 0 || u->objective > 3 ||
      u->optimizer < 0 || u->optimizer > 1 || !(u->t_beta > 0.f))
    return fail(ctx, DVI_ERR_INVALID_ARG, "update: bad hyper-parameters");
  const bool full = ctx->rt.head_mode == 1;
  if (!full && ctx->r == 0) return fail(ctx, DVI_ERR_UNIMPLEMENTED, "update: no LoRA factors (lora_rank 0)");
  cudaStream_t s = ctx->stream;
  UpdateArgs a{};
  a.cap = ctx->cap_rows;
  a.V = ctx->V;
  a.d = ctx->d;
  a.r = ctx->r;
  a.dtype = ctx->cfg.dtype;
  a.B = ctx->B;
  a.K = ctx->K;
  a.log_u = ctx->log_u;
  a.log_plane = act_plane(ctx, ctx->log_u, ctx->d);
  a.log_logits = ctx->log_logits;
  a.log_meta = ctx->log_meta;
  a.log_step = ctx->log_step;
  a.Z = ctx->Z;
  a.rowstat = ctx->rowstat;
  a.stat_part = ctx->stat_part;
  a.coef = ctx->coef;
  a.ub = ctx->ub;
  a.ga = ctx->ga;
  a.ga_part = ctx->ga_part;
  a.n_vtiles = (ctx->V + 127) / 128;
  a.lora_a = ctx->w.lora_a;
  a.lora_b = ctx->w.lora_b;
  a.gamma = ctx->cfg.lora_gamma;
  a.m_a = ctx->m_a;
  a.v_a = ctx->v_a;
  a.m_b = ctx->m_b;
  a.v_b = ctx->v_b;
  a.grad_a = ctx->grad_a;
  a.grad_b = ctx->grad_b;
  a.w_head = ctx->w.draft_head;
  a.w_master = ctx->w_master;
  a.m_w = ctx->m_w;
  a.v_w = ctx->v_w;
  a.G = ctx->G;
  a.grad_w = ctx->grad_w;
  a.keep_grad_w = u->keep_grad_w ? 1 : 0;
  a.dev_state = ctx->dev_state;
  a.ctr = ctx->upd_ctr;
  a.counters = ctx->counters;
  a.status = ctx->status;
  a.cfg = *u;
  cudaEvent_t t0 = mark_begin(ctx);
  if (!full && update_fused_ok(a, ctx->n_sms)) {
    // one cooperative launch: the drafter logits were logged while drafting
    DVI_CUDA(launch_update_fused(a, ctx->n_sms, s));
    ctx->launches += 1;
    mark_end(ctx, 2, t0);
    return DVI_OK;
  }
  DVI_CUDA(launch_update_prep(a, s));
  // drafter logits of every buffer row: Z = U W^S^T + gamma (U B^T) A^T
  Pass ps{nullptr, nullptr, 0, ctx->cap_rows, 1, 0, 1, 0, nullptr, nullptr};
  ProjArgs p = base_args(ctx, EPI_HEAD, ctx->p_head, ps);
  p.act = ctx->log_u;
  p.ld_act = ctx->d;
  p.K = ctx->d;
  p.n_out = ctx->V;
  p.w0 = ctx->w.draft_head;
  p.logits_mode = 1;
  p.logits_out = ctx->Z;
  p.ld_logits = ctx->V;
  p.lora_a = ctx->w.lora_a;
  p.lora_bu = ctx->ub;
  p.lora_r = ctx->r;
  p.gamma = ctx->cfg.lora_gamma;
  ProjMaps pm{};
  if (ctx->tc) pm = with_act(ctx->head_s, &ctx->map_log_u);
  DVI_CUDA(launch_proj_ctx(ctx, p, ctx->tc ? &pm : nullptr, s));
  // row statistics; the last row's CTA forms the loss and the coefficients
  DVI_CUDA(launch_update_rowstats(a, s));
  if (full) {
    DVI_CUDA(launch_update_full(a, s));
    DVI_CUDA(launch_update_finish(a, s));
    ctx->launches += (ctx->r > 0 ? 1 : 0) + 5;
  } else {
    // dA with Adam on A, the G A reduction, then dB with Adam on B; the last
    // grad_b CTA ends the update
    DVI_CUDA(launch_update_grad_a(a, s));
    DVI_CUDA(launch_update_grad_b(a, s));
    ctx->launches += 6;
  }
  mark_end(ctx, 2, t0);
  return DVI_OK;
}

dvi_status dvi_ar_step(dvi_ctx* ctx, int32_t* d_out_ids) {
  if (!ctx) return DVI_ERR_INVALID_ARG;
  cudaStream_t s = ctx->stream;
  ctx->ar_calls += 1;
  // like the decode step: the first call runs eagerly, later calls replay
  // its captured graph (every input of the step is device-side state)
  const bool g = ctx->rt.use_graphs && ctx->ar_calls > 1;
  dvi_status rc = run_graph(ctx, &ctx->ar_exec, &ctx->ar_launches, g, [&]() -> dvi_status {
    StepState st = step_state(ctx);
    st.out_ids = ctx->ar_out;
    DepScope dep(ctx);
    Pass ps{ctx->x_dr, ctx->ss_dr, ctx->B, ctx->B, 1, 0, ctx->B, 0, ctx->xg_dr, &ctx->map_xg_dr};
    dvi_status r;
    if (ctx->mk_on) {
      // the shallow layers as in a draft pass (same arithmetic: the DVI
      // stream stays bit-identical to AR), the deep ones as in verify
      if ((r = enqueue_mk(ctx, MK_AR)) != DVI_OK) return r;
      if ((r = enqueue_layers(ctx, ctx->k, ctx->L, ps)) != DVI_OK) return r;
    } else {
      DVI_CUDA(dep_begin(ctx));
      if ((r = enqueue_layers(ctx, 0, ctx->L, ps)) != DVI_OK) return r;
    }
    FinArgs fa{};
    fa.kind = FIN_AR;
    fa.st = st;
    bool fin_done = false;
    if ((r = enqueue_head(ctx, false, ctx->B, 0, ctx->xg_dr, &ctx->map_xg_dr, 0, ctx->ss_dr, ctx->B, false, 0, &fa,
                          &fin_done)) != DVI_OK)
      return r;
    if (!fin_done) {
      dep_break(ctx);
      DVI_CUDA(launch_finalize_ar(st, s));
      ctx->launches += 1;
    }
    return DVI_OK;
  });
  if (rc != DVI_OK) return rc;
  if (d_out_ids) DVI_CUDA(cudaMemcpyAsync(d_out_ids, ctx->ar_out, sizeof(int) * ctx->B, cudaMemcpyDeviceToDevice, s));
  return DVI_OK;
}

dvi_status dvi_get_stats(dvi_ctx* ctx, dvi_stats* out) {
  if (!ctx || !out) return DVI_ERR_INVALID_ARG;
  DVI_CUDA(cudaStreamSynchronize(ctx->stream));
  long long c[8];
  float ds[16];
  int status = 0;
  DVI_CUDA(cudaMemcpy(c, ctx->counters, sizeof(c), cudaMemcpyDeviceToHost));
  DVI_CUDA(cudaMemcpy(ds, ctx->dev_state, sizeof(ds), cudaMemcpyDeviceToHost));
  DVI_CUDA(cudaMemcpy(&status, ctx->status, sizeof(int), cudaMemcpyDeviceToHost));
  memset(out, 0, sizeof(*out));
  out->steps = c[0];
  out->drafted = c[1];
  out->accepted = c[2];
  out->committed = c[3];
  out->updates = c[4];
  out->kernel_launches = ctx->launches;
  out->update_t = static_cast<int>(ds[0]);
  out->baseline_b = ds[1];
  out->last_loss = ds[2];
  out->last_kl = ds[3];
  out->last_pg = ds[4];
  out->last_ce = ds[5];
  out->last_ent = ds[6];
  out->last_rl = ds[7];
  out->last_kl1 = ds[8];
  out->last_accept_rate = ds[9];
  out->device_status = status;
  out->persistent_ctas = ctx->chain_ctas;
  out->megakernel_ctas = ctx->mk_on ? ctx->n_sms : 0;
  return DVI_OK;
}

const char* dvi_last_error(const dvi_ctx* ctx) { return ctx ? ctx->err.c_str() : "null context"; }

dvi_status dvi_destroy(dvi_ctx* ctx) {
  if (!ctx) return DVI_ERR_INVALID_ARG;
  drop_graphs(ctx);
  for (auto& m : ctx->ev_marks) {
    cudaEventDestroy(m.second.first);
    cudaEventDestroy(m.second.second);
  }
  for (cudaEvent_t e : ctx->ev_pool) cudaEventDestroy(e);
  delete ctx;
  return DVI_OK;
}

dvi_status dvi_debug_buffer(dvi_ctx* ctx, int which, void** dptr, size_t* bytes) {
  if (!ctx || !dptr || !bytes) return DVI_ERR_INVALID_ARG;
  const size_t e = ctx->esz;
  const size_t kv = static_cast<size_t>(ctx->L) * ctx->B * ctx->Hkv * ctx->max_len * ctx->hd * e;
  const int rr = ctx->r > 0 ? ctx->r : 1;
  switch (which) {
    case DVI_BUF_LENS: *dptr = ctx->lens; *bytes = sizeof(int) * ctx->B; break;
    case DVI_BUF_PENDING: *dptr = ctx->pending; *bytes = sizeof(int) * ctx->B; break;
    case DVI_BUF_DRAFT_IDS: *dptr = ctx->draft_ids; *bytes = sizeof(int) * ctx->B * (ctx->K + 1); break;
    case DVI_BUF_LOG_U: *dptr = ctx->log_u; *bytes = (ctx->tc ? 2 : 1) * e * ctx->cap_rows * ctx->d; break;
    case DVI_BUF_LOG_LOGITS: *dptr = ctx->log_logits; *bytes = sizeof(float) * ctx->cap_rows * static_cast<size_t>(ctx->V); break;
    case DVI_BUF_LOG_META: *dptr = ctx->log_meta; *bytes = sizeof(int) * 6 * ctx->cap_rows; break;
    case DVI_BUF_GRAD_A: *dptr = ctx->grad_a; *bytes = sizeof(float) * static_cast<size_t>(ctx->V) * rr; break;
    case DVI_BUF_GRAD_B: *dptr = ctx->grad_b; *bytes = sizeof(float) * static_cast<size_t>(rr) * ctx->d; break;
    case DVI_BUF_X_DRAFT: *dptr = ctx->x_dr; *bytes = sizeof(float) * ctx->B * ctx->d; break;
    case DVI_BUF_X_VERIFY: *dptr = ctx->x_ver; *bytes = sizeof(float) * ctx->B * ctx->Kv * ctx->d; break;
    case DVI_BUF_K_CACHE: *dptr = ctx->kcache; *bytes = kv; break;
    case DVI_BUF_V_CACHE: *dptr = ctx->vcache; *bytes = kv; break;
    case DVI_BUF_STATUS: *dptr = ctx->status; *bytes = sizeof(int); break;
    case DVI_BUF_GRAD_W:
      if (!ctx->grad_w) return fail(ctx, DVI_ERR_INVALID_ARG, "debug_buffer: GRAD_W exists in head_mode 1 only");
      *dptr = ctx->grad_w;
      *bytes = sizeof(float) * static_cast<size_t>(ctx->V) * ctx->d;
      break;
    case DVI_BUF_Z: *dptr = ctx->Z; *bytes = sizeof(float) * ctx->cap_rows * static_cast<size_t>(ctx->V); break;
    default: return fail(ctx, DVI_ERR_INVALID_ARG, "debug_buffer: unknown buffer");
  }
  return DVI_OK;
}

dvi_status dvi_timing(dvi_ctx* ctx, int enable) {
  if (!ctx) return DVI_ERR_INVALID_ARG;
  ctx->timing = enable ? 1 : 0;
  return DVI_OK;
}

dvi_status dvi_get_timing(dvi_ctx* ctx, double* ms, int* counts) {
  if (!ctx || !ms || !counts) return DVI_ERR_INVALID_ARG;
  DVI_CUDA(cudaStreamSynchronize(ctx->stream));
  for (int i = 0; i < 3; ++i) {
    ms[i] = 0.0;
    counts[i] = 0;
  }
  for (auto& m : ctx->ev_marks) {
    float t = 0.f;
    if (cudaEventElapsedTime(&t, m.second.first, m.second.second) == cudaSuccess && m.first >= 0 && m.first < 3) {
      ms[m.first] += t;
      counts[m.first] += 1;
    }
    ctx->ev_pool.push_back(m.second.first);
    ctx->ev_pool.push_back(m.second.second);
  }
  ctx->ev_marks.clear();
  return DVI_OK;
}

dvi_status dvi_linear(dvi_ctx* ctx, const void* d_w, int n_out, int k_in, const float* d_x, int m_rows,
                      float* d_y) {
  if (!ctx) return DVI_ERR_INVALID_ARG;
  if (!d_w || !d_x || !d_y || n_out < 1 || k_in < 1 || m_rows < 1 || m_rows > kMaxTokens)
    return fail(ctx, DVI_ERR_INVALID_ARG, "linear: bad arguments");
  if (ctx->tc && (k_in % 8 || !aligned16(d_w) || !aligned16(d_x)))
    return fail(ctx, DVI_ERR_INVALID_ARG, "linear: bf16 needs k_in % 8 == 0 and 16-byte aligned pointers");
  Plan pl = plan_for(ctx, EPI_HEAD, n_out, k_in, 0, 0, 0);
  Pass ps{nullptr, nullptr, 0, m_rows, 1, 0, 1, 0, nullptr, nullptr};
  ProjArgs a = base_args(ctx, EPI_HEAD, pl, ps);
  a.b_mode = B_SOFT_F32;
  a.act = d_x;
  a.ld_act = k_in;
  a.K = k_in;
  a.n_out = n_out;
  a.w0 = d_w;
  a.logits_mode = 1;
  a.logits_out = d_y;
  a.ld_logits = n_out;
  const int ntt = ctx->tc ? 1 : (m_rows + kChunk - 1) / kChunk;
  if (proj_partial_floats(a, ctx->tc) > ctx->part_floats || a.n_tiles * ntt > ctx->n_proj_counters)
    return fail(ctx, DVI_ERR_CAPACITY, "linear: shape needs more split-K scratch than the workspace has");
  ProjMaps m{};
  if (ctx->tc && !make_weight_map(&m.m0, d_w, n_out, k_in))
    return fail(ctx, DVI_ERR_INVALID_ARG, "linear: TMA descriptor creation failed");
  DVI_CUDA(launch_proj_ctx(ctx, a, ctx->tc ? &m : nullptr, ctx->stream));
  ctx->launches += 1;
  return DVI_OK;
}

}  // extern "C"
