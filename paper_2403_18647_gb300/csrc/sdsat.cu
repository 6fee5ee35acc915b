// libsdsat host side: the C ABI declared in include/sdsat.h.
//
// A context holds the borrowed weight pointers, one TMA descriptor per
// weight matrix, the RoPE table and the workspaces of one block forward; a KV
// object holds the cache and the device-resident committed lengths.  Every
// compute entry point only validates arguments and enqueues kernels on the
// context stream (programmatic dependent launch between consecutive kernels),
// so the whole decode loop can run, and be graph-captured, without the host.
#include <cudaTypedefs.h>

#include <algorithm>
#include <cmath>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <new>
#include <vector>

#include "sdsat.h"
#include "internal.h"

using namespace sdsat;
static_assert(TRACE_WORDS == SDSAT_TRACE_WORDS, "trace record size");
static_assert(TREE_MAX_ROWS == SDSAT_MAX_ROWS && SDSAT_ATT_MAXQ == SDSAT_MAX_Q, "tree kernel limits");

namespace {

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
std::once_flag g_encode_once;

bool get_encode() {
  std::call_once(g_encode_once, [] {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  });
  return g_encode != nullptr;
}

// bf16 [rows][cols] row-major, boxes of 64 rows x 64 columns, 128-byte swizzle
bool make_wmap(CUtensorMap* map, const void* ptr, int rows, int cols) {
  if (!get_encode()) return false;
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
  cuuint32_t box[2] = {64, 64};
  cuuint32_t estr[2] = {1, 1};
  return g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// bf16 [rows][cols] activation operand, boxes of `box_rows` rows x 64 columns, 128-byte swizzle
bool make_xmap(CUtensorMap* map, const void* ptr, int rows, int cols, int box_rows) {
  if (!get_encode()) return false;
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
  cuuint32_t box[2] = {64, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1, 1};
  return g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// bf16 KV cache viewed as [rows][hd], boxes of 64 dims x ATT_UNIT rows, 128-byte swizzle
bool make_kvmap(CUtensorMap* map, const void* ptr, long long rows, int hd) {
  if (!get_encode()) return false;
  cuuint64_t dims[2] = {(cuuint64_t)hd, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)hd * 2};
  cuuint32_t box[2] = {64, (cuuint32_t)ATT_UNIT};
  cuuint32_t estr[2] = {1, 1};
  return g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int mpad_index(int M) { return M <= 16 ? 0 : (M <= 32 ? 1 : 2); }

bool aligned16(const void* p) { return p && (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

struct LayerMaps {
  CUtensorMap q, k, v, o, gate, up, down;
};

// kernel classes for the profiling hook
enum KClass : int {
  K_RMSNORM = 0, K_GEMM_QKV, K_ATTENTION, K_GEMM_O, K_GEMM_GATEUP, K_GEMM_DOWN, K_GEMM_LM_HEAD, K_ACCEPT,
  K_BUILD_BLOCK, K_KV_COMMIT, K_PREFILL_COMMIT, K_GEMM_OP, K_ATTENTION_OP, K_TREE_PREP, K_TREE_COMPACT,
  K_PF_GEMM, K_PF_ROPE_KV, K_PF_ATTENTION, K_COUNT
};
const char* const KCLASS_NAME[K_COUNT] = {"rmsnorm", "gemm_qkv", "attention", "gemm_o", "gemm_gateup", "gemm_down",
                                          "gemm_lm_head", "accept", "build_block", "kv_commit", "prefill_commit",
                                          "gemm_op", "attention_op", "tree_prep", "tree_compact", "prefill_gemm",
                                          "prefill_rope_kv", "prefill_attention"};

constexpr int MAX_GEMM_TILES = 1 << 16;
constexpr int OP_MAX_K = 32768;   // K limit of sdsat_op_gemm (its operand scratch is sized at create)

// the GEMM activation operands (bf16 hi + lo), one pair per producer
enum XSrc : int { X_NORM = 0, X_ATTN = 1, X_FFN = 2, X_COUNT = 3 };

}  // namespace

struct sdsat_ctx {
  sdsat_config cfg{};
  bool has_weights = false;
  sdsat_weights w{};
  std::vector<sdsat_layer_weights> layers;
  std::vector<LayerMaps> maps;
  CUtensorMap head_map{};
  cudaStream_t stream = nullptr;
  int device = 0, num_sms = 0;
  bool pdl = true;   // programmatic dependent launch between consecutive kernels
  // workspaces
  float2* rope = nullptr;
  float* h = nullptr;
  float* qbuf = nullptr;
  float* attn = nullptr;
  float* act = nullptr;
  float* partials = nullptr;
  int* gemm_counters = nullptr;
  float* ssq = nullptr;        // [SDSAT_MAX_ROWS][ssq_ld] per-tile sums of h^2 (RMSNorm folded into the GEMMs)
  int ssq_ld = 0;
  int* acc_targets = nullptr;
  int* acc_counters = nullptr;
  int* tree_pos = nullptr;     // [SDSAT_MAX_ROWS] tree block positions (len + depth)
  uint32_t* tree_anc = nullptr;   // [SDSAT_MAX_ROWS] tree block attention masks
  int* tree_ws = nullptr;      // [SDSAT_MAX_ROWS][TREE_WS_STRIDE] tree commit: len, m, path
  int* adaptive = nullptr;
  uint32_t* err = nullptr;
  // prefill workspaces (chunks of up to PF_ROWS positions; allocated with the weights)
  float* pf_h = nullptr;         // [PF_ROWS][d] residual stream
  float* pf_qkv = nullptr;       // [PF_ROWS][3R] projections before RoPE
  float* pf_q = nullptr;         // [PF_ROWS][R] rotated queries
  float* pf_attn = nullptr;      // [PF_ROWS][R] attention output
  __nv_bfloat16* pf_hi[X_COUNT] = {};   // GEMM operands [PF_ROWS][K] (normed x, attention, act)
  __nv_bfloat16* pf_lo[X_COUNT] = {};
  CUtensorMap pf_xmap[X_COUNT][2];      // boxes of 64 x 128
  __nv_bfloat16* x_hi[X_COUNT] = {};
  __nv_bfloat16* x_lo[X_COUNT] = {};
  CUtensorMap xmap[X_COUNT][3][2];     // [source][MPAD 16/32/64][hi/lo]
  __nv_bfloat16* xop_hi = nullptr;     // operand scratch of sdsat_op_gemm
  __nv_bfloat16* xop_lo = nullptr;
  std::vector<void*> allocs;
  // device trace (opt-in)
  unsigned long long* trace_rec = nullptr;
  unsigned int* trace_count = nullptr;
  unsigned int trace_cap = 0;
  unsigned int trace_seq = 0;
  // profiling hook
  bool prof = false;
  std::vector<cudaEvent_t> prof_events;
  std::vector<int> prof_class;
  size_t prof_used = 0;
};

struct sdsat_kv {
  sdsat_ctx* ctx = nullptr;
  int batch = 0, cap = 0;
  __nv_bfloat16* k = nullptr;
  __nv_bfloat16* v = nullptr;
  int* len = nullptr;
  long long* emitted = nullptr;
  CUtensorMap kmap, vmap;   // the caches as 2-D tensors for the attention kernel
};

namespace {

// trace descriptor for the next launch of kernel class `cls` (empty when tracing is off)
Trace next_trace(sdsat_ctx* c, int cls) {
  Trace t{};
  if (c->trace_rec) {
    t.rec = c->trace_rec;
    t.count = c->trace_count;
    t.cap = c->trace_cap;
    t.tag = ((unsigned)cls << 24) | (c->trace_seq++ & 0xFFFFFFu);
  }
  return t;
}

// Run one kernel launch, bracketed by profiling events when the hook is on.
template <typename F>
cudaError_t timed(sdsat_ctx* c, int cls, F&& launch) {
  if (!c->prof || 2 * (c->prof_used + 1) > c->prof_events.size()) return launch();
  const size_t i = c->prof_used++;
  cudaEventRecord(c->prof_events[2 * i], c->stream);
  const cudaError_t e = launch();
  cudaEventRecord(c->prof_events[2 * i + 1], c->stream);
  c->prof_class[i] = cls;
  return e;
}

template <typename T>
bool dalloc(sdsat_ctx* c, T** p, size_t count) {
  void* q = nullptr;
  if (cudaMalloc(&q, std::max<size_t>(count, 1) * sizeof(T)) != cudaSuccess) {
    cudaGetLastError();   // clear the runtime's record of the failed allocation (not sticky)
    return false;
  }
  if (cudaMemset(q, 0, std::max<size_t>(count, 1) * sizeof(T)) != cudaSuccess) {
    cudaFree(q);
    return false;
  }
  c->allocs.push_back(q);
  *p = static_cast<T*>(q);
  return true;
}

sdsat_status check_cfg(const sdsat_config& c) {
  if (c.n_layers < 1 || c.d_model < 8 || c.n_heads < 1 || c.head_dim < 1 || c.ffn_dim < 8 || c.vocab < 2 ||
      c.max_position < 1 || c.n_adaptive < 1 || c.n_adaptive > SDSAT_MAX_ADAPTIVE || !(c.rms_eps >= 0.f) ||
      !(c.rope_theta > 0.f))
    return SDSAT_EINVAL;
  if (c.d_model % 8 || c.ffn_dim % 8) return SDSAT_EINVAL;
  if (c.d_model > 64 * 128) return SDSAT_EUNSUPPORTED;   // the folded RMSNorm keeps <= 64 tile sums per row
  if (c.n_kv_heads != c.n_heads) return SDSAT_EUNSUPPORTED;
  if (c.head_dim != 64 && c.head_dim != 128) return SDSAT_EUNSUPPORTED;
  if ((c.n_heads * c.head_dim) % 128) return SDSAT_EUNSUPPORTED;
  for (int i = 0; i < c.n_adaptive; ++i)
    if (c.adaptive_ids[i] < 0 || c.adaptive_ids[i] >= c.vocab) return SDSAT_EINVAL;
  return SDSAT_OK;
}

GemmParams gemm_base(sdsat_ctx* c, int M, int xsrc) {
  GemmParams g;
  std::memset(&g, 0, sizeof(g));
  g.M = M;
  g.partials = c->partials;
  g.counters = c->gemm_counters;
  g.err = c->err;
  if (xsrc >= 0) {
    g.tmap_x[0] = c->xmap[xsrc][mpad_index(M)][0];
    g.tmap_x[1] = c->xmap[xsrc][mpad_index(M)][1];
  }
  return g;
}

void set_plain(GemmParams& g, const CUtensorMap& m, int N, int K) {
  g.tmap[0] = m;
  g.map_mode = MAP_PLAIN;
  g.N = N;
  g.K = K;
  g.n_tiles = (N + 127) / 128;
  g.kc = (K + 63) / 64;
}

// one block forward of sequences seq0 .. seq0+nb-1, q rows each (anc: tree attention masks)
sdsat_status forward(sdsat_ctx* c, sdsat_kv* kv, int seq0, int nb, int q, const int32_t* tokens,
                     const int32_t* positions, float* logits, const uint32_t* anc = nullptr) {
  const sdsat_config& cf = c->cfg;
  const int M = nb * q, d = cf.d_model, H = cf.n_heads, hd = cf.head_dim, F = cf.ffn_dim, R = H * hd, L = cf.n_layers;
  cudaStream_t st = c->stream;
  const size_t layer_elems = (size_t)kv->batch * H * kv->cap * hd;
  auto norm = [&](const int32_t* toks, const void* gain) {
    return timed(c, K_RMSNORM, [&] {
      return launch_rmsnorm(toks, static_cast<const __nv_bfloat16*>(c->w.embed), cf.vocab, c->h, d, M,
                            static_cast<const __nv_bfloat16*>(gain), cf.rms_eps, c->x_hi[X_NORM], c->x_lo[X_NORM],
                            c->err, st, c->pdl);
    });
  };
  // The residual-producing GEMMs (O, down) also emit the next RMSNorm's operand h * g
  // and per-tile sums of h^2; the consuming GEMM (gate/up, the next QKV, the LM head)
  // scales its result rows by the RMSNorm factor.  Only the first norm is a kernel,
  // fused with the embedding gather.
  auto fold_in = [&](GemmParams& g) {
    g.ssq_in = c->ssq;
    g.ssq_n = c->ssq_ld;
    g.ssq_ld = c->ssq_ld;
    g.norm_dim = d;
    g.norm_eps = cf.rms_eps;
  };
  auto fold_out = [&](GemmParams& g, const void* gain) {
    g.gain_next = static_cast<const __nv_bfloat16*>(gain);
    g.xn_hi = c->x_hi[X_NORM];
    g.xn_lo = c->x_lo[X_NORM];
    g.ssq_out = c->ssq;
    g.ssq_ld = c->ssq_ld;
  };
  // QKV projection with RoPE and the KV append fused into its epilogue
  auto make_qkv = [&](int l) {
    const LayerMaps& mp = c->maps[l];
    GemmParams g = gemm_base(c, M, X_NORM);
    g.tmap[0] = mp.q;
    g.tmap[1] = mp.k;
    g.tmap[2] = mp.v;
    g.map_mode = MAP_QKV3;
    g.N = 3 * R;
    g.K = d;
    g.rows_per_map = R;
    g.n_tiles = 3 * R / 128;
    g.kc = (d + 63) / 64;
    g.epi = EPI_QKV;
    g.out = c->qbuf;
    g.out_ld = R;
    g.k_layer = kv->k + l * layer_elems;
    g.v_layer = kv->v + l * layer_elems;
    g.H = H;
    g.hd = hd;
    g.cap = kv->cap;
    g.q = q;
    g.seq0 = seq0;
    g.len = kv->len;
    g.positions = positions;
    g.rope = c->rope;
    g.rope_len = cf.max_position;
    if (l > 0) fold_in(g);
    return g;
  };
  // O projection + residual
  auto make_o = [&](int l) {
    GemmParams g = gemm_base(c, M, X_ATTN);
    set_plain(g, c->maps[l].o, d, R);
    g.epi = EPI_RESID;
    g.out = c->h;
    g.out_ld = d;
    fold_out(g, c->layers[l].ffn_norm);
    return g;
  };
  // gate/up with SiLU(gate) * up fused; emits the down projection's operand
  auto make_gateup = [&](int l) {
    GemmParams g = gemm_base(c, M, X_NORM);
    g.tmap[0] = c->maps[l].gate;
    g.tmap[1] = c->maps[l].up;
    g.map_mode = MAP_GATEUP;
    g.N = F;
    g.K = d;
    g.n_tiles = (F + 63) / 64;
    g.kc = (d + 63) / 64;
    g.epi = EPI_SWIGLU;
    g.out = c->act;
    g.out_ld = F;
    g.out_hi = c->x_hi[X_FFN];
    g.out_lo = c->x_lo[X_FFN];
    fold_in(g);
    return g;
  };
  // down projection + residual, emitting the next layer's attention RMSNorm operand (or
  // the final RMSNorm's before the LM head)
  auto make_down = [&](int l) {
    GemmParams g = gemm_base(c, M, X_FFN);
    set_plain(g, c->maps[l].down, d, F);
    g.epi = EPI_RESID;
    g.out = c->h;
    g.out_ld = d;
    fold_out(g, l + 1 < L ? c->layers[l + 1].attn_norm : c->w.final_norm);
    return g;
  };
  auto make_head = [&]() {
    GemmParams g = gemm_base(c, M, X_NORM);
    set_plain(g, c->head_map, cf.vocab, d);
    fold_in(g);
    g.epi = EPI_STORE;
    g.out = logits;
    g.out_ld = cf.vocab;
    return g;
  };
  auto gemm = [&](GemmParams& g, int cls) {
    g.trace = next_trace(c, cls);
    return timed(c, cls, [&] { return launch_gemm(g, c->num_sms, st, c->pdl); });
  };
  if (norm(tokens, c->layers[0].attn_norm) != cudaSuccess) return SDSAT_ECUDA;
  GemmParams gq = make_qkv(0);
  for (int l = 0; l < L; ++l) {
    GemmParams go = make_o(l), gg = make_gateup(l), gd = make_down(l), gn{};
    if (l + 1 < L) gn = make_qkv(l + 1);
    else if (logits) gn = make_head();
    if (gemm(gq, K_GEMM_QKV) != cudaSuccess) return SDSAT_ECUDA;
    // block-causal attention; its merge emits the O projection's operand
    AttnParams a;
    std::memset(&a, 0, sizeof(a));
    a.kmap = kv->kmap;
    a.vmap = kv->vmap;
    a.row0 = l * kv->batch * H * kv->cap;
    a.Q = c->qbuf;
    a.q_ld = R;
    a.len = kv->len;
    a.anc = anc;
    a.seq0 = seq0;
    a.nb = nb;
    a.q = q;
    a.H = H;
    a.hd = hd;
    a.cap = kv->cap;
    a.out = c->attn;
    a.out_ld = R;
    a.out_hi = c->x_hi[X_ATTN];
    a.out_lo = c->x_lo[X_ATTN];
    a.err = c->err;
    a.trace = next_trace(c, K_ATTENTION);
    if (timed(c, K_ATTENTION, [&] { return launch_attention(a, c->num_sms, st, c->pdl); }) != cudaSuccess)
      return SDSAT_ECUDA;
    if (gemm(go, K_GEMM_O) != cudaSuccess || gemm(gg, K_GEMM_GATEUP) != cudaSuccess ||
        gemm(gd, K_GEMM_DOWN) != cudaSuccess)
      return SDSAT_ECUDA;
    gq = gn;
  }
  if (logits && gemm(gq, K_GEMM_LM_HEAD) != cudaSuccess) return SDSAT_ECUDA;
  return SDSAT_OK;
}

// one prefill chunk: M (a multiple of SDSAT_MAX_Q, <= PF_ROWS) prompt positions of sequence seq
// through every layer on the tiled GEMM, then committed
sdsat_status prefill_chunk(sdsat_ctx* c, sdsat_kv* kv, int seq, const int32_t* tokens, int M) {
  const sdsat_config& cf = c->cfg;
  const int d = cf.d_model, H = cf.n_heads, hd = cf.head_dim, F = cf.ffn_dim, R = H * hd, L = cf.n_layers;
  cudaStream_t st = c->stream;
  const size_t layer_elems = (size_t)kv->batch * H * kv->cap * hd;
  const int ntb = (M + 127) / 128;
  auto norm = [&](const int32_t* toks, const void* gain) {
    return timed(c, K_RMSNORM, [&] {
      return launch_rmsnorm(toks, static_cast<const __nv_bfloat16*>(c->w.embed), cf.vocab, c->pf_h, d, M,
                            static_cast<const __nv_bfloat16*>(gain), cf.rms_eps, c->pf_hi[X_NORM], c->pf_lo[X_NORM],
                            c->err, st, c->pdl);
    });
  };
  auto base = [&](int xsrc, int K) {
    PfGemmParams g;
    std::memset(&g, 0, sizeof(g));
    g.tmap_x[0] = c->pf_xmap[xsrc][0];
    g.tmap_x[1] = c->pf_xmap[xsrc][1];
    g.kc = (K + 63) / 64;
    g.n_tblocks = ntb;
    g.M = M;
    g.err = c->err;
    return g;
  };
  auto gemm = [&](PfGemmParams& g) {
    return timed(c, K_PF_GEMM, [&] { return launch_prefill_gemm(g, c->num_sms, st, c->pdl); });
  };
  if (norm(tokens, c->layers[0].attn_norm) != cudaSuccess) return SDSAT_ECUDA;
  for (int l = 0; l < L; ++l) {
    const LayerMaps& mp = c->maps[l];
    PfGemmParams gq = base(X_NORM, d);
    gq.tmap[0] = mp.q;
    gq.tmap[1] = mp.k;
    gq.tmap[2] = mp.v;
    gq.map_mode = MAP_QKV3;
    gq.rows_per_map = R;
    gq.N = 3 * R;
    gq.n_wtiles = 3 * R / 128;
    gq.epi = EPI_STORE;
    gq.out = c->pf_qkv;
    gq.out_ld = 3 * R;
    if (gemm(gq) != cudaSuccess) return SDSAT_ECUDA;
    RopeKvParams rp{c->pf_qkv, c->pf_q, kv->k + l * layer_elems, kv->v + l * layer_elems, kv->len, seq, H, hd,
                    kv->cap, c->rope, cf.max_position, c->err};
    if (timed(c, K_PF_ROPE_KV, [&] { return launch_rope_kv(rp, M, st, c->pdl); }) != cudaSuccess) return SDSAT_ECUDA;
    // causal attention of the chunk's positions over the cache
    PfAttnParams a;
    std::memset(&a, 0, sizeof(a));
    a.kmap = kv->kmap;
    a.vmap = kv->vmap;
    a.row0 = l * kv->batch * H * kv->cap;
    a.Q = c->pf_q;
    a.q_ld = R;
    a.len = kv->len;
    a.seq = seq;
    a.M = M;
    a.H = H;
    a.hd = hd;
    a.cap = kv->cap;
    a.out = c->pf_attn;
    a.out_ld = R;
    a.out_hi = c->pf_hi[X_ATTN];
    a.out_lo = c->pf_lo[X_ATTN];
    a.err = c->err;
    if (timed(c, K_PF_ATTENTION, [&] { return launch_prefill_attention(a, st, c->pdl); }) != cudaSuccess)
      return SDSAT_ECUDA;
    PfGemmParams go = base(X_ATTN, R);
    go.tmap[0] = mp.o;
    go.map_mode = MAP_PLAIN;
    go.N = d;
    go.n_wtiles = (d + 127) / 128;
    go.epi = EPI_RESID;
    go.out = c->pf_h;
    go.out_ld = d;
    if (gemm(go) != cudaSuccess) return SDSAT_ECUDA;
    if (norm(nullptr, c->layers[l].ffn_norm) != cudaSuccess) return SDSAT_ECUDA;
    PfGemmParams gg = base(X_NORM, d);
    gg.tmap[0] = mp.gate;
    gg.tmap[1] = mp.up;
    gg.map_mode = MAP_GATEUP;
    gg.N = F;
    gg.n_wtiles = (F + 63) / 64;
    gg.epi = EPI_SWIGLU;
    gg.out_hi = c->pf_hi[X_FFN];
    gg.out_lo = c->pf_lo[X_FFN];
    gg.out_ld = F;
    if (gemm(gg) != cudaSuccess) return SDSAT_ECUDA;
    PfGemmParams gd = base(X_FFN, F);
    gd.tmap[0] = mp.down;
    gd.map_mode = MAP_PLAIN;
    gd.N = d;
    gd.n_wtiles = (d + 127) / 128;
    gd.epi = EPI_RESID;
    gd.out = c->pf_h;
    gd.out_ld = d;
    if (gemm(gd) != cudaSuccess) return SDSAT_ECUDA;
    if (l + 1 < L && norm(nullptr, c->layers[l + 1].attn_norm) != cudaSuccess) return SDSAT_ECUDA;
  }
  return timed(c, K_PREFILL_COMMIT, [&] { return launch_add_len(kv->len, seq, M, kv->cap, c->err, st, c->pdl); }) ==
                 cudaSuccess
             ? SDSAT_OK
             : SDSAT_ECUDA;
}

sdsat_status accept_common(sdsat_ctx* c, sdsat_kv* kv, const float* logits, const int32_t* drafts, int b, int q,
                           int n_verify, float top_p, float temperature, uint64_t seed, int top_k, int32_t* acc,
                           int32_t* out, int commit, const int32_t* parent = nullptr, int32_t* path = nullptr,
                           const int32_t* n_verify_dev = nullptr) {
  if (!c || !kv || kv->ctx != c || !logits || !drafts || !acc || !out) return SDSAT_EINVAL;
  if (b < 1 || b > kv->batch || q < 1 || q > SDSAT_MAX_Q || b * q > SDSAT_MAX_ROWS) return SDSAT_EINVAL;
  if (n_verify < 0 || n_verify >= q || top_k < 0) return SDSAT_EINVAL;
  if (temperature > 0.f && !(top_p >= 0.f)) return SDSAT_EINVAL;
  if (temperature > 0.f && c->cfg.vocab > 32768) return SDSAT_EUNSUPPORTED;
  AcceptParams p;
  std::memset(&p, 0, sizeof(p));
  p.logits = logits;
  p.drafts = drafts;
  p.seq0 = 0;
  p.nb = b;
  p.q = q;
  p.V = c->cfg.vocab;
  p.n_verify = n_verify;
  p.temperature = temperature;
  p.top_p = top_p;
  const double pf = std::nearbyint((double)top_p * 16777216.0);
  p.p_fixed = (uint32_t)std::min(std::max(pf, 0.0), 16777216.0);
  p.seed = seed;
  p.top_k = top_k;
  p.len = kv->len;
  p.cap = kv->cap;
  p.commit = commit;
  p.accepted_len = acc;
  p.out_tokens = out;
  p.targets = c->acc_targets;
  p.counters = c->acc_counters;
  p.err = c->err;
  p.emitted = kv->emitted;
  p.parent = parent;
  p.path = path;
  p.n_verify_dev = n_verify_dev;
  p.tree_ws = c->tree_ws;
  if (timed(c, K_ACCEPT, [&] { return launch_accept(p, c->stream, c->pdl); }) != cudaSuccess) return SDSAT_ECUDA;
  if (!parent) return SDSAT_OK;
  const sdsat_config& cf = c->cfg;
  return timed(c, K_TREE_COMPACT, [&] {
           return launch_tree_compact(c->tree_ws, b, cf.n_layers, cf.n_heads, cf.head_dim, kv->cap, kv->batch, kv->k,
                                      kv->v, c->stream, c->pdl);
         }) == cudaSuccess
             ? SDSAT_OK
             : SDSAT_ECUDA;
}

}  // namespace

extern "C" {

const char* sdsat_status_string(sdsat_status s) {
  switch (s) {
    case SDSAT_OK: return "ok";
    case SDSAT_EINVAL: return "invalid argument";
    case SDSAT_ENOMEM: return "device allocation failed";
    case SDSAT_ECAPACITY: return "capacity exceeded";
    case SDSAT_ECUDA: return "CUDA error";
    case SDSAT_EDEVICE: return "device-detected error";
    case SDSAT_EUNSUPPORTED: return "unsupported configuration";
  }
  return "unknown status";
}

void sdsat_destroy(sdsat_ctx* c) {
  if (!c) return;
  cudaStreamSynchronize(c->stream);
  for (cudaEvent_t e : c->prof_events) cudaEventDestroy(e);
  cudaFree(c->trace_rec);
  cudaFree(c->trace_count);
  for (void* p : c->allocs) cudaFree(p);
  delete c;
}

sdsat_status sdsat_create(const sdsat_config* cfg, const sdsat_weights* w, void* stream, sdsat_ctx** out) {
  if (!cfg || !out) return SDSAT_EINVAL;
  *out = nullptr;
  const sdsat_status cs = check_cfg(*cfg);
  if (cs != SDSAT_OK) return cs;
  sdsat_ctx* c = new (std::nothrow) sdsat_ctx();
  if (!c) return SDSAT_ENOMEM;
  c->cfg = *cfg;
  c->stream = static_cast<cudaStream_t>(stream);
  {
    const char* e = std::getenv("SDSAT_NO_PDL");   // e.g. for tools that cannot follow PDL launches
    c->pdl = !(e && e[0] && e[0] != '0');
  }
  if (cudaGetDevice(&c->device) != cudaSuccess ||
      cudaDeviceGetAttribute(&c->num_sms, cudaDevAttrMultiProcessorCount, c->device) != cudaSuccess ||
      gemm_prepare() != cudaSuccess || attention_prepare() != cudaSuccess || prefill_prepare() != cudaSuccess) {
    delete c;
    return SDSAT_ECUDA;
  }
  const int L = cfg->n_layers, d = cfg->d_model, R = cfg->n_heads * cfg->head_dim, F = cfg->ffn_dim;
  if (w) {
    if (!w->layers || !aligned16(w->embed) || !aligned16(w->final_norm) || !aligned16(w->lm_head)) {
      delete c;
      return SDSAT_EINVAL;
    }
    c->has_weights = true;
    c->w = *w;
    c->layers.assign(w->layers, w->layers + L);
    c->maps.resize(L);
    for (int l = 0; l < L; ++l) {
      const sdsat_layer_weights& W = c->layers[l];
      if (!aligned16(W.attn_norm) || !aligned16(W.ffn_norm) || !aligned16(W.wq) || !aligned16(W.wk) ||
          !aligned16(W.wv) || !aligned16(W.wo) || !aligned16(W.w_gate) || !aligned16(W.w_up) ||
          !aligned16(W.w_down)) {
        delete c;
        return SDSAT_EINVAL;
      }
      LayerMaps& m = c->maps[l];
      if (!make_wmap(&m.q, W.wq, R, d) || !make_wmap(&m.k, W.wk, R, d) || !make_wmap(&m.v, W.wv, R, d) ||
          !make_wmap(&m.o, W.wo, d, R) || !make_wmap(&m.gate, W.w_gate, F, d) || !make_wmap(&m.up, W.w_up, F, d) ||
          !make_wmap(&m.down, W.w_down, d, F)) {
        delete c;
        return SDSAT_ECUDA;
      }
    }
    if (!make_wmap(&c->head_map, w->lm_head, cfg->vocab, d)) {
      delete c;
      return SDSAT_ECUDA;
    }
  }
  // RoPE table: angle = pos * theta^(-2i/hd), computed in double
  const int half = cfg->head_dim / 2;
  std::vector<float2> rope((size_t)cfg->max_position * half);
  for (int p = 0; p < cfg->max_position; ++p)
    for (int i = 0; i < half; ++i) {
      const double ang = (double)p * std::pow((double)cfg->rope_theta, -2.0 * i / cfg->head_dim);
      rope[(size_t)p * half + i] = make_float2((float)std::cos(ang), (float)std::sin(ang));
    }
  const int rows = SDSAT_MAX_ROWS;
  c->ssq_ld = (d + 127) / 128;
  bool ok = dalloc(c, &c->rope, rope.size()) && dalloc(c, &c->h, (size_t)rows * d) &&
            dalloc(c, &c->qbuf, (size_t)rows * R) && dalloc(c, &c->attn, (size_t)rows * R) &&
            dalloc(c, &c->act, (size_t)rows * F) && dalloc(c, &c->partials, (size_t)c->num_sms * 2 * 2 * 64 * 128) &&
            dalloc(c, &c->gemm_counters, MAX_GEMM_TILES) &&
            dalloc(c, &c->acc_targets, rows) &&
            dalloc(c, &c->acc_counters, rows) && dalloc(c, &c->adaptive, SDSAT_MAX_ADAPTIVE) &&
            dalloc(c, &c->tree_pos, rows) && dalloc(c, &c->tree_anc, rows) &&
            dalloc(c, &c->tree_ws, (size_t)rows * TREE_WS_STRIDE) &&
            dalloc(c, &c->err, 1) && dalloc(c, &c->xop_hi, (size_t)PF_ROWS * OP_MAX_K) &&
            dalloc(c, &c->ssq, (size_t)rows * ((d + 127) / 128)) &&
            dalloc(c, &c->xop_lo, (size_t)PF_ROWS * OP_MAX_K);
  const int xcols[X_COUNT] = {d, R, F};
  for (int xs = 0; ok && xs < X_COUNT; ++xs) {
    ok = dalloc(c, &c->x_hi[xs], (size_t)rows * xcols[xs]) && dalloc(c, &c->x_lo[xs], (size_t)rows * xcols[xs]);
    for (int mi = 0; ok && mi < 3; ++mi)
      ok = make_xmap(&c->xmap[xs][mi][0], c->x_hi[xs], rows, xcols[xs], 16 << mi) &&
           make_xmap(&c->xmap[xs][mi][1], c->x_lo[xs], rows, xcols[xs], 16 << mi);
  }
  if (ok && c->has_weights) {
    const int pr = PF_ROWS;
    ok = dalloc(c, &c->pf_h, (size_t)pr * d) && dalloc(c, &c->pf_qkv, (size_t)pr * 3 * R) &&
         dalloc(c, &c->pf_q, (size_t)pr * R) && dalloc(c, &c->pf_attn, (size_t)pr * R);
    for (int xs = 0; ok && xs < X_COUNT; ++xs)
      ok = dalloc(c, &c->pf_hi[xs], (size_t)pr * xcols[xs]) && dalloc(c, &c->pf_lo[xs], (size_t)pr * xcols[xs]) &&
           make_xmap(&c->pf_xmap[xs][0], c->pf_hi[xs], pr, xcols[xs], 128) &&
           make_xmap(&c->pf_xmap[xs][1], c->pf_lo[xs], pr, xcols[xs], 128);
  }
  if (!ok) {
    sdsat_destroy(c);
    return SDSAT_ENOMEM;
  }
  int ids[SDSAT_MAX_ADAPTIVE];
  for (int i = 0; i < SDSAT_MAX_ADAPTIVE; ++i)
    ids[i] = cfg->n_adaptive == 1 ? cfg->adaptive_ids[0] : cfg->adaptive_ids[std::min(i, cfg->n_adaptive - 1)];
  if (cudaMemcpy(c->rope, rope.data(), rope.size() * sizeof(float2), cudaMemcpyHostToDevice) != cudaSuccess ||
      cudaMemcpy(c->adaptive, ids, sizeof(ids), cudaMemcpyHostToDevice) != cudaSuccess ||
      cudaDeviceSynchronize() != cudaSuccess) {
    sdsat_destroy(c);
    return SDSAT_ECUDA;
  }
  *out = c;
  return SDSAT_OK;
}

sdsat_status sdsat_set_stream(sdsat_ctx* c, void* stream) {
  if (!c) return SDSAT_EINVAL;
  c->stream = static_cast<cudaStream_t>(stream);
  return SDSAT_OK;
}

sdsat_status sdsat_kv_create(sdsat_ctx* c, int batch, int max_len, sdsat_kv** out) {
  if (!c || !out || batch < 1 || max_len < 1) return SDSAT_EINVAL;
  *out = nullptr;
  if (max_len > c->cfg.max_position || max_len > ATT_MAX_CAP) return SDSAT_ECAPACITY;
  sdsat_kv* kv = new (std::nothrow) sdsat_kv();
  if (!kv) return SDSAT_ENOMEM;
  kv->ctx = c;
  kv->batch = batch;
  kv->cap = max_len;
  const size_t n = (size_t)c->cfg.n_layers * batch * c->cfg.n_heads * max_len * c->cfg.head_dim;
  void *k = nullptr, *v = nullptr, *len = nullptr, *em = nullptr;
  if (cudaMalloc(&k, n * 2) != cudaSuccess || cudaMalloc(&v, n * 2) != cudaSuccess ||
      cudaMalloc(&len, batch * sizeof(int)) != cudaSuccess || cudaMalloc(&em, batch * sizeof(long long)) != cudaSuccess) {
    cudaGetLastError();   // clear the runtime's record of the failed allocation (not sticky)
    cudaFree(k);
    cudaFree(v);
    cudaFree(len);
    cudaFree(em);
    delete kv;
    return SDSAT_ENOMEM;
  }
  if (cudaMemset(k, 0, n * 2) != cudaSuccess || cudaMemset(v, 0, n * 2) != cudaSuccess ||
      cudaMemset(len, 0, batch * sizeof(int)) != cudaSuccess ||
      cudaMemset(em, 0, batch * sizeof(long long)) != cudaSuccess || cudaDeviceSynchronize() != cudaSuccess) {
    cudaFree(k);
    cudaFree(v);
    cudaFree(len);
    cudaFree(em);
    delete kv;
    return SDSAT_ECUDA;
  }
  kv->emitted = static_cast<long long*>(em);
  const long long rows = (long long)c->cfg.n_layers * batch * c->cfg.n_heads * max_len;
  if (rows > 0x7FFFFFFFll || !make_kvmap(&kv->kmap, k, rows, c->cfg.head_dim) ||
      !make_kvmap(&kv->vmap, v, rows, c->cfg.head_dim)) {
    cudaFree(k);
    cudaFree(v);
    cudaFree(len);
    cudaFree(em);
    delete kv;
    return SDSAT_EUNSUPPORTED;
  }
  kv->k = static_cast<__nv_bfloat16*>(k);
  kv->v = static_cast<__nv_bfloat16*>(v);
  kv->len = static_cast<int*>(len);
  *out = kv;
  return SDSAT_OK;
}

void sdsat_kv_destroy(sdsat_kv* kv) {
  if (!kv) return;
  cudaStreamSynchronize(kv->ctx->stream);
  cudaFree(kv->k);
  cudaFree(kv->v);
  cudaFree(kv->len);
  cudaFree(kv->emitted);
  delete kv;
}

sdsat_status sdsat_kv_info(const sdsat_kv* kv, void** k_dev, void** v_dev, int32_t** len_dev, int* batch,
                           int* max_len) {
  if (!kv) return SDSAT_EINVAL;
  if (k_dev) *k_dev = kv->k;
  if (v_dev) *v_dev = kv->v;
  if (len_dev) *len_dev = kv->len;
  if (batch) *batch = kv->batch;
  if (max_len) *max_len = kv->cap;
  return SDSAT_OK;
}

static sdsat_status kv_copy(sdsat_ctx* c, const sdsat_kv* kv, int layer, int seq, int slot0, int n, const void* ks,
                            const void* vs, void* kd, void* vd) {
  if (!c || !kv || kv->ctx != c || layer < 0 || layer >= c->cfg.n_layers || seq < 0 || seq >= kv->batch ||
      slot0 < 0 || n < 0 || slot0 + n > kv->cap)
    return SDSAT_EINVAL;
  if (n == 0) return SDSAT_OK;
  const int H = c->cfg.n_heads, hd = c->cfg.head_dim;
  const size_t layer_elems = (size_t)kv->batch * H * kv->cap * hd;
  const size_t off = layer * layer_elems + ((size_t)seq * H * kv->cap + slot0) * hd;
  const size_t cache_pitch = (size_t)kv->cap * hd * 2, buf_pitch = (size_t)n * hd * 2, width = buf_pitch;
  for (int which = 0; which < 2; ++which) {
    __nv_bfloat16* cache = (which == 0 ? kv->k : kv->v) + off;
    cudaError_t e;
    if (ks || vs) {
      e = cudaMemcpy2DAsync(cache, cache_pitch, which == 0 ? ks : vs, buf_pitch, width, H, cudaMemcpyDeviceToDevice,
                            c->stream);
    } else {
      e = cudaMemcpy2DAsync(which == 0 ? kd : vd, buf_pitch, cache, cache_pitch, width, H, cudaMemcpyDeviceToDevice,
                            c->stream);
    }
    if (e != cudaSuccess) return SDSAT_ECUDA;
  }
  return SDSAT_OK;
}

sdsat_status sdsat_kv_write(sdsat_ctx* c, sdsat_kv* kv, int layer, int seq, int slot0, int n, const void* k_src_dev,
                            const void* v_src_dev) {
  if (!k_src_dev || !v_src_dev) return SDSAT_EINVAL;
  return kv_copy(c, kv, layer, seq, slot0, n, k_src_dev, v_src_dev, nullptr, nullptr);
}

sdsat_status sdsat_kv_read(sdsat_ctx* c, const sdsat_kv* kv, int layer, int seq, int slot0, int n, void* k_dst_dev,
                           void* v_dst_dev) {
  if (!k_dst_dev || !v_dst_dev) return SDSAT_EINVAL;
  return kv_copy(c, kv, layer, seq, slot0, n, nullptr, nullptr, k_dst_dev, v_dst_dev);
}

sdsat_status sdsat_block_forward(sdsat_ctx* c, sdsat_kv* kv, const int32_t* tokens_dev,
                                 const int32_t* positions_dev, int b, int q, float* logits_dev) {
  if (!c || !kv || kv->ctx != c || !c->has_weights || !tokens_dev || !logits_dev) return SDSAT_EINVAL;
  if (b < 1 || b > kv->batch || q < 1 || q > SDSAT_MAX_Q || b * q > SDSAT_MAX_ROWS) return SDSAT_EINVAL;
  return forward(c, kv, 0, b, q, tokens_dev, positions_dev, logits_dev);
}

sdsat_status sdsat_block_forward_tree(sdsat_ctx* c, sdsat_kv* kv, const int32_t* tokens_dev,
                                      const int32_t* parent_dev, int b, int q, float* logits_dev) {
  if (!c || !kv || kv->ctx != c || !c->has_weights || !tokens_dev || !parent_dev || !logits_dev) return SDSAT_EINVAL;
  if (b < 1 || b > kv->batch || q < 1 || q > SDSAT_MAX_Q || b * q > SDSAT_MAX_ROWS) return SDSAT_EINVAL;
  if (timed(c, K_TREE_PREP, [&] {
        return launch_tree_prep(parent_dev, kv->len, b, q, c->tree_pos, c->tree_anc, c->err, c->stream, c->pdl);
      }) != cudaSuccess)
    return SDSAT_ECUDA;
  return forward(c, kv, 0, b, q, tokens_dev, c->tree_pos, logits_dev, c->tree_anc);
}

sdsat_status sdsat_prefill(sdsat_ctx* c, sdsat_kv* kv, int seq, const int32_t* tokens_dev, int n) {
  if (!c || !kv || kv->ctx != c || !c->has_weights || !tokens_dev || seq < 0 || seq >= kv->batch || n < 0)
    return SDSAT_EINVAL;
  if (n > kv->cap) return SDSAT_ECAPACITY;
  // chunks of up to PF_ROWS positions (a multiple of SDSAT_MAX_Q) on the tiled GEMM; a tail
  // shorter than SDSAT_MAX_Q runs as one ordinary block
  for (int i = 0; i < n;) {
    const int rem = n - i;
    if (rem >= SDSAT_MAX_Q) {
      const int M = std::min(PF_ROWS, rem / SDSAT_MAX_Q * SDSAT_MAX_Q);
      const sdsat_status s = prefill_chunk(c, kv, seq, tokens_dev + i, M);
      if (s != SDSAT_OK) return s;
      i += M;
      continue;
    }
    const sdsat_status s = forward(c, kv, seq, 1, rem, tokens_dev + i, nullptr, nullptr);
    if (s != SDSAT_OK) return s;
    if (timed(c, K_PREFILL_COMMIT, [&] { return launch_add_len(kv->len, seq, rem, kv->cap, c->err, c->stream, c->pdl); }) !=
        cudaSuccess)
      return SDSAT_ECUDA;
    i += rem;
  }
  return SDSAT_OK;
}

sdsat_status sdsat_accept_greedy(sdsat_ctx* c, sdsat_kv* kv, const float* logits_dev, const int32_t* drafts_dev,
                                 int b, int q, int n_verify, int32_t* accepted_len_dev, int32_t* out_tokens_dev,
                                 int commit) {
  return accept_common(c, kv, logits_dev, drafts_dev, b, q, n_verify, 1.f, 0.f, 0, 0, accepted_len_dev,
                       out_tokens_dev, commit);
}

sdsat_status sdsat_accept_nucleus(sdsat_ctx* c, sdsat_kv* kv, const float* logits_dev, const int32_t* drafts_dev,
                                  int b, int q, int n_verify, float top_p, float temperature, uint64_t rng_seed,
                                  int top_k, int32_t* accepted_len_dev, int32_t* out_tokens_dev, int commit) {
  return accept_common(c, kv, logits_dev, drafts_dev, b, q, n_verify, top_p, temperature, rng_seed, top_k,
                       accepted_len_dev, out_tokens_dev, commit);
}

sdsat_status sdsat_accept_tree(sdsat_ctx* c, sdsat_kv* kv, const float* logits_dev, const int32_t* tokens_dev,
                               const int32_t* parent_dev, int b, int q, float temperature, float top_p,
                               uint64_t rng_seed, int top_k, int32_t* accepted_len_dev, int32_t* out_tokens_dev,
                               int32_t* path_dev, int commit) {
  if (!parent_dev || !(temperature >= 0.f)) return SDSAT_EINVAL;
  return accept_common(c, kv, logits_dev, tokens_dev, b, q, q - 1, temperature > 0.f ? top_p : 1.f,
                       temperature, rng_seed, top_k, accepted_len_dev, out_tokens_dev, commit, parent_dev, path_dev);
}

sdsat_status sdsat_accept_pipelined(sdsat_ctx* c, sdsat_kv* kv, const float* logits_dev, const int32_t* tokens_dev,
                                    const int32_t* n_verify_dev, int b, int q, float temperature, float top_p,
                                    uint64_t rng_seed, int top_k, int32_t* accepted_len_dev, int32_t* out_tokens_dev,
                                    int commit) {
  if (!n_verify_dev || !(temperature >= 0.f) || q < 2) return SDSAT_EINVAL;
  return accept_common(c, kv, logits_dev, tokens_dev, b, q, q - 1, temperature > 0.f ? top_p : 1.f, temperature,
                       rng_seed, top_k, accepted_len_dev, out_tokens_dev, commit, nullptr, nullptr, n_verify_dev);
}

sdsat_status sdsat_kv_commit(sdsat_ctx* c, sdsat_kv* kv, const int32_t* new_len_dev, int b) {
  if (!c || !kv || kv->ctx != c || !new_len_dev || b < 1 || b > kv->batch || b > 64) return SDSAT_EINVAL;
  return timed(c, K_KV_COMMIT, [&] { return launch_commit(kv->len, new_len_dev, b, kv->cap, c->err, c->stream, c->pdl); }) ==
                 cudaSuccess
             ? SDSAT_OK
             : SDSAT_ECUDA;
}

sdsat_status sdsat_kv_lengths(sdsat_ctx* c, const sdsat_kv* kv, int32_t* lens_dev, int b) {
  if (!c || !kv || kv->ctx != c || !lens_dev || b < 1 || b > kv->batch) return SDSAT_EINVAL;
  return cudaMemcpyAsync(lens_dev, kv->len, b * sizeof(int), cudaMemcpyDeviceToDevice, c->stream) == cudaSuccess
             ? SDSAT_OK
             : SDSAT_ECUDA;
}

sdsat_status sdsat_kv_emitted(sdsat_ctx* c, sdsat_kv* kv, int64_t* emitted_dev, int b, int reset) {
  if (!c || !kv || kv->ctx != c || !emitted_dev || b < 1 || b > kv->batch) return SDSAT_EINVAL;
  if (cudaMemcpyAsync(emitted_dev, kv->emitted, b * sizeof(long long), cudaMemcpyDeviceToDevice, c->stream) !=
      cudaSuccess)
    return SDSAT_ECUDA;
  if (reset && cudaMemsetAsync(kv->emitted, 0, b * sizeof(long long), c->stream) != cudaSuccess) return SDSAT_ECUDA;
  return SDSAT_OK;
}

sdsat_status sdsat_trace_begin(sdsat_ctx* c, int max_records) {
  if (!c || max_records < 1) return SDSAT_EINVAL;
  if (cudaStreamSynchronize(c->stream) != cudaSuccess) return SDSAT_ECUDA;
  cudaFree(c->trace_rec);
  cudaFree(c->trace_count);
  c->trace_rec = nullptr;
  c->trace_count = nullptr;
  void *r = nullptr, *n = nullptr;
  if (cudaMalloc(&r, (size_t)max_records * TRACE_WORDS * sizeof(unsigned long long)) != cudaSuccess) return SDSAT_ENOMEM;
  if (cudaMalloc(&n, sizeof(unsigned int)) != cudaSuccess || cudaMemset(n, 0, sizeof(unsigned int)) != cudaSuccess) {
    cudaFree(r);
    return SDSAT_ENOMEM;
  }
  c->trace_rec = static_cast<unsigned long long*>(r);
  c->trace_count = static_cast<unsigned int*>(n);
  c->trace_cap = (unsigned)max_records;
  c->trace_seq = 0;
  return SDSAT_OK;
}

sdsat_status sdsat_trace_end(sdsat_ctx* c, uint64_t* records, int max_records, int* n_records) {
  if (!c || !c->trace_rec) return SDSAT_EINVAL;
  unsigned int n = 0;
  if (cudaStreamSynchronize(c->stream) != cudaSuccess ||
      cudaMemcpy(&n, c->trace_count, sizeof(n), cudaMemcpyDeviceToHost) != cudaSuccess)
    return SDSAT_ECUDA;
  n = std::min(n, c->trace_cap);
  const unsigned int m = records ? std::min<unsigned int>(n, (unsigned)std::max(max_records, 0)) : 0;
  if (m && cudaMemcpy(records, c->trace_rec, (size_t)m * TRACE_WORDS * sizeof(uint64_t), cudaMemcpyDeviceToHost) != cudaSuccess)
    return SDSAT_ECUDA;
  if (n_records) *n_records = (int)m;
  cudaFree(c->trace_rec);
  cudaFree(c->trace_count);
  c->trace_rec = nullptr;
  c->trace_count = nullptr;
  return SDSAT_OK;
}

const char* sdsat_kernel_class_name(int cls) { return (cls >= 0 && cls < K_COUNT) ? KCLASS_NAME[cls] : "?"; }

sdsat_status sdsat_profile_begin(sdsat_ctx* c, int max_launches) {
  if (!c || max_launches < 1) return SDSAT_EINVAL;
  for (cudaEvent_t e : c->prof_events) cudaEventDestroy(e);
  c->prof_events.assign(2 * (size_t)max_launches, nullptr);
  for (auto& e : c->prof_events)
    if (cudaEventCreate(&e) != cudaSuccess) return SDSAT_ECUDA;
  c->prof_class.assign(max_launches, 0);
  c->prof_used = 0;
  c->prof = true;
  return SDSAT_OK;
}

sdsat_status sdsat_profile_end(sdsat_ctx* c, sdsat_kernel_stat* out, int max_out, int* n_out) {
  if (!c || !c->prof) return SDSAT_EINVAL;
  c->prof = false;
  if (cudaStreamSynchronize(c->stream) != cudaSuccess) return SDSAT_ECUDA;
  long long cnt[K_COUNT] = {0};
  double ms[K_COUNT] = {0};
  for (size_t i = 0; i < c->prof_used; ++i) {
    float t = 0.f;
    if (cudaEventElapsedTime(&t, c->prof_events[2 * i], c->prof_events[2 * i + 1]) != cudaSuccess) return SDSAT_ECUDA;
    cnt[c->prof_class[i]] += 1;
    ms[c->prof_class[i]] += t;
  }
  int n = 0;
  for (int k = 0; k < K_COUNT; ++k) {
    if (!cnt[k]) continue;
    if (out && n < max_out) {
      std::memset(&out[n], 0, sizeof(out[n]));
      std::strncpy(out[n].name, KCLASS_NAME[k], sizeof(out[n].name) - 1);
      out[n].launches = cnt[k];
      out[n].total_ms = ms[k];
    }
    ++n;
  }
  if (n_out) *n_out = n;
  for (cudaEvent_t e : c->prof_events) cudaEventDestroy(e);
  c->prof_events.clear();
  c->prof_used = 0;
  return SDSAT_OK;
}

sdsat_status sdsat_build_block(sdsat_ctx* c, sdsat_kv* kv, int mode, const int32_t* prev_out_dev,
                               const int32_t* prev_acc_dev, const int32_t* draft_table_dev, int table_stride,
                               int b, int q, int32_t* tokens_out_dev) {
  if (!c || !kv || kv->ctx != c || !prev_out_dev || !prev_acc_dev || !tokens_out_dev) return SDSAT_EINVAL;
  if ((mode != 1 && mode != 2) || b < 1 || b > kv->batch || q < 1 || q > SDSAT_MAX_Q) return SDSAT_EINVAL;
  if (mode == 1 && c->cfg.n_adaptive > 1 && q - 1 > c->cfg.n_adaptive) return SDSAT_EINVAL;
  if (draft_table_dev && table_stride < kv->cap + SDSAT_MAX_Q) return SDSAT_EINVAL;
  BuildParams bp{mode, prev_out_dev, q, prev_acc_dev, draft_table_dev, table_stride, kv->batch, kv->len,
                 c->adaptive, b, q, q - 1, tokens_out_dev};
  return timed(c, K_BUILD_BLOCK, [&] { return launch_build_block(bp, c->stream, c->pdl); }) == cudaSuccess
             ? SDSAT_OK
             : SDSAT_ECUDA;
}

sdsat_status sdsat_build_tree_block(sdsat_ctx* c, sdsat_kv* kv, int mode, const int32_t* prev_out_dev, int prev_q,
                                    const int32_t* prev_acc_dev, const int32_t* draft_tables_dev, int width,
                                    int table_stride, int b, int k, int32_t* tokens_out_dev) {
  if (!c || !kv || kv->ctx != c || !prev_out_dev || !prev_acc_dev || !tokens_out_dev) return SDSAT_EINVAL;
  if ((mode != 1 && mode != 2) || b < 1 || b > kv->batch || k < 1 || width < 1 || prev_q < 1 ||
      prev_q > SDSAT_MAX_Q)
    return SDSAT_EINVAL;
  const int q = mode == 1 ? k + 1 : 1 + width * k;
  if (q > SDSAT_MAX_Q || b * q > SDSAT_MAX_ROWS) return SDSAT_EINVAL;
  if (mode == 1 && c->cfg.n_adaptive > 1 && k > c->cfg.n_adaptive) return SDSAT_EINVAL;
  if (mode == 2 && !draft_tables_dev && (width > 1 || k >= prev_q)) return SDSAT_EINVAL;
  if (draft_tables_dev && table_stride < kv->cap + SDSAT_MAX_Q) return SDSAT_EINVAL;
  BuildParams bp{mode, prev_out_dev, prev_q, prev_acc_dev, draft_tables_dev, table_stride, kv->batch, kv->len,
                 c->adaptive, b, q, k, tokens_out_dev};
  return timed(c, K_BUILD_BLOCK, [&] { return launch_build_block(bp, c->stream, c->pdl); }) == cudaSuccess
             ? SDSAT_OK
             : SDSAT_ECUDA;
}

sdsat_status sdsat_build_pipelined_block(sdsat_ctx* c, sdsat_kv* kv, const int32_t* prev_out_dev,
                                         const int32_t* prev_acc_dev, int32_t* mode_dev, int32_t* n_verify_dev,
                                         const int32_t* draft_table_dev, int table_stride, int b, int k,
                                         int32_t* tokens_out_dev) {
  if (!c || !kv || kv->ctx != c || !prev_out_dev || !prev_acc_dev || !mode_dev || !n_verify_dev || !tokens_out_dev)
    return SDSAT_EINVAL;
  const int q = 2 * k + 1;
  if (b < 1 || b > kv->batch || k < 1 || q > SDSAT_MAX_Q || b * q > SDSAT_MAX_ROWS) return SDSAT_EINVAL;
  if (c->cfg.n_adaptive > 1 && k > c->cfg.n_adaptive) return SDSAT_EINVAL;
  if (draft_table_dev && table_stride < kv->cap + SDSAT_MAX_Q) return SDSAT_EINVAL;
  BuildParams bp{3, prev_out_dev, q, prev_acc_dev, draft_table_dev, table_stride, kv->batch, kv->len,
                 c->adaptive, b, q, k, tokens_out_dev, mode_dev, n_verify_dev};
  return timed(c, K_BUILD_BLOCK, [&] { return launch_build_block(bp, c->stream, c->pdl); }) == cudaSuccess
             ? SDSAT_OK
             : SDSAT_ECUDA;
}

sdsat_status sdsat_attention_grid(int pairs, const int32_t* max_clusters, int cs_cap, int num_sms,
                                  int* cs, int* nclusters) {
  if (pairs < 1 || !max_clusters || cs_cap < 1 || num_sms < 1 || !cs || !nclusters) return SDSAT_EINVAL;
  attention_grid(pairs, max_clusters, cs_cap, num_sms, cs, nclusters);
  return SDSAT_OK;
}

sdsat_status sdsat_debug_wait_timeout(sdsat_ctx* c) {
  if (!c) return SDSAT_EINVAL;
  return launch_wait_timeout(c->err, c->stream) == cudaSuccess ? SDSAT_OK : SDSAT_ECUDA;
}

sdsat_status sdsat_get_error(sdsat_ctx* c, uint32_t* flags) {
  if (!c) return SDSAT_EINVAL;
  uint32_t f = 0;
  if (cudaStreamSynchronize(c->stream) != cudaSuccess) return SDSAT_ECUDA;
  if (cudaMemcpy(&f, c->err, sizeof(f), cudaMemcpyDeviceToHost) != cudaSuccess) return SDSAT_ECUDA;
  if (cudaMemset(c->err, 0, sizeof(f)) != cudaSuccess) return SDSAT_ECUDA;
  if (flags) *flags = f;
  return f ? SDSAT_EDEVICE : SDSAT_OK;
}

sdsat_status sdsat_op_gemm(sdsat_ctx* c, const float* x_dev, int M, int K, const void* w_dev, int N, float* y_dev) {
  if (!c || !x_dev || !y_dev || !aligned16(w_dev) || !aligned16(x_dev)) return SDSAT_EINVAL;
  if (M < 1 || M > PF_ROWS || K < 8 || K % 8 || K > OP_MAX_K || N < 1 || (N + 127) / 128 > MAX_GEMM_TILES)
    return SDSAT_EINVAL;
  if (M > SDSAT_MAX_ROWS) {
    // the prefill GEMM (tiles of 128 weight rows x 128 positions)
    const int rows = (M + 127) / 128 * 128;   // <= PF_ROWS rows of the operand scratch
    PfGemmParams g;
    std::memset(&g, 0, sizeof(g));
    if (!make_wmap(&g.tmap[0], w_dev, N, K) || !make_xmap(&g.tmap_x[0], c->xop_hi, rows, K, 128) ||
        !make_xmap(&g.tmap_x[1], c->xop_lo, rows, K, 128))
      return SDSAT_ECUDA;
    g.map_mode = MAP_PLAIN;
    g.N = N;
    g.kc = (K + 63) / 64;
    g.n_wtiles = (N + 127) / 128;
    g.n_tblocks = rows / 128;
    g.M = M;
    g.epi = EPI_STORE;
    g.out = y_dev;
    g.out_ld = N;
    g.err = c->err;
    if (launch_split(x_dev, M, K, c->xop_hi, c->xop_lo, c->stream, c->pdl) != cudaSuccess) return SDSAT_ECUDA;
    return timed(c, K_GEMM_OP, [&] { return launch_prefill_gemm(g, c->num_sms, c->stream, c->pdl); }) == cudaSuccess
               ? SDSAT_OK
               : SDSAT_ECUDA;
  }
  GemmParams g = gemm_base(c, M, -1);
  CUtensorMap m;
  if (!make_wmap(&m, w_dev, N, K) || !make_xmap(&g.tmap_x[0], c->xop_hi, SDSAT_MAX_ROWS, K, 16 << mpad_index(M)) ||
      !make_xmap(&g.tmap_x[1], c->xop_lo, SDSAT_MAX_ROWS, K, 16 << mpad_index(M)))
    return SDSAT_ECUDA;
  set_plain(g, m, N, K);
  if (launch_split(x_dev, M, K, c->xop_hi, c->xop_lo, c->stream, c->pdl) != cudaSuccess) return SDSAT_ECUDA;
  g.epi = EPI_STORE;
  g.out = y_dev;
  g.out_ld = N;
  return timed(c, K_GEMM_OP, [&] { return launch_gemm(g, c->num_sms, c->stream, c->pdl); }) == cudaSuccess ? SDSAT_OK
                                                                                                  : SDSAT_ECUDA;
}

sdsat_status sdsat_op_attention(sdsat_ctx* c, const float* q_dev, const void* k_dev, const void* v_dev,
                                const int32_t* len_dev, int b, int q, int H, int hd, int cap, float* out_dev) {
  if (!c || !q_dev || !k_dev || !v_dev || !len_dev || !out_dev) return SDSAT_EINVAL;
  if (b < 1 || q < 1 || q > SDSAT_MAX_Q || b * q > SDSAT_MAX_ROWS || (hd != 64 && hd != 128) || H < 1 || cap < 1 ||
      cap > ATT_MAX_CAP)
    return SDSAT_EINVAL;
  AttnParams a;
  std::memset(&a, 0, sizeof(a));
  if (!aligned16(k_dev) || !aligned16(v_dev) || !aligned16(out_dev) || (long long)b * H * cap > 0x7FFFFFFFll)
    return SDSAT_EINVAL;
  if (!make_kvmap(&a.kmap, k_dev, (long long)b * H * cap, hd) || !make_kvmap(&a.vmap, v_dev, (long long)b * H * cap, hd))
    return SDSAT_ECUDA;
  a.row0 = 0;
  a.Q = q_dev;
  a.q_ld = H * hd;
  a.len = len_dev;
  a.seq0 = 0;
  a.nb = b;
  a.q = q;
  a.H = H;
  a.hd = hd;
  a.cap = cap;
  a.out = out_dev;
  a.out_ld = H * hd;
  if ((size_t)b * q * H * hd > (size_t)SDSAT_MAX_ROWS * c->cfg.n_heads * c->cfg.head_dim) return SDSAT_EINVAL;
  a.out_hi = c->x_hi[X_ATTN];
  a.out_lo = c->x_lo[X_ATTN];
  a.err = c->err;
  return timed(c, K_ATTENTION_OP, [&] { return launch_attention(a, c->num_sms, c->stream, c->pdl); }) == cudaSuccess
             ? SDSAT_OK
                                                                                                   : SDSAT_ECUDA;
}

sdsat_status sdsat_debug_workspace(sdsat_ctx* c, int which, int rows, float* dst_dev) {
  if (!c || !dst_dev || rows < 1 || rows > SDSAT_MAX_ROWS || which < 0 || which > 3) return SDSAT_EINVAL;
  const int R = c->cfg.n_heads * c->cfg.head_dim;
  const float* src[4] = {c->h, c->qbuf, c->attn, c->act};
  const int cols[4] = {c->cfg.d_model, R, R, c->cfg.ffn_dim};
  return cudaMemcpyAsync(dst_dev, src[which], (size_t)rows * cols[which] * sizeof(float), cudaMemcpyDeviceToDevice,
                         c->stream) == cudaSuccess
             ? SDSAT_OK
             : SDSAT_ECUDA;
}

sdsat_status sdsat_op_exp(sdsat_ctx* c, const float* in_dev, float* out_dev, int n) {
  if (!c || !in_dev || !out_dev || n < 0) return SDSAT_EINVAL;
  if (n == 0) return SDSAT_OK;
  return launch_exp(in_dev, out_dev, n, c->stream) == cudaSuccess ? SDSAT_OK : SDSAT_ECUDA;
}

}  // extern "C"
