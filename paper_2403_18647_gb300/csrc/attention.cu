// Block-causal attention of the q block rows against the KV cache (flash decoding).
//
// In one block forward, row j of sequence s attends to the committed slots
// [0, len[s]) and to block rows 0..j (slots len[s] .. len[s]+j), which the QKV
// epilogue has just written; this is how Eq. 1-2 evaluate every appended
// position of the block in one pass.  A tree block (Sec. 2.1.2) replaces the
// rows 0..j by row j's ancestors and itself, given as one bit mask per row.
// (Prefill attention, many query rows per sequence, is a separate kernel at the
// end of this file.)
// The bytes are the K and V rows (bf16, hd*2 bytes each), read once per
// (sequence, head) for all q rows together.
//
// Work: the grid is nclusters thread-block clusters of cs CTAs, all resident
// at once (launch_attention picks the largest cs <= ATT_CS_MAX for which one
// cluster per (sequence, head) pair fits on the GPU with room to spare; else
// cs = 1 and each CTA takes several pairs).  Three CTAs fit on an SM for q <= 8
// (two for q <= 16).  Cluster c takes the pairs c, c + nclusters, ...; the
// nu units of ATT_UNIT = 64 consecutive slots of a pair are split over the
// cluster's CTAs as [r*nu/cs, (r+1)*nu/cs) for CTA rank r.  One thread keeps a
// two-stage ring of K and V tiles (TMA, boxes of 64 dims x 64 rows, 128-byte
// swizzle) full, walking the CTA's units pair by pair; tiles made of committed
// slots only are requested before the QKV projection has finished, and the
// next ATT_PREFETCH tiles (one for long slices) are kept on their way into L2.  Per unit, on the
// tensor cores (mma.sync m16n8k16) in transposed form, so that the q <= 8
// block rows fill an N = 8 tile instead of padding an M = 16 one: S^T = K Q^T
// with each warp on 16 keys, an online-softmax update of the running row max
// and exp-sum (reductions over the warp's lanes, then the warps via shared
// memory), then O^T = O^T * alpha + V^T P^T with each warp on hd/4
// dimensions.  Q and P enter as bf16 hi + lo pairs (two MMAs each), K and V
// are the cache's own bf16 values, accumulation is fp32.
//
// Each CTA's run over its units of a pair ends in a partial result (row max,
// exp-sum, unnormalised output) that it leaves in its own shared memory; after
// a cluster barrier every CTA merges its share of the pair's output elements
// from the cs partials through distributed shared memory, in rank order with
// the usual log-sum-exp rescaling (deterministic), and writes them in fp32 and
// as the O projection's bf16 hi + lo operand.  A second cluster barrier keeps
// the partials in place until every CTA of the cluster has read them.
#include <algorithm>
#include <cstdlib>

#include "common.cuh"
#include "internal.h"

namespace sdsat {

constexpr int ATT_STAGES = 2;
constexpr int ATT_PREFETCH = 4;   // units past the ring requested into L2 ahead of their loads
// ... but only one for a CTA whose slice has at least this many units.  Thread 0 issues the
// window before the dependency wait, and the TMA unit works through the requests of the SM's
// three CTAs in order: with long slices (13B at context 4096: 7-8 units) thread 0 reached the
// wait 2.8 us after the QKV projection ended with a window of 4 (1.0 us with 1; 13B forward
// 5.303 -> 5.256 ms), while shorter slices (batch 4 at context 1024: 5-6 units) lose more from
// the later units' missed L2 hits than they gain (attention 13.7 -> 15.1 us with 1)
constexpr int ATT_LONG_SLICE = 7;
constexpr int ATT_SPARE_CLUSTERS = 8;   // room left for this many more clusters (measured: 7B/13B shapes, b = 1, 4)

template <int HD, int QT = 2>
struct AttCfg {
  static constexpr int ROWS = QT * 8;                    // query rows the tiles hold
  static constexpr int HALVES = HD / 64;                 // 64-dim column boxes per row
  static constexpr int HALF_BYTES = ATT_UNIT * 128;      // one box: 64 rows x 64 dims bf16
  static constexpr int TILE = HALF_BYTES * HALVES;       // K (or V) of one unit
  static constexpr int STAGE = 2 * TILE;                 // K then V
  static constexpr int QSTRIDE = HD * 2 + 16;            // bytes per row of the bf16 Q tiles (padded)
  static constexpr int PSTRIDE = ATT_UNIT * 2 + 16;      // bytes per row of the bf16 P tiles (padded)
  static constexpr int RED = 17;                         // floats per row of the row-reduction scratch
  // Q hi + lo tiles; once the CTA's units of a pair are done, its partial output [ROWS][HD] fp32
  static constexpr size_t OFF_Q = (size_t)ATT_STAGES * STAGE;
  // P hi + lo tiles
  static constexpr size_t OFF_P = OFF_Q + 2 * ROWS * QSTRIDE;
  static constexpr size_t OFF_RED = OFF_P + 2 * ROWS * PSTRIDE;   // [16][RED]: unit row max, sums; partial stats
  static constexpr size_t OFF_SEQ = OFF_RED + 16 * RED * 4;                         // len, units [64]
  static constexpr size_t OFF_ANC = OFF_SEQ + (64 + 64) * 4;                        // [16] visible block rows per row
  static constexpr size_t OFF_BAR = (OFF_ANC + 16 * 4 + 7) / 8 * 8;
  static constexpr size_t SMEM = 1024 + OFF_BAR + ATT_STAGES * 8 + 16;
  static_assert(ROWS * HD * 4 <= 2 * ROWS * QSTRIDE, "the partial output fits in the Q tiles");
};

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
// D (16x8 fp32) += A (16x16 bf16, row) * B (16x8 bf16, col)
__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                               uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}
__device__ __forceinline__ uint32_t pack_bf16(float lo_elem, float hi_elem) {
  return (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(lo_elem)) |
         ((uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(hi_elem)) << 16);
}

// QT: tiles of 8 query rows (1 for q <= 8, 2 for q <= 16)
template <int HD, int QT>
__global__ void __launch_bounds__(128, QT == 1 ? 3 : 1) attention_kernel(const __grid_constant__ AttnParams p) {
  using C = AttCfg<HD, QT>;
  constexpr int KSTEPS = HD / 16;          // MMA k-steps over the head dimension
  constexpr int MT = HD / 64;              // 16-dimension tiles per warp in V^T P^T
  constexpr int D4 = HD / 4;               // float4 columns of an output row
  constexpr int QI = QT * 8 * (HD / 2) / 128;   // (row, 2 dims) items of the q tiles per thread
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* Qh = smem + C::OFF_Q;                    // bf16 [ROWS][HD] (scaled q, hi part), padded rows
  uint8_t* Ql = Qh + C::ROWS * C::QSTRIDE;          // lo part
  float* po = reinterpret_cast<float*>(smem + C::OFF_Q);        // [ROWS][HD] partial output (after the units)
  uint8_t* Ph = smem + C::OFF_P;                    // bf16 [ROWS][ATT_UNIT] softmax numerators, hi part
  uint8_t* Pl = Ph + C::ROWS * C::PSTRIDE;
  float* red = reinterpret_cast<float*>(smem + C::OFF_RED);     // row-reduction scratch [4][16] max, [4][16] sums
  float* pml = red + 128;                                       // [ROWS][2] partial row max, exp-sum (after the units)
  int* len_seq = reinterpret_cast<int*>(smem + C::OFF_SEQ);     // [64] committed length of each sequence
  int* nu_seq = len_seq + 64;                                   // [64] units per head of each sequence
  uint32_t* anc_s = reinterpret_cast<uint32_t*>(smem + C::OFF_ANC);   // [16] block rows row j sees (bit i)
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + C::OFF_BAR);   // [ATT_STAGES] K and V of the stage landed
  volatile int* abort_flag = reinterpret_cast<volatile int*>(full + ATT_STAGES);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, tig = lane & 3;
  const int mi = lane >> 3, r8 = lane & 7;        // ldmatrix: this thread's matrix and row
  const int q = p.q, H = p.H;
  const int CS = p.cs, NC = p.nclusters;
  const int rank = (int)cluster_ctarank(), cl = (int)blockIdx.x / CS;
  const unsigned long long t_entry = p.trace.rec ? globaltimer_ns() : 0;
  pdl_trigger();
  if (tid == 64) {   // the tensor maps into the TMA unit while the lengths are read
    tma_prefetch_desc(&p.kmap);
    tma_prefetch_desc(&p.vmap);
  }

  // The committed lengths are final before this kernel can start: the block forward's
  // first kernel (RMSNorm) lets its dependents launch only after every earlier kernel
  // has completed.  Slots below them are not written during this forward either.
  if (tid < p.nb) {
    const int len = __ldcg(p.len + p.seq0 + tid);
    len_seq[tid] = len;
    nu_seq[tid] = (min(len + q, p.cap) + ATT_UNIT - 1) / ATT_UNIT;
  }
  if (tid == 0) {
    for (int s = 0; s < ATT_STAGES; ++s) mbar_init(&full[s], 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();
  const int npairs = p.nb * H;

  // this CTA's units [cb, ce) of pair pi (sequence pi / H, head pi % H)
  auto slice = [&](int pi, int& cb, int& ce) {
    const int nu = nu_seq[pi / H];
    cb = nu * rank / CS;
    ce = nu * (rank + 1) / CS;
  };
  // a position in the CTA's sequence of units: unit c of pair pi, its slice ending at ce
  struct Cursor {
    int pi, c, ce;
  };
  auto seek = [&](Cursor& u, int pi) {   // the first unit of the CTA's slices from pair pi on
    for (; pi < npairs; pi += NC) {
      int cb, ce;
      slice(pi, cb, ce);
      if (cb < ce) {
        u.pi = pi;
        u.c = cb;
        u.ce = ce;
        return;
      }
    }
    u.pi = npairs;
    u.c = u.ce = 0;
  };
  auto advance = [&](Cursor& u) {
    if (++u.c == u.ce) seek(u, u.pi + NC);
  };
  // first cache row of the cursor's unit, and whether all of its slots are committed
  auto unit_row = [&](const Cursor& u, bool& committed) {
    const int s = u.pi / H, hh = u.pi - s * H;
    committed = (u.c + 1) * ATT_UNIT <= len_seq[s];
    return p.row0 + ((p.seq0 + s) * H + hh) * p.cap + u.c * ATT_UNIT;
  };
  uint64_t pol = 0;
  auto issue = [&](int k, int row) {   // the CTA's unit k into stage k % ATT_STAGES
    uint8_t* st = smem + (size_t)(k % ATT_STAGES) * C::STAGE;
    uint64_t* bar = &full[k % ATT_STAGES];
    mbar_arrive_expect_tx(bar, C::STAGE);
#pragma unroll
    for (int hh = 0; hh < C::HALVES; ++hh) tma_load_2d(st + hh * C::HALF_BYTES, &p.kmap, bar, hh * 64, row, pol);
#pragma unroll
    for (int hh = 0; hh < C::HALVES; ++hh)
      tma_load_2d(st + C::TILE + hh * C::HALF_BYTES, &p.vmap, bar, hh * 64, row, pol);
  };
  auto prefetch = [&](int row) {   // a unit's K and V tiles into L2
#pragma unroll
    for (int hh = 0; hh < C::HALVES; ++hh) {
      tma_prefetch_l2_2d(&p.kmap, hh * 64, row);
      tma_prefetch_l2_2d(&p.vmap, hh * 64, row);
    }
  };
  // thread 0: units whose loads were issued, the next unit to load (isu) and the next
  // to prefetch into L2 (pfc, ATT_PREFETCH units past the ring)
  int issued = 0;
  Cursor isu{npairs, 0, 0}, pfc{npairs, 0, 0};
  if (tid == 0) {
    pol = l2_policy_evict_first();
    // Tiles of committed slots do not depend on the QKV projection: the first ones go
    // to the ring now, the next ATT_PREFETCH into L2 (and one more each time the ring is
    // refilled), so that the ring's loads are L2 hits instead of HBM round trips.
    seek(isu, cl);
    for (; issued < ATT_STAGES && isu.pi < npairs; ++issued) {
      bool committed;
      const int row = unit_row(isu, committed);
      if (!committed) break;
      issue(issued, row);
      advance(isu);
    }
    pfc = isu;
    for (int k = issued; k < ATT_STAGES && pfc.pi < npairs; ++k) advance(pfc);
    int cb0 = 0, ce0 = 0;
    if (cl < npairs) slice(cl, cb0, ce0);
    const int window = ce0 - cb0 >= ATT_LONG_SLICE ? 1 : ATT_PREFETCH;
    for (int k = 0; k < window && pfc.pi < npairs; ++k) {
      bool committed;
      const int row = unit_row(pfc, committed);
      if (committed) prefetch(row);
      advance(pfc);
    }
  }
  pdl_wait();   // q and this forward's new K/V rows come from the QKV projection
  const unsigned long long t_wait = p.trace.rec ? globaltimer_ns() : 0;
  if (tid == 0) {
    for (; issued < ATT_STAGES && isu.pi < npairs; ++issued) {
      bool committed;
      issue(issued, unit_row(isu, committed));
      advance(isu);
    }
  }
  unsigned long long t_k = 0, t_part = 0, t_merge = 0;
  unsigned pairs_done = 0;

  const float scale = rsqrtf((float)HD);
  const int kb = warp * 16;                       // first key (within the unit) of this warp's scores
  const int db = warp * (HD / 4);                 // first dimension of this warp's outputs
  // O^T of this warp's HD/4 dimensions (MT tiles of 16) x the query tiles, products with the
  // hi and with the lo part of P (summed when published); this thread holds query rows
  // t*8 + 2*tig + {0, 1} and keeps their running max and exp-sum in registers
  float O[MT][QT][4], Ol[MT][QT][4];
  float mr[QT][2], lr[QT][2];
  int k = 0;                                      // units of this CTA consumed (ring position)
  for (int pi = cl; pi < npairs; pi += NC) {
    const int sl = pi / H, h = pi - sl * H;
    int cb, ce;
    slice(pi, cb, ce);
#pragma unroll
    for (int t = 0; t < QT; ++t) mr[t][0] = mr[t][1] = -INFINITY, lr[t][0] = lr[t][1] = 0.f;
#pragma unroll
    for (int mt = 0; mt < MT; ++mt)
#pragma unroll
      for (int t = 0; t < QT; ++t)
#pragma unroll
        for (int e = 0; e < 4; ++e) O[mt][t][e] = Ol[mt][t][e] = 0.f;
    if (cb < ce) {
      // ---- the rows' visible block rows (causal: 0..j; tree: the ancestors and the row
      // itself), q (scaled by 1/sqrt(hd)) as bf16 hi + lo, rows >= q zero; every load first
      if (tid < 16) anc_s[tid] = (p.anc && tid < q) ? __ldcg(p.anc + sl * q + tid) : (2u << tid) - 1u;
      float2 qv[QI];
#pragma unroll
      for (int r = 0; r < QI; ++r) {
        const int i = tid + 128 * r, j = i / (HD / 2), d = (i % (HD / 2)) * 2;
        qv[r] = j < q ? __ldcg(reinterpret_cast<const float2*>(p.Q + (size_t)(sl * q + j) * p.q_ld + h * HD + d))
                      : make_float2(0.f, 0.f);
      }
#pragma unroll
      for (int r = 0; r < QI; ++r) {
        const int i = tid + 128 * r, j = i / (HD / 2), d = (i % (HD / 2)) * 2;
        const float x0 = qv[r].x * scale, x1 = qv[r].y * scale;
        const __nv_bfloat16 h0 = __float2bfloat16_rn(x0), h1 = __float2bfloat16_rn(x1);
        *reinterpret_cast<uint32_t*>(Qh + j * C::QSTRIDE + d * 2) =
            (uint32_t)__bfloat16_as_ushort(h0) | ((uint32_t)__bfloat16_as_ushort(h1) << 16);
        *reinterpret_cast<uint32_t*>(Ql + j * C::QSTRIDE + d * 2) =
            pack_bf16(x0 - __bfloat162float(h0), x1 - __bfloat162float(h1));
      }
      __syncthreads();
    }
    const int len = len_seq[sl];
    const int nkeys = min(len + q, p.cap);
    for (int c = cb; c < ce; ++c, ++k) {
      const int c0 = c * ATT_UNIT;                  // slot of the unit's first key
      const uint8_t* Kt = smem + (size_t)(k % ATT_STAGES) * C::STAGE;
      const uint8_t* Vt = Kt + C::TILE;
      // one decision per warp (mma.sync needs every lane; a wait can run out for some only)
      const bool ok = __all_sync(0xffffffffu, mbar_wait_bounded(&full[k % ATT_STAGES], (k / ATT_STAGES) & 1,
                                                              abort_flag, p.err));
      if (k == 0 && p.trace.rec) t_k = globaltimer_ns();

      // ---- S^T = K Q^T for this warp's 16 keys: m16n8k16 with A = K (16 keys x 16 dims) and
      // B = Q^T (16 dims x 8 query rows), so up to 8 block rows fill one N = 8 tile
      float St[QT][4], Sl[QT][4];   // products with the hi and the lo part of q
#pragma unroll
      for (int t = 0; t < QT; ++t)
#pragma unroll
        for (int e = 0; e < 4; ++e) St[t][e] = Sl[t][e] = 0.f;
      if (ok) {
#pragma unroll
        for (int kk = 0; kk < KSTEPS; ++kk) {
          const int hh = kk >> 2, cg = 2 * (kk & 3);  // 64-dim half and first 16-byte granule
          const int key = kb + r8 + 8 * (mi & 1), cc = cg + (mi >> 1);
          uint32_t a0, a1, a2, a3;
          ldsm_x4(smem_u32(Kt + hh * C::HALF_BYTES + key * 128 + ((cc ^ (key & 7)) << 4)), a0, a1, a2, a3);
#pragma unroll
          for (int t = 0; t < QT; ++t) {
            uint32_t bh0, bh1, bl0, bl1;   // q rows t*8 .. t*8+7: hi (matrices 0, 1), lo (2, 3)
            const uint8_t* qsrc = (mi >> 1) ? Ql : Qh;
            ldsm_x4(smem_u32(qsrc + (t * 8 + r8) * C::QSTRIDE + (kk * 16 + 8 * (mi & 1)) * 2), bh0, bh1, bl0, bl1);
            mma_bf16_16816(St[t], a0, a1, a2, a3, bh0, bh1);
            mma_bf16_16816(Sl[t], a0, a1, a2, a3, bl0, bl1);
          }
        }
#pragma unroll
        for (int t = 0; t < QT; ++t)
#pragma unroll
          for (int e = 0; e < 4; ++e) St[t][e] += Sl[t][e];
      }
      // St[t][e] is the score of key kb + g + 8*(e >> 1) for query row t*8 + 2*tig + (e & 1).
      // mask: row j sees key slot kp iff kp < len, or kp = len + i for a block row i that
      // anc_s[j] marks (and kp < nkeys, j < q)
      // (a unit of committed slots only is seen whole by every row; rows j >= q are never
      // merged, so their unmasked scores of zero do no harm)
      if (!ok || c0 + ATT_UNIT > len) {
#pragma unroll
        for (int t = 0; t < QT; ++t)
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const int j = t * 8 + 2 * tig + (e & 1);
            const int kp = c0 + kb + g + 8 * (e >> 1);
            if (!ok || j >= q || kp >= nkeys || (kp >= len && !((anc_s[j] >> (kp - len)) & 1u))) St[t][e] = -INFINITY;
          }
      }
      // ---- the unit's row maxima: over the warp's lanes holding other keys (g), then the four
      // warps through shared memory; the running statistics stay in registers
      float* redm = red;          // [4 warps][16 rows] unit row maxima
      float* redl = red + 64;     // [4 warps][16 rows] unit row exp-sums
      float mx[QT][2];
#pragma unroll
      for (int t = 0; t < QT; ++t) {
        mx[t][0] = fmaxf(St[t][0], St[t][2]);
        mx[t][1] = fmaxf(St[t][1], St[t][3]);
#pragma unroll
        for (int o = 4; o < 32; o <<= 1) {
          mx[t][0] = fmaxf(mx[t][0], __shfl_xor_sync(0xffffffffu, mx[t][0], o));
          mx[t][1] = fmaxf(mx[t][1], __shfl_xor_sync(0xffffffffu, mx[t][1], o));
        }
        if (g == 0) {
          redm[warp * 16 + t * 8 + 2 * tig] = mx[t][0];
          redm[warp * 16 + t * 8 + 2 * tig + 1] = mx[t][1];
        }
      }
      __syncthreads();   // every warp is also done with the previous unit (its stage, P, red)
      if (tid == 0 && k >= 1 && isu.pi < npairs && !*abort_flag) {
        // refill the previous unit's stage with unit k + 1, extend the L2 window
        bool committed;
        issue(issued, unit_row(isu, committed));
        advance(isu);
        ++issued;
        if (pfc.pi < npairs) {
          prefetch(unit_row(pfc, committed));
          advance(pfc);
        }
      }
      float al[QT][2];   // rescale of what the units before contributed
#pragma unroll
      for (int t = 0; t < QT; ++t)
#pragma unroll
        for (int i = 0; i < 2; ++i) {
          const int j = t * 8 + 2 * tig + i;
          const float mc = fmaxf(fmaxf(redm[j], redm[16 + j]), fmaxf(redm[32 + j], redm[48 + j]));
          const float mn = fmaxf(mr[t][i], mc);
          al[t][i] = (mn == -INFINITY) ? 1.f : __expf(mr[t][i] - mn);
          mr[t][i] = mn;
        }
      // ---- P^T = exp(S^T - m) as bf16 hi + lo, stored as P [query row][key], and its row sums
      float rs[QT][2];   // this thread's part of the unit row sums
#pragma unroll
      for (int t = 0; t < QT; ++t) {
        rs[t][0] = rs[t][1] = 0.f;
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int i = e & 1, j = t * 8 + 2 * tig + i, key = kb + g + 8 * (e >> 1);
          const float pv = (St[t][e] == -INFINITY) ? 0.f : __expf(St[t][e] - mr[t][i]);
          rs[t][i] += pv;
          const __nv_bfloat16 hi = __float2bfloat16_rn(pv);
          *reinterpret_cast<__nv_bfloat16*>(Ph + j * C::PSTRIDE + key * 2) = hi;
          *reinterpret_cast<__nv_bfloat16*>(Pl + j * C::PSTRIDE + key * 2) = __float2bfloat16_rn(pv - __bfloat162float(hi));
        }
#pragma unroll
        for (int o = 4; o < 32; o <<= 1) {
          rs[t][0] += __shfl_xor_sync(0xffffffffu, rs[t][0], o);
          rs[t][1] += __shfl_xor_sync(0xffffffffu, rs[t][1], o);
        }
        if (g == 0) {
          redl[warp * 16 + t * 8 + 2 * tig] = rs[t][0];
          redl[warp * 16 + t * 8 + 2 * tig + 1] = rs[t][1];
        }
      }
      __syncthreads();   // P tiles and the row sums are complete
#pragma unroll
      for (int t = 0; t < QT; ++t)
#pragma unroll
        for (int i = 0; i < 2; ++i) {
          const int j = t * 8 + 2 * tig + i;
          lr[t][i] = lr[t][i] * al[t][i] + ((redl[j] + redl[16 + j]) + (redl[32 + j] + redl[48 + j]));
        }
      // ---- O^T = O^T * alpha + V^T P^T: A = V^T (16 dims x 16 keys, transposed loads of the V
      // tile), B = P^T (16 keys x 8 query rows), for this warp's dimensions and every query tile
#pragma unroll
      for (int mt = 0; mt < MT; ++mt)
#pragma unroll
        for (int t = 0; t < QT; ++t)
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            O[mt][t][e] *= al[t][e & 1];
            Ol[mt][t][e] *= al[t][e & 1];
          }
      if (ok) {
#pragma unroll
        for (int kk = 0; kk < ATT_UNIT / 16; ++kk) {
          uint32_t va[MT][4];
#pragma unroll
          for (int mt = 0; mt < MT; ++mt) {
            const int key = kk * 16 + r8 + 8 * (mi >> 1);
            const int dim = db + 16 * mt + 8 * (mi & 1);
            const int hh = dim >> 6, cc = (dim & 63) >> 3;
            ldsm_x4_t(smem_u32(Vt + hh * C::HALF_BYTES + key * 128 + ((cc ^ (key & 7)) << 4)), va[mt][0], va[mt][1],
                      va[mt][2], va[mt][3]);
          }
#pragma unroll
          for (int t = 0; t < QT; ++t) {
            uint32_t ph0, ph1, pl0, pl1;   // P rows t*8 .. t*8+7, keys kk*16 ..: hi (0, 1), lo (2, 3)
            const uint8_t* psrc = (mi >> 1) ? Pl : Ph;
            ldsm_x4(smem_u32(psrc + (t * 8 + r8) * C::PSTRIDE + (kk * 16 + 8 * (mi & 1)) * 2), ph0, ph1, pl0, pl1);
#pragma unroll
            for (int mt = 0; mt < MT; ++mt) {
              mma_bf16_16816(O[mt][t], va[mt][0], va[mt][1], va[mt][2], va[mt][3], ph0, ph1);
              mma_bf16_16816(Ol[mt][t], va[mt][0], va[mt][1], va[mt][2], va[mt][3], pl0, pl1);
            }
          }
        }
      }
    }

    // ---- this CTA's partial for the pair into its own shared memory (the output over the
    // Q tiles, which no warp reads any more; the statistics beside the row-reduction
    // scratch): O^T[mt][t][e] is dimension db + 16*mt + g + 8*(e >> 1) of query row
    // t*8 + 2*tig + (e & 1); a CTA without units of the pair leaves (-inf, 0, 0)
#pragma unroll
    for (int mt = 0; mt < MT; ++mt)
#pragma unroll
      for (int t = 0; t < QT; ++t)
#pragma unroll
        for (int e = 0; e < 4; ++e)
          po[(t * 8 + 2 * tig + (e & 1)) * HD + db + 16 * mt + g + 8 * (e >> 1)] = O[mt][t][e] + Ol[mt][t][e];
    if (warp == 0 && g == 0) {
#pragma unroll
      for (int t = 0; t < QT; ++t)
#pragma unroll
        for (int i = 0; i < 2; ++i) {
          pml[(t * 8 + 2 * tig + i) * 2] = mr[t][i];
          pml[(t * 8 + 2 * tig + i) * 2 + 1] = lr[t][i];
        }
    }
    if (p.trace.rec) t_part = globaltimer_ns();
    cluster_sync_all();   // the cluster's cs partials of the pair are complete
    // ---- merge this CTA's share of the pair's (row, 4 dimensions) outputs over the cs
    // partials, read in rank order from the cluster's shared memory: w_r = exp(m_r - max m),
    // L = sum_r w_r l_r, O = (sum_r w_r o_r) / L.  The second cluster barrier only keeps the
    // partials in place until every CTA has read them, so each thread arrives at it right
    // after its last remote loads and waits only at the end: the barrier's round trip
    // overlaps the merge arithmetic and the output stores.
    bool arrived = false;
    {
      const int items = q * D4, i0 = items * rank / CS, i1 = items * (rank + 1) / CS;
      for (int it = i0 + tid; it < i1; it += 128) {
        const int j = it / D4, d4 = it - j * D4;
        const uint32_t a_ml = smem_u32(pml + 2 * j), a_o = smem_u32(po + j * HD + 4 * d4);
        float2 ml[ATT_CS_MAX];
        float4 ov[ATT_CS_MAX];
#pragma unroll
        for (int r = 0; r < ATT_CS_MAX; ++r)
          if (r < CS) {
            ml[r] = ld_dsmem_f2(mapa_shared(a_ml, r));
            ov[r] = ld_dsmem_f4(mapa_shared(a_o, r));
          }
        if (it + 128 >= i1) {   // this thread's last item: its reads of the partials are done
          cluster_arrive_thread();
          arrived = true;
        }
        float mx = -INFINITY;
#pragma unroll
        for (int r = 0; r < ATT_CS_MAX; ++r)
          if (r < CS) mx = fmaxf(mx, ml[r].x);
        float L = 0.f;
        float4 a = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int r = 0; r < ATT_CS_MAX; ++r)
          if (r < CS) {
            const float w = (ml[r].x == -INFINITY) ? 0.f : __expf(ml[r].x - mx);
            L += w * ml[r].y;
            a.x += w * ov[r].x;
            a.y += w * ov[r].y;
            a.z += w * ov[r].z;
            a.w += w * ov[r].w;
          }
        const float iv = 1.0f / L;
        const float4 o = make_float4(a.x * iv, a.y * iv, a.z * iv, a.w * iv);
        const size_t idx = (size_t)(sl * q + j) * p.out_ld + h * HD + 4 * d4;
        *reinterpret_cast<float4*>(p.out + idx) = o;
        const __nv_bfloat16 h0 = __float2bfloat16_rn(o.x), h1 = __float2bfloat16_rn(o.y);
        const __nv_bfloat16 h2 = __float2bfloat16_rn(o.z), h3 = __float2bfloat16_rn(o.w);
        uint2 hi, lo;
        hi.x = (uint32_t)__bfloat16_as_ushort(h0) | ((uint32_t)__bfloat16_as_ushort(h1) << 16);
        hi.y = (uint32_t)__bfloat16_as_ushort(h2) | ((uint32_t)__bfloat16_as_ushort(h3) << 16);
        lo.x = pack_bf16(o.x - __bfloat162float(h0), o.y - __bfloat162float(h1));
        lo.y = pack_bf16(o.z - __bfloat162float(h2), o.w - __bfloat162float(h3));
        *reinterpret_cast<uint2*>(p.out_hi + idx) = hi;
        *reinterpret_cast<uint2*>(p.out_lo + idx) = lo;
      }
    }
    if (p.trace.rec) t_merge = globaltimer_ns();
    ++pairs_done;
    if (!arrived) cluster_arrive_thread();   // a thread without an item to merge
    cluster_wait_thread();   // every CTA of the cluster has read this CTA's partial
  }
  if (*abort_flag && tid == 0) {   // let the copies in flight land before the CTA exits
    for (int i = max(0, issued - ATT_STAGES); i < issued; ++i) {
      const uint64_t t0 = globaltimer_ns();
      while (!mbar_try_wait(&full[i % ATT_STAGES], (i / ATT_STAGES) & 1))
        if (globaltimer_ns() - t0 > WAIT_LIMIT_NS) break;
    }
  }
  if (tid == 0 && p.trace.rec)
    trace_write(p.trace, pairs_done | ((unsigned)k << 8), t_entry, t_wait, t_k, t_part, t_merge, globaltimer_ns());
}

// ---- prefill attention ----------------------------------------------------------------
// Causal attention of a prefill chunk over the cache (flash attention, mma.sync m16n8k16).
// One CTA per (head, block of 64 chunk positions), heaviest blocks first; four warps of 16
// query rows each.  Units of 64 keys stream through a two-stage TMA ring (the decode
// kernel's tiles).  Per unit and warp: S = Q K^T (16 rows x 64 keys; Q as bf16 hi + lo, both
// products into one accumulator), the causal mask on the units that reach the block's
// positions, the online-softmax update (row max over the four lanes of a row), then
// O = O * alpha + P V with P taken straight from the S accumulators as the A operand (bf16
// hi + lo) and V through transposed ldmatrix loads.
template <int HD>
struct PfAttCfg {
  static constexpr int QS = HD * 2 + 16;                             // bytes per Q row (padded)
  static constexpr size_t OFF_Q = (size_t)ATT_STAGES * AttCfg<HD>::STAGE;
  static constexpr size_t OFF_BAR = OFF_Q + 2 * 64 * QS;
  static constexpr size_t SMEM = 1024 + OFF_BAR + ATT_STAGES * 8 + 16;
};

template <int HD>
__global__ void __launch_bounds__(128) prefill_attention_kernel(const __grid_constant__ PfAttnParams p) {
  using C = AttCfg<HD>;
  using F = PfAttCfg<HD>;
  constexpr int KSTEPS = HD / 16;   // k-steps of Q K^T over the head dimension
  constexpr int NT = HD / 8;        // 8-dimension tiles of O
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* Qh = smem + F::OFF_Q;          // bf16 [64][HD] scaled q, hi part (padded rows)
  uint8_t* Ql = Qh + 64 * F::QS;          // lo part
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + F::OFF_BAR);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(full + ATT_STAGES);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, tig = lane & 3;
  const int mi = lane >> 3, r8 = lane & 7;
  const int NQB = (p.M + 63) / 64;
  const int qb = NQB - 1 - (int)blockIdx.x / p.H, h = (int)blockIdx.x % p.H;
  const int q0 = qb * 64;
  if (tid == 0) {
    for (int s = 0; s < ATT_STAGES; ++s) mbar_init(&full[s], 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  pdl_wait();   // q and this chunk's K / V rows come from the kernels before
  pdl_trigger();
  const int len = __ldcg(p.len + p.seq);
  const int kend = len + min(q0 + 64, p.M);    // keys this block's positions may see
  const int nu = (kend + ATT_UNIT - 1) / ATT_UNIT;
  const int rowbase = p.row0 + (p.seq * p.H + h) * p.cap;
  __syncthreads();
  auto issue = [&](int u) {
    uint8_t* st = smem + (size_t)(u % ATT_STAGES) * C::STAGE;
    uint64_t* bar = &full[u % ATT_STAGES];
    mbar_arrive_expect_tx(bar, C::STAGE);
#pragma unroll
    for (int hh = 0; hh < C::HALVES; ++hh)
      tma_load_2d(st + hh * C::HALF_BYTES, &p.kmap, bar, hh * 64, rowbase + u * ATT_UNIT, l2_policy_evict_last());
#pragma unroll
    for (int hh = 0; hh < C::HALVES; ++hh)
      tma_load_2d(st + C::TILE + hh * C::HALF_BYTES, &p.vmap, bar, hh * 64, rowbase + u * ATT_UNIT,
                  l2_policy_evict_last());
  };
  if (tid == 0) {
    tma_prefetch_desc(&p.kmap);
    tma_prefetch_desc(&p.vmap);
    for (int u = 0; u < min(nu, ATT_STAGES); ++u) issue(u);
  }
  // the block's queries, scaled by 1/sqrt(hd), as bf16 hi + lo (positions >= M: zero)
  const float scale = rsqrtf((float)HD);
  for (int i = tid; i < 64 * (HD / 2); i += 128) {
    const int j = i / (HD / 2), d = (i % (HD / 2)) * 2;
    float x0 = 0.f, x1 = 0.f;
    if (q0 + j < p.M) {
      const float2 v = __ldcg(reinterpret_cast<const float2*>(p.Q + (size_t)(q0 + j) * p.q_ld + h * HD + d));
      x0 = v.x * scale;
      x1 = v.y * scale;
    }
    const __nv_bfloat16 h0 = __float2bfloat16_rn(x0), h1 = __float2bfloat16_rn(x1);
    *reinterpret_cast<uint32_t*>(Qh + j * F::QS + d * 2) =
        (uint32_t)__bfloat16_as_ushort(h0) | ((uint32_t)__bfloat16_as_ushort(h1) << 16);
    *reinterpret_cast<uint32_t*>(Ql + j * F::QS + d * 2) = pack_bf16(x0 - __bfloat162float(h0), x1 - __bfloat162float(h1));
  }
  __syncthreads();

  const int wr = warp * 16;                            // this warp's first row in the block
  const int pos0 = len + q0 + wr + g;                  // absolute position of row g (row g + 8: +8)
  float O[NT][4];
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) O[nt][0] = O[nt][1] = O[nt][2] = O[nt][3] = 0.f;
  float mrow[2] = {-INFINITY, -INFINITY}, lrow[2] = {0.f, 0.f};
  for (int u = 0; u < nu; ++u) {
    const uint8_t* Kt = smem + (size_t)(u % ATT_STAGES) * C::STAGE;
    const uint8_t* Vt = Kt + C::TILE;
    const bool ok = __all_sync(0xffffffffu, mbar_wait_bounded(&full[u % ATT_STAGES], (u / ATT_STAGES) & 1,
                                                            abort_flag, p.err));
    float s[8][4];
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.f;
    if (ok) {
#pragma unroll
      for (int ks = 0; ks < KSTEPS; ++ks) {
        uint32_t ah0, ah1, ah2, ah3, al0, al1, al2, al3;
        const int qrow = wr + r8 + 8 * (mi & 1), qcol = ks * 16 + 8 * (mi >> 1);
        ldsm_x4(smem_u32(Qh + qrow * F::QS + qcol * 2), ah0, ah1, ah2, ah3);
        ldsm_x4(smem_u32(Ql + qrow * F::QS + qcol * 2), al0, al1, al2, al3);
#pragma unroll
        for (int np = 0; np < 4; ++np) {
          const int key = np * 16 + r8 + 8 * (mi >> 1);
          const int c = ks * 2 + (mi & 1), hh = c >> 3, cc = c & 7;
          uint32_t b0, b1, b2, b3;
          ldsm_x4(smem_u32(Kt + hh * C::HALF_BYTES + key * 128 + ((cc ^ (key & 7)) << 4)), b0, b1, b2, b3);
          mma_bf16_16816(s[2 * np], ah0, ah1, ah2, ah3, b0, b1);
          mma_bf16_16816(s[2 * np], al0, al1, al2, al3, b0, b1);
          mma_bf16_16816(s[2 * np + 1], ah0, ah1, ah2, ah3, b2, b3);
          mma_bf16_16816(s[2 * np + 1], al0, al1, al2, al3, b2, b3);
        }
      }
    }
    // causal mask: key slot kp is visible to the row at position pos iff kp <= pos
    const int kbase = u * ATT_UNIT;
    const bool need_mask = !ok || kbase + ATT_UNIT - 1 > pos0 - g;   // some key passes the warp's first row
    if (need_mask) {
#pragma unroll
      for (int nt = 0; nt < 8; ++nt)
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int kp = kbase + nt * 8 + 2 * tig + (e & 1);
          if (!ok || kp > pos0 + 8 * (e >> 1)) s[nt][e] = -INFINITY;
        }
    }
    // online softmax: rows g (e = 0, 1) and g + 8 (e = 2, 3); the four lanes of a row share it
    float alpha[2];
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      float mx = -INFINITY;
#pragma unroll
      for (int nt = 0; nt < 8; ++nt) mx = fmaxf(mx, fmaxf(s[nt][2 * r], s[nt][2 * r + 1]));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
      const float mn = fmaxf(mrow[r], mx);
      alpha[r] = (mn == -INFINITY) ? 1.f : __expf(mrow[r] - mn);
      mrow[r] = mn;
    }
    float rs[2] = {0.f, 0.f};
#pragma unroll
    for (int nt = 0; nt < 8; ++nt)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float v = (s[nt][e] == -INFINITY) ? 0.f : __expf(s[nt][e] - mrow[e >> 1]);
        s[nt][e] = v;
        rs[e >> 1] += v;
      }
    lrow[0] = lrow[0] * alpha[0] + rs[0];
    lrow[1] = lrow[1] * alpha[1] + rs[1];
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
      O[nt][0] *= alpha[0];
      O[nt][1] *= alpha[0];
      O[nt][2] *= alpha[1];
      O[nt][3] *= alpha[1];
    }
    // O += P V, k-steps of 16 keys; P's A fragments are the S accumulators of two key tiles
    if (ok) {
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        uint32_t ph[4], pl[4];
        const float* s0 = s[2 * j];
        const float* s1 = s[2 * j + 1];
        const float pv[8] = {s0[0], s0[1], s0[2], s0[3], s1[0], s1[1], s1[2], s1[3]};
#pragma unroll
        for (int f = 0; f < 4; ++f) {
          const __nv_bfloat16 h0 = __float2bfloat16_rn(pv[2 * f]), h1 = __float2bfloat16_rn(pv[2 * f + 1]);
          ph[f] = (uint32_t)__bfloat16_as_ushort(h0) | ((uint32_t)__bfloat16_as_ushort(h1) << 16);
          pl[f] = pack_bf16(pv[2 * f] - __bfloat162float(h0), pv[2 * f + 1] - __bfloat162float(h1));
        }
        // A fragment order: (row g, keys 0-7), (row g+8, keys 0-7), (row g, keys 8-15), (row g+8, keys 8-15)
#pragma unroll
        for (int dp = 0; dp < NT / 2; ++dp) {
          const int key = j * 16 + r8 + 8 * (mi & 1);
          const int dim = dp * 16 + 8 * (mi >> 1);
          const int hh = dim >> 6, cc = (dim & 63) >> 3;
          uint32_t b0, b1, b2, b3;
          ldsm_x4_t(smem_u32(Vt + hh * C::HALF_BYTES + key * 128 + ((cc ^ (key & 7)) << 4)), b0, b1, b2, b3);
          mma_bf16_16816(O[2 * dp], ph[0], ph[1], ph[2], ph[3], b0, b1);
          mma_bf16_16816(O[2 * dp], pl[0], pl[1], pl[2], pl[3], b0, b1);
          mma_bf16_16816(O[2 * dp + 1], ph[0], ph[1], ph[2], ph[3], b2, b3);
          mma_bf16_16816(O[2 * dp + 1], pl[0], pl[1], pl[2], pl[3], b2, b3);
        }
      }
    }
    __syncthreads();   // every warp is done with the stage
    if (tid == 0 && u + ATT_STAGES < nu && !*abort_flag) issue(u + ATT_STAGES);
  }
  if (*abort_flag && tid == 0) {   // let the copies in flight land before the CTA exits
    for (int u = max(0, nu - ATT_STAGES); u < nu; ++u) {
      const uint64_t t0 = globaltimer_ns();
      while (!mbar_try_wait(&full[u % ATT_STAGES], (u / ATT_STAGES) & 1))
        if (globaltimer_ns() - t0 > WAIT_LIMIT_NS) break;
    }
  }
  // O / L for the rows of this block inside the chunk, fp32 and bf16 hi + lo
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    float l = lrow[r];
    l += __shfl_xor_sync(0xffffffffu, l, 1);
    l += __shfl_xor_sync(0xffffffffu, l, 2);
    const float inv = l > 0.f ? 1.0f / l : 0.f;
    const int row = q0 + wr + g + 8 * r;
    if (row >= p.M) continue;
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
      const float o0 = O[nt][2 * r] * inv, o1 = O[nt][2 * r + 1] * inv;
      const size_t idx = (size_t)row * p.out_ld + h * HD + nt * 8 + 2 * tig;
      *reinterpret_cast<float2*>(p.out + idx) = make_float2(o0, o1);
      const __nv_bfloat16 h0 = __float2bfloat16_rn(o0), h1 = __float2bfloat16_rn(o1);
      *reinterpret_cast<uint32_t*>(p.out_hi + idx) =
          (uint32_t)__bfloat16_as_ushort(h0) | ((uint32_t)__bfloat16_as_ushort(h1) << 16);
      *reinterpret_cast<uint32_t*>(p.out_lo + idx) = pack_bf16(o0 - __bfloat162float(h0), o1 - __bfloat162float(h1));
    }
  }
}

size_t attention_smem_bytes(int hd, int q) {
  if (hd == 64) return q <= 8 ? AttCfg<64, 1>::SMEM : AttCfg<64, 2>::SMEM;
  return q <= 8 ? AttCfg<128, 1>::SMEM : AttCfg<128, 2>::SMEM;
}

namespace {
// most clusters of cs CTAs resident at once, per decode kernel instance (hd 64 / 128,
// one or two query tiles) and cs = 1 .. ATT_CS_MAX; 0 = that cluster size cannot launch
int g_att_clusters[2][2][ATT_CS_MAX + 1];
bool g_att_clusters_known = false;
int g_att_cs_cap = ATT_CS_MAX;   // SDSAT_ATT_CLUSTER_MAX: the largest cluster size launch_attention may pick

template <int HD, int QT>
cudaError_t prepare_decode_kernel(int (&maxc)[ATT_CS_MAX + 1]) {
  cudaError_t e;
  if ((e = cudaFuncSetAttribute(attention_kernel<HD, QT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)AttCfg<HD, QT>::SMEM)) != cudaSuccess)
    return e;
  if ((e = cudaFuncSetAttribute(attention_kernel<HD, QT>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1)) !=
      cudaSuccess)
    return e;
  for (int cs = 1; cs <= ATT_CS_MAX; ++cs) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(cs * 64);
    cfg.blockDim = dim3(128);
    cfg.dynamicSmemBytes = AttCfg<HD, QT>::SMEM;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = cs;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, attention_kernel<HD, QT>, &cfg) != cudaSuccess) {
      (void)cudaGetLastError();   // this cluster size is not available: never chosen
      n = 0;
    }
    maxc[cs] = n;
  }
  return cudaSuccess;
}
}  // namespace

cudaError_t attention_prepare() {
  const cudaFuncAttribute a = cudaFuncAttributeMaxDynamicSharedMemorySize;
  cudaError_t e;
  if (!g_att_clusters_known) {
    const char* cap = std::getenv("SDSAT_ATT_CLUSTER_MAX");
    if (cap && cap[0]) g_att_cs_cap = std::max(1, std::min(ATT_CS_MAX, std::atoi(cap)));
    if ((e = prepare_decode_kernel<64, 1>(g_att_clusters[0][0])) != cudaSuccess) return e;
    if ((e = prepare_decode_kernel<64, 2>(g_att_clusters[0][1])) != cudaSuccess) return e;
    if ((e = prepare_decode_kernel<128, 1>(g_att_clusters[1][0])) != cudaSuccess) return e;
    if ((e = prepare_decode_kernel<128, 2>(g_att_clusters[1][1])) != cudaSuccess) return e;
    g_att_clusters_known = true;
  }
  if ((e = cudaFuncSetAttribute(prefill_attention_kernel<64>, a, (int)PfAttCfg<64>::SMEM)) != cudaSuccess) return e;
  return cudaFuncSetAttribute(prefill_attention_kernel<128>, a, (int)PfAttCfg<128>::SMEM);
}

void attention_grid(int pairs, const int* maxc, int cs_cap, int num_sms, int* cs, int* nclusters) {
  // One cluster per (sequence, head) pair, of the largest size cs that leaves room for
  // ATT_SPARE_CLUSTERS more clusters among the CTAs resident at once: clusters are placed
  // whole within one GPC, and grids that filled the GPU left some clusters waiting for
  // a second wave.  If not even pairs of CTAs fit, single CTAs (as many as are resident
  // at once) take several pairs each.
  const int resident = maxc[1] > 0 ? maxc[1] : 2 * num_sms;
  *cs = 1;
  for (int c = std::min(cs_cap, ATT_CS_MAX); c >= 2; --c)
    if (maxc[c] >= pairs && c * (pairs + ATT_SPARE_CLUSTERS) <= resident) {
      *cs = c;
      break;
    }
  *nclusters = *cs > 1 ? pairs : std::max(1, std::min(pairs, resident));
}

cudaError_t launch_attention(const AttnParams& p0, int num_sms, cudaStream_t st, bool pdl) {
  AttnParams p = p0;
  attention_grid(p.nb * p.H, g_att_clusters[p.hd == 128][p.q > 8], g_att_cs_cap, num_sms, &p.cs, &p.nclusters);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.nclusters * p.cs);
  cfg.blockDim = dim3(128);
  cfg.dynamicSmemBytes = attention_smem_bytes(p.hd, p.q);
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = p.cs;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 2 : 1;
  const bool one = p.q <= 8;
  if (p.hd == 64) return one ? cudaLaunchKernelEx(&cfg, attention_kernel<64, 1>, p) : cudaLaunchKernelEx(&cfg, attention_kernel<64, 2>, p);
  return one ? cudaLaunchKernelEx(&cfg, attention_kernel<128, 1>, p) : cudaLaunchKernelEx(&cfg, attention_kernel<128, 2>, p);
}

cudaError_t launch_prefill_attention(const PfAttnParams& p, cudaStream_t st, bool pdl) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(((p.M + 63) / 64) * p.H);
  cfg.blockDim = dim3(128);
  cfg.dynamicSmemBytes = p.hd == 64 ? PfAttCfg<64>::SMEM : PfAttCfg<128>::SMEM;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return p.hd == 64 ? cudaLaunchKernelEx(&cfg, prefill_attention_kernel<64>, p)
                    : cudaLaunchKernelEx(&cfg, prefill_attention_kernel<128>, p);
}

}  // namespace sdsat
