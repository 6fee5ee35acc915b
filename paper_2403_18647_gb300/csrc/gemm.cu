// Skinny-M weight-streaming GEMM on the 5th-generation tensor cores.
//
// Every projection of the block forward (QKV, O, gate/up, down, LM head) is
// Y[M, N] = X[M, K] W[N, K]^T with M = b*q <= 64 rows and a weight matrix of
// 30-330 MB.  The weights are read once per step, so the kernel is bound by
// HBM bandwidth (decoding is memory-bandwidth bound, Sec. 1; the loop time is
// almost flat in k, Sec. 3.4.1).  Design:
//
//  * Persistent grid of P CTAs; the (128-row tile, 64-wide K chunk) work units
//    are split evenly in one flat range ("stream-K"), so every CTA streams the
//    same number of 16 KB weight chunks.  A tile cut between CTAs is reduced
//    by its last finisher (per-tile counter), summing the partials in CTA
//    order: deterministic, no spin-wait.
//  * Warp 0 streams weight chunks with TMA (128-byte swizzle, L2 evict-first)
//    into a ring of shared-memory stages; it needs nothing from the previous
//    kernel, so with programmatic dependent launch it starts prefetching while
//    the previous kernel drains.
//    The activation operand X arrives the same way, once the previous kernel
//    has finished: its producer (RMSNorm, attention merge, SwiGLU epilogue)
//    stored it as two bf16 matrices hi + lo with x ~= hi + lo to ~16 mantissa
//    bits, so the tensor-core product keeps fp32-like accuracy in X.
//  * Warp 1 (one thread) issues tcgen05.mma: D[128 x 2*MPAD] (fp32, TMEM) +=
//    Wtile[128 x 16] * [Xhi; Xlo]^T -- the hi and lo operands sit back to back
//    in shared memory, so one MMA with N = 2*MPAD covers both and the epilogue
//    adds column m and column MPAD + m.  Four K-steps per chunk.  Two TMEM
//    accumulators alternate so a tile's epilogue overlaps the next tile's MMAs.
//  * Warps 2-5 read the accumulator (tcgen05.ld) and run the fused epilogue:
//    plain store, residual add, RoPE + KV-cache append, or SiLU(gate) * up
//    (which also emits the next GEMM's hi/lo operand).
#include <algorithm>

#include "common.cuh"
#include "internal.h"

namespace sdsat {

// Pipeline depth and CTAs per SM (compile-time tuning).  Measured on GB300: one CTA
// per SM streams ~5 TB/s whatever its depth (3..10 stages), two CTAs per SM ~7 TB/s.
// For M <= 16 a CTA has 4 stages (~91 KB of shared memory), so exactly two fit on an
// SM.  With 3 stages (~71 KB) a third fits: the next kernel's CTAs then start early,
// but the scheduler also stacks three CTAs of one GEMM on some SMs and one on others,
// and the equal stream-K shares finish unevenly (7B step 3.80 ms vs 3.70 with 4).
#ifndef SDSAT_GEMM_STAGES16
#define SDSAT_GEMM_STAGES16 4
#endif
// Stream-K split points within the first SDSAT_GEMM_SNAP units of a tile move to the tile's
// start, for GEMMs with at least SDSAT_GEMM_SNAP_MIN_UNITS units per CTA.
#ifndef SDSAT_GEMM_SNAP
#define SDSAT_GEMM_SNAP 3
#endif
#ifndef SDSAT_GEMM_SNAP_MIN_UNITS
#define SDSAT_GEMM_SNAP_MIN_UNITS 24
#endif
// Minimum resident CTAs per SM the register allocation must allow (192 threads each).
#ifndef SDSAT_GEMM_MINB
#define SDSAT_GEMM_MINB 2
#endif
// Epilogue rows handled per group: a group's loads are all issued before its stores.
#ifndef SDSAT_GEMM_EPI_GROUP
#define SDSAT_GEMM_EPI_GROUP 16
#endif
constexpr int EG = SDSAT_GEMM_EPI_GROUP;

template <int MPAD>
struct GemmCfg {
  static constexpr int STAGES = MPAD <= 16 ? SDSAT_GEMM_STAGES16 : 3;   // M <= 32: two CTAs per SM
  static constexpr int W_BYTES = 128 * 128;      // 128 rows x 64 bf16
  static constexpr int X_BYTES = MPAD * 128;     // MPAD rows x 64 bf16 (hi or lo)
  static constexpr int STAGE_BYTES = W_BYTES + 2 * X_BYTES;
  static constexpr int STAGING = 128 * (MPAD + 1) + 128;   // [128][MPAD+1] exchange + [128/MPAD][MPAD] sums
  static constexpr int ACC_COLS = 2 * MPAD;     // hi and lo products side by side
  static constexpr int TMEM_COLS = 2 * ACC_COLS;  // two accumulators
  static constexpr int NBAR = 2 * STAGES + 6;
  static constexpr int CS = MPAD * 64;           // EPI_QKV: RoPE (cos, sin) of every row and frequency
  // residual rows loaded before the accumulator wait: every row up to 32 (MPAD 64 keeps
  // the register budget with groups of EG)
  static constexpr int EGR = MPAD <= 32 ? MPAD : EG;
  static constexpr size_t SMEM =
      1024 + (size_t)STAGES * STAGE_BYTES + STAGING * 4 + 2 * 64 * 4 + 64 * 8 + CS * 8 + NBAR * 8 + 128;
};

// First unit of CTA b's range.  The even split b*T/P moves back to the start of its tile
// when it falls within that tile's first `snap` units: CTA b-1 would otherwise end with a
// segment of a few units, whose epilogue waits behind the publication (or the reduction) of
// the CTA's first tile and so usually arrives last and reduces that tile late.  The units go
// to CTA b instead, at the start of its range.
// (32-bit arithmetic: the host keeps T * P below 2^31.)
__device__ __forceinline__ int unit_begin(int b, int T, int P, int kc, int snap) {
  int x = (int)((unsigned)b * (unsigned)T / (unsigned)P);
  if (b > 0 && b < P) {
    const int r = x % kc;
    if (r >= 1 && r <= snap) x -= r;
  }
  return x;
}

// The CTA whose range holds unit g.  Without snapping it is the largest b with b*T/P <= g;
// snapping moves split points back by at most snap < T/P units, so it is that b or b + 1.
__device__ __forceinline__ int cta_of_chunk(int g, int T, int P, int kc, int snap) {
  const int b = (int)(((unsigned)g * (unsigned)P + (unsigned)(P - 1)) / (unsigned)T);
  return (b + 1 < P && unit_begin(b + 1, T, P, kc, snap) <= g) ? b + 1 : b;
}

// (tensor map, first row) of half h (0: tile rows 0-63, 1: rows 64-127) of tile t
__device__ __forceinline__ void tile_half_src(int map_mode, int rows_per_map, int t, int h, int& map, int& row) {
  if (map_mode == MAP_GATEUP) {
    map = h;
    row = 64 * t;
  } else if (map_mode == MAP_QKV3) {
    const int g = 128 * t;
    map = g / rows_per_map;
    row = g % rows_per_map + 64 * h;
  } else {
    map = 0;
    row = 128 * t + 64 * h;
  }
}

__device__ __forceinline__ bool mbar_wait_drain(uint64_t* bar, uint32_t parity) {
  const uint64_t t0 = globaltimer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (globaltimer_ns() - t0 > WAIT_LIMIT_NS) return false;
  }
  return true;
}

template <int MPAD>
__device__ __forceinline__ void epilogue_final(const GemmParams& p, int tile, int r, float (&acc)[MPAD],
                                               float* staging, const float* sinv, const long long* s_rowbase,
                                               const float (&pre)[GemmCfg<MPAD>::EGR], float pre_gn,
                                               const float2* s_cs) {
  const int M = p.M;
  constexpr int GR = GemmCfg<MPAD>::EGR;
  if (p.ssq_in) {
#pragma unroll
    for (int m = 0; m < MPAD; ++m) acc[m] *= sinv[m];
  }
  if (p.epi == EPI_RESID && p.gain_next) {
    // Residual update h += y, the next RMSNorm's operand h * g and this tile's sums of
    // h^2.  The sums go through shared memory in two conflict-free passes (warp shuffles
    // measured ~0.15 us each here, serialised per row), and the global stores come last.
    const int n = 128 * tile + r;
    const bool valid = n < p.N;
#pragma unroll
    for (int m0 = 0; m0 < MPAD; m0 += GR) {
      float hv[GR];
#pragma unroll
      for (int u = 0; u < GR; ++u)
        hv[u] = m0 == 0 ? pre[u] : (m0 + u < M && valid) ? __ldcg(p.out + (size_t)(m0 + u) * p.out_ld + n) : 0.f;
#pragma unroll
      for (int u = 0; u < GR; ++u) {
        const int m = m0 + u;
        if (m >= M) break;
        acc[m] = valid ? hv[u] + acc[m] : 0.f;   // h after the update
        staging[r * (MPAD + 1) + m] = acc[m] * acc[m];
      }
    }
    named_bar_sync(1, 128);
    // pass 1: thread (part, m) sums lanes part*RPP .. part*RPP+RPP-1 of row m
    constexpr int PARTS = 128 / MPAD, RPP = 128 / PARTS;   // parts of the 128 lanes, lanes per part
    float* part_sum = staging + 128 * (MPAD + 1);          // [PARTS][MPAD], beyond the [128][MPAD+1] block
    {
      const int m = r % MPAD, part = r / MPAD;
      float sq = 0.f;
      if (m < M) {
#pragma unroll 8
        for (int i = 0; i < RPP; ++i) sq += staging[(part * RPP + i) * (MPAD + 1) + m];
      }
      part_sum[part * MPAD + m] = sq;
    }
    named_bar_sync(1, 128);
    float ssq = 0.f;   // pass 2: row r < M adds its parts
    if (r < M) {
#pragma unroll
      for (int part = 0; part < PARTS; ++part) ssq += part_sum[part * MPAD + r];
    }
    named_bar_sync(1, 128);
    if (r < M) p.ssq_out[r * p.ssq_ld + tile] = ssq;
    if (valid) {
#pragma unroll
      for (int m = 0; m < MPAD; ++m) {
        if (m >= M) break;
        const size_t o = (size_t)m * p.out_ld + n;
        p.out[o] = acc[m];
        const float x = acc[m] * pre_gn;
        const __nv_bfloat16 hi = __float2bfloat16_rn(x);
        p.xn_hi[o] = hi;
        p.xn_lo[o] = __float2bfloat16_rn(x - __bfloat162float(hi));
      }
    }
    return;
  }
  if (p.epi == EPI_STORE || p.epi == EPI_RESID) {
    const int n = 128 * tile + r;
    if (n < p.N) {
      if (p.epi == EPI_RESID) {
#pragma unroll
        for (int m0 = 0; m0 < MPAD; m0 += GR) {
          float hv[GR];
#pragma unroll
          for (int u = 0; u < GR; ++u)
            hv[u] = m0 == 0 ? pre[u] : (m0 + u < M) ? __ldcg(p.out + (size_t)(m0 + u) * p.out_ld + n) : 0.f;
#pragma unroll
          for (int u = 0; u < GR; ++u) acc[m0 + u] += hv[u];
        }
      }
#pragma unroll
      for (int m = 0; m < MPAD; ++m)
        if (m < M) p.out[(size_t)m * p.out_ld + n] = acc[m];
    }
    return;
  }
  // epilogues that combine two TMEM lanes of the tile: exchange through shared memory
#pragma unroll
  for (int m = 0; m < MPAD; ++m) staging[r * (MPAD + 1) + m] = acc[m];
  named_bar_sync(1, 128);
  // These epilogues run once per launch, on the tiles' reducers, so their instructions are
  // fetched cold: the row loops stay rolled (a few dozen instructions) and read the
  // accumulators back from the exchange area instead of unrolling over MPAD rows.
  const float* mine = staging + r * (MPAD + 1);
  if (p.epi == EPI_SWIGLU) {
    // 64 output columns per tile: column c pairs gate lane c with up lane c + 64; threads
    // c and c + 64 take its even and odd rows
    const int c = r & 63, j = 64 * tile + c;
    if (j < p.N) {
      const float* gate = staging + c * (MPAD + 1);
      const float* up = staging + (c + 64) * (MPAD + 1);
      // SiLU through the fast exponential and division (a few ulp, far inside the tolerances
      // of an fp32 operand): the row loop is one dependent chain on the reducers' critical path
#pragma unroll 1
      for (int m = r >> 6; m < M; m += 2) {
        const float g = gate[m];
        const float a = __fdividef(g, 1.0f + __expf(-g)) * up[m];
        p.out[(size_t)m * p.out_ld + j] = a;
        const __nv_bfloat16 hi = __float2bfloat16_rn(a);
        p.out_hi[(size_t)m * p.out_ld + j] = hi;
        p.out_lo[(size_t)m * p.out_ld + j] = __float2bfloat16_rn(a - __bfloat162float(hi));
      }
    }
  } else {  // EPI_QKV
    // This runs once per launch on the reducers' critical path, so no division: the
    // projection by comparison, head and dimension by shift and mask (hd is 64 or 128), and
    // each row's cache offset from the table the setup filled.
    const int R = p.rows_per_map;
    const int gf = 128 * tile + r;
    const int which = (gf >= R) + (gf >= 2 * R);
    const int f = gf - which * R;
    const int hd = p.hd, half = hd >> 1;
    const int head = f >> (__ffs(hd) - 1), i = f & (hd - 1);
    const int ih = i & (half - 1);
    const int partner = (i < half) ? r + half : r - half;
    const float* other = staging + partner * (MPAD + 1);
    const float sgn = (i < half) ? -1.f : 1.f;   // rotate-half RoPE: x cos -+ partner sin
    __nv_bfloat16* cache = ((which == 1) ? p.k_layer : p.v_layer) + ((long long)head * p.cap * hd + i);
    float* qout = p.out + f;
#pragma unroll 2   // two rows in flight (4 made the cold loop slower)
    for (int m = 0; m < M; ++m, qout += p.out_ld) {
      float val = mine[m];
      if (which < 2) {
        const float2 cs = s_cs[m * 64 + ih];
        val = val * cs.x + sgn * (other[m] * cs.y);
      }
      if (which == 0) {
        *qout = val;
      } else {
        const long long base = s_rowbase[m];   // the row's cache element (seq, head 0, slot, 0)
        if (base >= 0) {
          cache[base] = __float2bfloat16_rn(val);
        } else if (i == 0 && which == 1) {
          set_error(p.err, ERR_CAPACITY);
        }
      }
    }
  }
  named_bar_sync(1, 128);
}

template <int MPAD>
__global__ void __launch_bounds__(192, SDSAT_GEMM_MINB) gemm_kernel(const __grid_constant__ GemmParams p) {
  using C = GemmCfg<MPAD>;
  constexpr int S = C::STAGES;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* stages = smem;
  float* staging = reinterpret_cast<float*>(smem + (size_t)S * C::STAGE_BYTES);
  float* sinv = staging + C::STAGING;   // [64] RMSNorm row factors of the operand
  int* s_pos = reinterpret_cast<int*>(sinv + 64);    // [64] EPI_QKV: RoPE position of each row
  // [64] EPI_QKV: offset of each row's cache element (sequence, head 0, slot, dimension 0),
  // -1 past the capacity (8-byte aligned: the area before is a multiple of 8 bytes)
  long long* s_rowbase = reinterpret_cast<long long*>(s_pos + 64);
  float2* s_cs = reinterpret_cast<float2*>(s_rowbase + 64);   // [MPAD][64] EPI_QKV: RoPE factors
  uint64_t* bars = reinterpret_cast<uint64_t*>(s_cs + C::CS);
  uint64_t* full = bars;             // weights and activations of the stage landed (TMA)
  uint64_t* empty = bars + S;        // stage consumed by the tensor core
  uint64_t* acc_full = bars + 2 * S; // [2] accumulator ready
  uint64_t* acc_empty = acc_full + 2;// [2] accumulator drained
  uint64_t* drain = acc_empty + 2;
  uint64_t* red_bar = drain + 1;     // partials of the tile being reduced landed (bulk copies)
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(red_bar + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  int* s_last = reinterpret_cast<int*>(tmem_slot + 2);
  // trace marks: first MMA issued, last accumulator ready, last tile reduced; [3] = flags
  unsigned long long* s_mark = reinterpret_cast<unsigned long long*>(tmem_slot + 4);
  int* s_share = reinterpret_cast<int*>(s_mark + 4);   // [6] split-K bookkeeping (see the epilogue)

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int cta = blockIdx.x;
  const int T = p.n_tiles * p.kc;
  const unsigned long long t_entry = p.trace.rec ? globaltimer_ns() : 0;
  unsigned long long t_wait = 0;
  const long long g0 = unit_begin(cta, T, p.P, p.kc, p.snap), g1 = unit_begin(cta + 1, T, p.P, p.kc, p.snap);
  const int tile_first = (int)g0 / p.kc, tile_last = ((int)g1 - 1) / p.kc;

  if (threadIdx.x == 64) {   // the tensor maps into the TMA unit while the CTA sets up
    const int nmaps = p.map_mode == MAP_QKV3 ? 3 : (p.map_mode == MAP_GATEUP ? 2 : 1);
    for (int i = 0; i < nmaps; ++i) tma_prefetch_desc(&p.tmap[i]);
    tma_prefetch_desc(&p.tmap_x[0]);
    tma_prefetch_desc(&p.tmap_x[1]);
  }
  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], 4);
    }
    mbar_init(drain, 1);
    mbar_init(red_bar, 1);
    *abort_flag = 0;
    s_mark[0] = s_mark[1] = s_mark[2] = s_mark[3] = 0;
    fence_mbar_init();
  }
  if (warp == 1) tmem_alloc(tmem_slot, C::TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_trigger();

  if (warp == 0) {
    // ------------------------------------------------ weight + activation stream (TMA)
    if (lane == 0) {
      const uint64_t pol_w = l2_policy_evict_first();   // weights: read once per step
      const uint64_t pol_x = l2_policy_evict_last();    // activations: read by every CTA
      constexpr uint32_t TX = C::W_BYTES + 2 * C::X_BYTES;
      const long long n = g1 - g0;
      const int npre = (int)std::min<long long>(S, n);
      // This thread's per-unit work sits on the streaming path (a stage is refilled only after
      // it has issued the copies), so the next unit's (tile, chunk) and its tile's two box
      // sources are advanced incrementally: no division per unit.
      int w_tile = (int)(g0 / p.kc), w_kc = (int)(g0 % p.kc), x_kc = w_kc;
      int map0, row0, map1, row1;
      tile_half_src(p.map_mode, p.rows_per_map, w_tile, 0, map0, row0);
      tile_half_src(p.map_mode, p.rows_per_map, w_tile, 1, map1, row1);
      auto load_w = [&](int it) {   // units in order, one call each
        uint8_t* dst = stages + (size_t)(it % S) * C::STAGE_BYTES;
        tma_load_2d(dst, &p.tmap[map0], &full[it % S], w_kc * 64, row0, pol_w);
        tma_load_2d(dst + 8192, &p.tmap[map1], &full[it % S], w_kc * 64, row1, pol_w);
        if (++w_kc == p.kc) {
          w_kc = 0;
          ++w_tile;
          tile_half_src(p.map_mode, p.rows_per_map, w_tile, 0, map0, row0);
          tile_half_src(p.map_mode, p.rows_per_map, w_tile, 1, map1, row1);
        }
      };
      auto load_x = [&](int it) {   // units in order, one call each
        const int kc = x_kc;
        if (++x_kc == p.kc) x_kc = 0;
        uint8_t* dst = stages + (size_t)(it % S) * C::STAGE_BYTES + C::W_BYTES;
        tma_load_2d(dst, &p.tmap_x[0], &full[it % S], kc * 64, 0, pol_x);
        tma_load_2d(dst + C::X_BYTES, &p.tmap_x[1], &full[it % S], kc * 64, 0, pol_x);
      };
      // weights of the first stages do not depend on the previous kernel: issue them now
      for (int it = 0; it < npre; ++it) {
        mbar_arrive_expect_tx(&full[it], TX);
        load_w(it);
      }
      pdl_wait();   // the activations are the previous kernel's output
      if (p.trace.rec) t_wait = globaltimer_ns();
      for (int it = 0; it < npre; ++it) load_x(it);
      int it = npre;
      for (; it < n; ++it) {
        const int s = it % S;
        if (!mbar_wait_bounded(&empty[s], ((it / S) & 1) ^ 1, abort_flag, p.err)) break;
        mbar_arrive_expect_tx(&full[s], TX);
        load_w(it);
        load_x(it);
      }
      if (*abort_flag) {  // let every copy in flight land before the CTA exits
        for (int i = std::max(0, it - S); i < it; ++i) mbar_wait_drain(&full[i % S], (i / S) & 1);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------ tensor-core issue
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(128, 2 * MPAD);
      int it = 0, seg = 0, tile = tile_first - 1;
      long long g = g0;
      bool ok = true;
      while (ok && g < g1) {
        ++tile;   // segments are consecutive tiles
        const long long gend = std::min(g1, (long long)(tile + 1) * p.kc);
        const int buf = seg & 1;
        if (!mbar_wait_bounded(&acc_empty[buf], ((seg >> 1) & 1) ^ 1, abort_flag, p.err)) break;
        tc_fence_after();
        const uint32_t d = tmem + buf * C::ACC_COLS;
        const long long gstart = g;
        for (; g < gend; ++g, ++it) {
          const int s = it % S;
          const uint32_t ph = (it / S) & 1;
          if (!mbar_wait_bounded(&full[s], ph, abort_flag, p.err)) {
            ok = false;
            break;
          }
          tc_fence_after();
          if (it == 0 && p.trace.rec) s_mark[0] = globaltimer_ns();
          const uint32_t wa = smem_u32(stages + (size_t)s * C::STAGE_BYTES);
          const uint32_t xh = wa + C::W_BYTES;   // [Xhi; Xlo]: 2*MPAD rows of 128 B
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            umma_bf16(d, sdesc_sw128(wa + kk * 32), sdesc_sw128(xh + kk * 32), idesc, (g != gstart || kk > 0) ? 1u : 0u);
          umma_commit(&empty[s]);
        }
        if (!ok) break;
        umma_commit(&acc_full[buf]);
        ++seg;
      }
      if (*abort_flag) {  // wait for issued MMAs before shared memory goes away
        umma_commit(drain);
        mbar_wait_drain(drain, 0);
      }
    }
  } else {
    // ------------------------------------------------ epilogue (TMEM -> registers -> global)
    const int e = warp & 3;   // TMEM lane quarter this warp may access (warps 2-5 -> 2, 3, 0, 1)
    const int r = e * 32 + lane;
    pdl_wait();
    if (p.ssq_in) {   // RMSNorm factor of each operand row, summed in a fixed order
      const int n = p.M * p.ssq_n;            // <= MPAD * 64 <= the staging area
      for (int i = r; i < n; i += 128) staging[i] = __ldcg(p.ssq_in + (i / p.ssq_n) * p.ssq_ld + i % p.ssq_n);
      named_bar_sync(1, 128);
      if (r < p.M) {
        float ssum = 0.f;
        for (int t = 0; t < p.ssq_n; ++t) ssum += staging[r * p.ssq_n + t];
        sinv[r] = 1.0f / sqrtf(ssum / (float)p.norm_dim + p.norm_eps);
      }
      named_bar_sync(1, 128);
    }
    if (p.epi == EPI_QKV) {   // cache slot and RoPE position of every row (fixed during the forward)
      if (r < p.M) {
        const int seq = p.seq0 + r / p.q;
        const int slot = __ldcg(p.len + seq) + r % p.q;
        int pos = p.positions ? __ldcg(p.positions + r) : slot;
        if (pos < 0 || pos >= p.rope_len) {
          set_error(p.err, ERR_POSITION);
          pos = pos < 0 ? 0 : p.rope_len - 1;
        }
        s_pos[r] = pos;
        s_rowbase[r] = slot < p.cap ? ((long long)seq * p.H * p.cap + slot) * p.hd : -1;
      }
      named_bar_sync(1, 128);
      // the RoPE factors of every row, in shared memory long before any accumulator is ready
      const int half = max(p.hd >> 1, 1);
      for (int i = r; i < p.M * half; i += 128)
        s_cs[(i / half) * 64 + i % half] = p.rope[(size_t)s_pos[i / half] * half + i % half];
      named_bar_sync(1, 128);
    }
    // Split-K bookkeeping of the only tiles this CTA can share, its first and its last: their
    // contributors lo..hi, and the partial slot of lo (0 when lo's range starts at the tile's
    // start, else 1).  Every later contributor's range starts inside the tile, so its partial
    // sits in slot 0.  Worked out once, here, into shared memory (read after the accumulator
    // barrier): the reduction at the CTA's end is latency-bound and these divisions would sit
    // on its path, and six values live in registers through the epilogue cost more registers
    // than the next kernel's early CTAs can spare.
    if (r == 0) {
#pragma unroll
      for (int i = 0; i < 2; ++i) {
        const int t = i ? tile_last : tile_first;
        const int lo = cta_of_chunk(t * p.kc, T, p.P, p.kc, p.snap);
        s_share[3 * i] = lo;
        s_share[3 * i + 1] = cta_of_chunk(t * p.kc + p.kc - 1, T, p.P, p.kc, p.snap);
        s_share[3 * i + 2] = unit_begin(lo, T, p.P, p.kc, p.snap) == t * p.kc ? 0 : 1;
      }
    }
    // partials per bulk-copy round of the last reducer (the idle stage ring holds them)
    const int red_per = max(1, (int)((S * C::STAGE_BYTES) / ((uint32_t)p.M * 512)));
    int seg = 0, tile = tile_first - 1;
    long long g = g0;
    while (g < g1) {
      ++tile;   // segments are consecutive tiles
      g = std::min(g1, (long long)(tile + 1) * p.kc);
      const int buf = seg & 1;
      // what this tile's epilogue reads from global memory (first row group), loaded while
      // the tensor cores work: residual rows and gain
      float pre[C::EGR];
      float pre_gn = 0.f;
      {
        const int n = 128 * tile + r;
        const bool resid = p.epi == EPI_RESID && n < p.N;
#pragma unroll
        for (int u = 0; u < C::EGR; ++u) pre[u] = (resid && u < p.M) ? __ldcg(p.out + (size_t)u * p.out_ld + n) : 0.f;
        if (resid && p.gain_next) pre_gn = __bfloat162float(p.gain_next[n]);
      }
      // the four epilogue warps decide together (lanes leave the polling loop at different
      // times, and a wait can run out for some of them only)
      const bool got = named_bar_and(1, 128, mbar_wait_bounded(&acc_full[buf], (seg >> 1) & 1, abort_flag, p.err));
      if (!got) break;
      tc_fence_after();
      const bool last_seg = g >= g1;
      if (r == 0 && last_seg && p.trace.rec) s_mark[1] = globaltimer_ns();
      float acc[MPAD];
      {
        float hl[2 * MPAD];
#pragma unroll
        for (int c = 0; c < 2 * MPAD; c += 16)
          tmem_ld16(tmem + ((uint32_t)(e * 32) << 16) + buf * C::ACC_COLS + c, hl + c);
        tmem_wait_ld();
#pragma unroll
        for (int m = 0; m < MPAD; ++m) acc[m] = hl[m] + hl[MPAD + m];
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&acc_empty[buf]);
      ++seg;

      // contributors of this tile (a tile between the first and the last is the CTA's alone)
      const int sh = tile == tile_first ? 0 : 3;
      const bool edge = tile == tile_first || tile == tile_last;
      const int c_lo = edge ? s_share[sh] : cta, c_hi = edge ? s_share[sh + 1] : cta;
      const int lo_slot = s_share[sh + 2];
      if (c_hi > c_lo) {
        // this tile is shared: publish the partial, the last contributor reduces
        const int slot = (tile == tile_first) ? 0 : 1;
        float* mine = p.partials + (size_t)(cta * 2 + slot) * MPAD * 128;
#pragma unroll
        for (int m = 0; m < MPAD; ++m)
          if (m < p.M) mine[m * 128 + r] = acc[m];
        // publish: the CTA's stores, then one release/acquire counter update (thread r = 0)
        named_bar_sync(1, 128);
        if (r == 0) *s_last = (atomic_add_acq_rel_gpu(&p.counters[tile], 1) == c_hi - c_lo);
        named_bar_sync(1, 128);
        if (r == 0 && last_seg && p.trace.rec) s_mark[3] = (unsigned long long)(*s_last) | ((c_hi - c_lo + 1) << 8);
        if (!*s_last) {
          if (r == 0 && last_seg && p.trace.rec) s_mark[2] = globaltimer_ns();
          continue;
        }
#pragma unroll
        for (int m = 0; m < MPAD; ++m) acc[m] = 0.f;
        const uint32_t pbytes = (uint32_t)p.M * 512;   // rows m < M of a [MPAD][128] fp32 partial
        if (last_seg) {
          // The stage ring is idle after the CTA's last tile (every TMA load landed and every
          // MMA that read it completed): bulk-copy the contributors' partials into it, as many
          // per round as fit, and sum them in CTA order.
          const int per = red_per;
          const float* ring = reinterpret_cast<const float*>(stages);
          uint32_t ph = 0;
          bool ok = true;
          for (int j0 = c_lo; j0 <= c_hi && ok; j0 += per) {
            const int cnt = min(per, c_hi - j0 + 1);
            if (r == 0) mbar_arrive_expect_tx(red_bar, (uint32_t)cnt * pbytes);
            named_bar_sync(1, 128);   // the previous round's shared-memory reads are done; bytes announced
            if (r < cnt) {            // one copy per thread
              const int j = j0 + r;
              fence_proxy_async_global();
              bulk_load_g2s(stages + (size_t)r * pbytes,
                            p.partials + (size_t)(j * 2 + (j == c_lo ? lo_slot : 0)) * MPAD * 128, pbytes, red_bar);
            }
            ok = named_bar_and(1, 128, mbar_wait_bounded(red_bar, ph, abort_flag, p.err));
            ph ^= 1u;
            if (ok) {
              for (int u = 0; u < cnt; ++u) {
#pragma unroll
                for (int m = 0; m < MPAD; ++m)
                  if (m < p.M) acc[m] += ring[(size_t)u * p.M * 128 + m * 128 + r];
              }
            } else if (r == 0) {
              mbar_wait_drain(red_bar, ph ^ 1u);   // copies in flight land before the CTA exits
            }
          }
          if (!ok) break;
        } else {
          for (int j = c_lo; j <= c_hi; ++j) {
            const float* src = p.partials + (size_t)(j * 2 + (j == c_lo ? lo_slot : 0)) * MPAD * 128;
#pragma unroll
            for (int m = 0; m < MPAD; ++m)
              if (m < p.M) acc[m] += __ldcg(src + m * 128 + r);
          }
        }
        if (r == 0) p.counters[tile] = 0;
      }
      if (r == 0 && last_seg && p.trace.rec) s_mark[2] = globaltimer_ns();
      epilogue_final<MPAD>(p, tile, r, acc, staging, sinv, s_rowbase, pre, pre_gn, s_cs);
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
  if (threadIdx.x == 0 && p.trace.rec)
    trace_write(p.trace, (unsigned)s_mark[3], t_entry, t_wait, s_mark[0], s_mark[1], s_mark[2], globaltimer_ns());
}

int gemm_mpad(int M) { return M <= 16 ? 16 : (M <= 32 ? 32 : 64); }

size_t gemm_smem_bytes(int mpad) {
  return mpad == 16 ? GemmCfg<16>::SMEM : (mpad == 32 ? GemmCfg<32>::SMEM : GemmCfg<64>::SMEM);
}

cudaError_t gemm_prepare() {
  cudaError_t e = cudaFuncSetAttribute(gemm_kernel<16>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)GemmCfg<16>::SMEM);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(gemm_kernel<32>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)GemmCfg<32>::SMEM);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(gemm_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)GemmCfg<64>::SMEM);
}

static int gemm_grid(const GemmParams& p, int num_sms) {
  const long long T = (long long)p.n_tiles * p.kc;
  const int per_sm = gemm_mpad(p.M) <= 32 ? GEMM_CTAS_PER_SM : 1;
  return (int)std::min<long long>((long long)num_sms * per_sm, T);
}

cudaError_t launch_gemm(GemmParams& p, int num_sms, cudaStream_t st, bool pdl) {
  const int mpad = gemm_mpad(p.M);
  p.P = gemm_grid(p, num_sms);
  if ((long long)p.n_tiles * p.kc * p.P >= (1LL << 31)) return cudaErrorInvalidValue;   // 32-bit split math
  // Snapping costs the next CTA up to `snap` units, so it is used only where a CTA's share
  // is long; it needs snap < T/P (a range never empties and a unit's owner stays b or b+1).
  const long long per = (long long)p.n_tiles * p.kc / p.P;
  p.snap = per >= SDSAT_GEMM_SNAP_MIN_UNITS ? (int)std::min<long long>(SDSAT_GEMM_SNAP, per - 1) : 0;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.P);
  cfg.blockDim = dim3(192);
  cfg.dynamicSmemBytes = gemm_smem_bytes(mpad);
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  if (mpad == 16) return cudaLaunchKernelEx(&cfg, gemm_kernel<16>, p);
  if (mpad == 32) return cudaLaunchKernelEx(&cfg, gemm_kernel<32>, p);
  return cudaLaunchKernelEx(&cfg, gemm_kernel<64>, p);
}

}  // namespace sdsat
