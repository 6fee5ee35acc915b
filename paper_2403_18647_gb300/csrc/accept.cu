// Target selection, verification and KV commit, plus the small kernels of the
// step (embedding gather, block-input building, explicit commit).
//
// Verification (Sec. 2.1.1, Eq. 3): with targets t_j (argmax or nucleus sample
// of block row j) and drafts d_i (the block's input token of row i), draft i is
// accepted while d_i == t_{i-1} for all i' <= i; the first mismatch stops the
// loop.  The emitted tokens are t_0 .. t_m and the committed KV length grows by
// 1 + m (the rejected rows, and in draft step 1 the adaptive-token rows, are
// rolled back by not being committed).
//
// One CTA per block row selects that row's target; the last CTA of a sequence
// (per-sequence counter, no waiting) runs the prefix scan and the commit.
//
// Tree blocks (Sec. 2.1.2): the rows are the nodes of a draft tree in
// topological order (parent[j] < j, row 0 the root).  Row j sits at position
// len + depth(j); a child is accepted when its parent is and its token equals
// the parent's target, and the deepest accepted node (lowest row among equally
// deep ones) ends the accepted path n_0 = 0, ..., n_m.  Its targets are
// emitted, and a compaction kernel moves the path's K and V rows to the slots
// len + 1 .. len + m before len advances by 1 + m.
#include "common.cuh"
#include "internal.h"

namespace sdsat {

// ---- the nucleus sampler's arithmetic -------------------------------------------
// exp(s) for s <= 0: Cody-Waite reduction with a two-part ln 2, degree-7 Taylor
// polynomial on |r| <= ln2/2 by Horner's rule, exact scaling by 2^n; every step
// is one correctly rounded fp32 operation (no contraction), so any IEEE
// implementation of the same steps gives the same bits.
__device__ __forceinline__ float exp_sd(float s) {
  if (!(s >= -87.0f)) return 0.0f;
  const float n = rintf(__fmul_rn(s, (float)1.4426950408889634));
  const float r = __fsub_rn(__fsub_rn(s, __fmul_rn(n, 0.693145751953125f)), __fmul_rn(n, (float)(0.6931471805599453 - 0.693145751953125)));
  float p = (float)(1.0 / 5040.0);        // 1/7!
  p = __fadd_rn(__fmul_rn(p, r), (float)(1.0 / 720.0));  // 1/6!
  p = __fadd_rn(__fmul_rn(p, r), (float)(1.0 / 120.0));  // 1/5!
  p = __fadd_rn(__fmul_rn(p, r), (float)(1.0 / 24.0));  // 1/4!
  p = __fadd_rn(__fmul_rn(p, r), (float)(1.0 / 6.0));  // 1/3!
  p = __fadd_rn(__fmul_rn(p, r), 0.5f);
  p = __fadd_rn(__fmul_rn(p, r), 1.0f);
  p = __fadd_rn(__fmul_rn(p, r), 1.0f);
  const float scale = __int_as_float(((int)n + 127) << 23);
  return __fmul_rn(p, scale);
}

// floor(w * 2^24) for 0 <= w <= 1, exactly, from the fp32 bits
__device__ __forceinline__ uint32_t fixed24(float w) {
  const uint32_t b = __float_as_uint(w);
  if (b == 0) return 0;
  const int sh = (int)((b >> 23) & 0xFF) - 127 + 1;   // W = mant * 2^(e - 23 + 24)
  const uint32_t mant = (b & 0x7FFFFFu) | 0x800000u;
  if (sh >= 0) return mant << sh;
  return sh <= -24 ? 0u : (mant >> (-sh));
}

// Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11)
__device__ __forceinline__ void philox4x32_10(uint32_t c[4], uint32_t k0, uint32_t k1) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    const uint32_t lo0 = 0xD2511F53u * c[0], hi0 = __umulhi(0xD2511F53u, c[0]);
    const uint32_t lo1 = 0xCD9E8D57u * c[2], hi1 = __umulhi(0xCD9E8D57u, c[2]);
    const uint32_t n0 = hi1 ^ c[1] ^ k0, n2 = hi0 ^ c[3] ^ k1;
    c[0] = n0;
    c[1] = lo1;
    c[2] = n2;
    c[3] = lo0;
    k0 += 0x9E3779B9u;
    k1 += 0xBB67AE85u;
  }
}

// ---- block-wide reductions (1024 threads) -----------------------------------------
constexpr int ACC_THREADS = 1024;
constexpr int ACC_EPT = 32;   // logits per thread in the nucleus kernel (vocab <= 32768)

__device__ __forceinline__ uint64_t block_sum_u64(uint64_t v, uint64_t* red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  __syncthreads();
  if (l == 0) red[w] = v;
  __syncthreads();
  uint64_t t = (l < (int)(blockDim.x >> 5)) ? red[l] : 0;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
  return t;
}

__device__ __forceinline__ float block_max_f(float v, float* red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  __syncthreads();
  if (l == 0) red[w] = v;
  __syncthreads();
  float t = (l < (int)(blockDim.x >> 5)) ? red[l] : -INFINITY;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) t = fmaxf(t, __shfl_xor_sync(0xffffffffu, t, o));
  return t;
}

// exclusive prefix sum over threads (in thread order) of v; returns this thread's offset
__device__ __forceinline__ uint64_t block_exscan_u64(uint64_t v, uint64_t* red) {
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  uint64_t x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint64_t y = __shfl_up_sync(0xffffffffu, x, o);
    if (l >= o) x += y;
  }
  __syncthreads();
  if (l == 31) red[w] = x;
  __syncthreads();
  if (w == 0) {
    uint64_t t = (l < (int)(blockDim.x >> 5)) ? red[l] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint64_t y = __shfl_up_sync(0xffffffffu, t, o);
      if (l >= o) t += y;
    }
    red[l] = t;   // inclusive prefix of warp sums
  }
  __syncthreads();
  return (w > 0 ? red[w - 1] : 0) + x - v;
}

// ---- greedy: argmax with the lowest id on ties, NaN as -inf ----------------------------
__device__ int row_argmax(const float* row, int V, uint32_t* err, float* redf, int* redi) {
  float best = -INFINITY;
  int bi = 0x7FFFFFFF;
  bool nan = false;
  auto take = [&](float x, int i) {
    if (x != x) {
      nan = true;
      x = -INFINITY;
    }
    if (x > best || (x == best && i < bi)) {
      best = x;
      bi = i;
    }
  };
  // float4 loads, a round of RN per thread issued before any is compared (the row is one
  // L2 round trip per round, not one per element); a thread visits its ids in increasing order
  constexpr int RN = 8;
  const bool vec = (reinterpret_cast<uintptr_t>(row) & 15u) == 0;
  const int V4 = vec ? V / 4 : 0;
  for (int i0 = 0; i0 < V4; i0 += RN * (int)blockDim.x) {
    float4 v[RN];
#pragma unroll
    for (int u = 0; u < RN; ++u) {
      const int i = i0 + u * (int)blockDim.x + threadIdx.x;
      if (i < V4) v[u] = __ldcg(reinterpret_cast<const float4*>(row) + i);
    }
#pragma unroll
    for (int u = 0; u < RN; ++u) {
      const int i = i0 + u * (int)blockDim.x + threadIdx.x;
      if (i < V4) {
        take(v[u].x, 4 * i);
        take(v[u].y, 4 * i + 1);
        take(v[u].z, 4 * i + 2);
        take(v[u].w, 4 * i + 3);
      }
    }
  }
  for (int i = 4 * V4 + threadIdx.x; i < V; i += blockDim.x) take(__ldcg(row + i), i);
  if (nan) set_error(err, ERR_NAN_LOGITS);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float ob = __shfl_xor_sync(0xffffffffu, best, o);
    const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
    if (ob > best || (ob == best && oi < bi)) {
      best = ob;
      bi = oi;
    }
  }
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  __syncthreads();
  if (l == 0) {
    redf[w] = best;
    redi[w] = bi;
  }
  __syncthreads();
  if (w == 0) {
    const int nw = blockDim.x >> 5;
    best = l < nw ? redf[l] : -INFINITY;
    bi = l < nw ? redi[l] : 0x7FFFFFFF;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float ob = __shfl_xor_sync(0xffffffffu, best, o);
      const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
      if (ob > best || (ob == best && oi < bi)) {
        best = ob;
        bi = oi;
      }
    }
    if (l == 0) redi[0] = (bi == 0x7FFFFFFF) ? 0 : bi;
  }
  __syncthreads();
  return redi[0];
}

// ---- nucleus: the fixed-point top-k / top-p sampler ------------------------------------
// Thread t owns ids [32t, 32t+32) (ascending id order is thread order, then
// slot) and keeps their weights W (uint32, <= 2^24) in registers.  Selections
// are predicates on (W, id); per-thread sums fit 32 bits, block sums 64.
struct Cut {
  uint32_t xk;  // top-k: candidates are W > xk, or W == xk and id <= idk
  int idk;
  uint32_t xp;  // top-p: kept candidates are W > xp, or W == xp and id <= idp
  int idp;
};
enum Pred : int {
  P_GE = 1,         // W >= x
  P_GT = 2,         // W > x
  P_EQ = 3,         // W == x
  P_CAND = 4,       // candidate
  P_CAND_GE = 5,    // candidate and W >= x
  P_CAND_GT = 6,    // candidate and W > x
  P_CAND_EQ = 7,    // candidate and W == x
  P_KEPT = 8,       // kept
};

template <int P>
__device__ __forceinline__ bool pred(uint32_t W, int id, const Cut& c, uint32_t x) {
  const bool cand = W > c.xk || (W == c.xk && id <= c.idk);
  switch (P) {
    case P_GE: return W >= x;
    case P_GT: return W > x;
    case P_EQ: return W == x;
    case P_CAND: return cand;
    case P_CAND_GE: return cand && W >= x;
    case P_CAND_GT: return cand && W > x;
    case P_CAND_EQ: return cand && W == x;
    default: return cand && (W > c.xp || (W == c.xp && id <= c.idp));
  }
}

// per-thread sum of W (COUNT: number of ids) over the owned ids selected by P
template <int P, bool COUNT>
__device__ __forceinline__ uint32_t lsum(const uint32_t (&W)[ACC_EPT], int base, const Cut& c, uint32_t x) {
  uint32_t s = 0;
#pragma unroll
  for (int e = 0; e < ACC_EPT; ++e)
    if (pred<P>(W[e], base + e, c, x)) s += COUNT ? 1u : W[e];
  return s;
}

// largest x in [0, 2^24] whose block total of lsum<P, COUNT>(x) is >= need (monotone in x)
template <int P, bool COUNT>
__device__ __forceinline__ uint32_t search_threshold(const uint32_t (&W)[ACC_EPT], int base, const Cut& c,
                                                     uint64_t need, uint64_t* red) {
  uint32_t lo = 0, hi = 1u << 24;
  while (lo < hi) {
    const uint32_t mid = lo + (hi - lo + 1) / 2;
    if (block_sum_u64(lsum<P, COUNT>(W, base, c, mid), red) >= need) lo = mid;
    else hi = mid - 1;
  }
  return lo;
}

// the n-th (n >= 1) smallest id selected by P, or INT_MAX if there are fewer
template <int P>
__device__ __forceinline__ int nth_id(const uint32_t (&W)[ACC_EPT], int base, const Cut& c, uint32_t x,
                                      uint64_t n, uint64_t* red, int* redi) {
  const uint64_t mine = lsum<P, true>(W, base, c, x);
  const uint64_t before = block_exscan_u64(mine, red);
  if (threadIdx.x == 0) redi[0] = 0x7FFFFFFF;
  __syncthreads();
  if (before < n && before + mine >= n) {
    uint64_t k = before;
    int hit = 0x7FFFFFFF;
#pragma unroll
    for (int e = 0; e < ACC_EPT; ++e)
      if (pred<P>(W[e], base + e, c, x) && ++k == n) hit = base + e;
    redi[0] = hit;
  }
  __syncthreads();
  const int out = redi[0];
  __syncthreads();
  return out;
}

// ---- the sampler on a compacted list ----------------------------------------------------
// The kept set is a prefix of the order (W desc, id asc), so it lies among the heaviest
// weights.  With a floor F such that the elements with W >= F provably contain it (top-k:
// at least k of them, or all non-zero weights; top-p alone: their mass reaches the top-p
// threshold), those elements are copied in ascending id order into shared memory and one
// warp runs the same selection on them: searches cost O(list / 32) per step and no block
// barrier.  Otherwise the block-wide searches over all ids run.
constexpr int NUC_LIST_MAX = 4096;
constexpr int NUC_FLOORS = 7;
// floor f: 2^24 (the largest weight), 2^22, 2^20, 2^18, 2^16 (ratio 2^-8), 2^8 (2^-16), then 1
// (every non-zero weight).  Weights of bucket b (nuc_bucket) are >= the floors f >= b.
__device__ __forceinline__ uint32_t nuc_floor(int f) { return f < 5 ? 1u << (24 - 2 * f) : (f == 5 ? 256u : 1u); }
__device__ __forceinline__ int nuc_bucket(uint32_t w) {
  if (w == 0) return NUC_FLOORS;
  const int e = 31 - __clz(w);
  return e >= 16 ? (25 - e) >> 1 : (e >= 8 ? 5 : 6);
}

struct NucList {
  uint32_t w[NUC_LIST_MAX];
  int id[NUC_LIST_MAX];
  uint32_t cnt[NUC_FLOORS];                 // block totals: weights >= floor f
  unsigned long long mhi[3], mlo[3];        // masses >= floors 4, 5, 6: sum(w >> 12), sum(w & 4095)
  unsigned long long kstar, sk;             // the kept prefix's last key and its mass
  int pick;
};

__device__ __forceinline__ uint64_t nuc_key(uint32_t w, int id) {   // larger: heavier, then lower id
  return ((uint64_t)w << 32) | (uint32_t)(0x7FFFFFFF - id);
}

// Steps 4-7 on the list (warp 0) when the candidates (top-k, k <= 32) or, without top-k, the
// kept prefix have at most 32 elements: up to 32 rounds of "largest key below the previous
// one" put them on the lanes in (W desc, id asc) order.  Returns -1 when this does not apply.
__device__ int list_small(const AcceptParams& p, const NucList& L, int n, uint64_t S_all, bool topk, uint64_t rnd) {
  const int lane = threadIdx.x & 31;
  if (topk && p.top_k > 32) return -1;
  uint64_t thr = 0;
  if (!topk) {
    const uint64_t prod = (uint64_t)p.p_fixed * S_all;
    thr = (prod >> 24) + ((prod & 0xFFFFFFull) ? 1 : 0);
  }
  const int rounds = topk ? min(p.top_k, n) : min(32, n);
  uint64_t prev = ~0ull, mine = 0, C = 0;
  int nc = 0;
  bool done = topk;
  for (int r = 0; r < rounds && !(nc > 0 && !topk && C >= thr); ++r) {
    uint64_t best = 0;
    for (int i = lane; i < n; i += 32) {
      const uint64_t k = nuc_key(L.w[i], L.id[i]);
      if (k < prev && k > best) best = k;
    }
    const uint32_t hi = __reduce_max_sync(0xffffffffu, (uint32_t)(best >> 32));
    const uint32_t lo = __reduce_max_sync(0xffffffffu, (uint32_t)(best >> 32) == hi ? (uint32_t)best : 0u);
    prev = ((uint64_t)hi << 32) | lo;
    if (lane == r) mine = prev;
    ++nc;
    C += hi;   // the round's weight
  }
  if (!topk) done = C >= thr;   // the kept prefix: the first nc elements reach the threshold
  if (!done) return -1;
  const uint32_t w = lane < nc ? (uint32_t)(mine >> 32) : 0u;
  const int id = 0x7FFFFFFF - (int)(uint32_t)mine;
  bool kept = lane < nc;
  if (topk) {
    // candidates = the nc lanes; kept = the shortest prefix whose mass reaches thr
    const uint64_t S = __reduce_add_sync(0xffffffffu, w);
    const uint64_t prod = (uint64_t)p.p_fixed * S;
    const uint64_t t = (prod >> 24) + ((prod & 0xFFFFFFull) ? 1 : 0);
    uint32_t incl = w;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t y = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += y;
    }
    kept = kept && (lane == 0 || (uint64_t)(incl - w) < t);
  }
  const uint32_t kw = kept ? w : 0u;
  const uint64_t Sk = __reduce_add_sync(0xffffffffu, kw);
  const uint64_t tau = __umul64hi(rnd, Sk);
  // ascending-id cumulative weight of the kept elements up to and including this lane's
  uint64_t cum = 0;
  for (int j = 0; j < nc; ++j) {
    const uint32_t wj = __shfl_sync(0xffffffffu, kw, j);
    const int idj = __shfl_sync(0xffffffffu, id, j);
    if (idj <= id) cum += wj;
  }
  const uint32_t m = __ballot_sync(0xffffffffu, kept && cum > tau && cum - kw <= tau);
  return __shfl_sync(0xffffffffu, id, __ffs(m) - 1);
}

// Steps 4-7 on the list with the whole block.  The list holds the first n elements of the
// order (W desc, id asc) in ascending id; its keys are sorted once (bitonic, descending, over
// the list's own storage), so the candidates (the first min(k, n)), their mass, the kept
// prefix (the shortest one whose mass reaches ceil(P S / 2^24)) and its mass are prefix sums
// of the sorted weights.  The pick then scans every id's weight, still in registers, in
// ascending id with "kept" = key >= the kept prefix's last key.
__device__ int list_sorted_select(const AcceptParams& p, NucList& L, int n, uint64_t S_all, uint64_t rnd,
                                  const uint32_t (&W)[ACC_EPT], int base, uint64_t* red, int* redi) {
  constexpr int PER = NUC_LIST_MAX / ACC_THREADS;   // list elements per thread
  uint64_t* K = reinterpret_cast<uint64_t*>(L.w);    // NUC_LIST_MAX keys over w[] and id[]
  int n2 = 32;
  while (n2 < n) n2 <<= 1;
  uint64_t kk[PER];
#pragma unroll
  for (int r = 0; r < PER; ++r) {
    const int i = threadIdx.x + r * ACC_THREADS;
    kk[r] = i < n ? nuc_key(L.w[i], L.id[i]) : 0ull;   // padding sorts last (every list W >= 1)
  }
  __syncthreads();
#pragma unroll
  for (int r = 0; r < PER; ++r) {
    const int i = threadIdx.x + r * ACC_THREADS;
    if (i < n2) K[i] = kk[r];
  }
  __syncthreads();
  for (int k = 2; k <= n2; k <<= 1)
    for (int j = k >> 1; j > 0; j >>= 1) {
      for (int i = threadIdx.x; i < n2; i += ACC_THREADS) {
        const int l = i ^ j;
        if (l > i) {
          const uint64_t a = K[i], b = K[l];
          if (((i & k) == 0) == (a < b)) {   // descending blocks where bit k of i is clear
            K[i] = b;
            K[l] = a;
          }
        }
      }
      __syncthreads();
    }
  // candidates and the kept prefix: thread t holds sorted elements PER*t .. PER*t + PER - 1
  const bool topk = p.top_k > 0 && p.top_k < p.V;
  const int nc = topk ? min(p.top_k, n) : n;
  const int i0 = threadIdx.x * PER;
  uint64_t wsum = 0;
#pragma unroll
  for (int e = 0; e < PER; ++e)
    if (i0 + e < nc) wsum += K[i0 + e] >> 32;
  const uint64_t S = topk ? block_sum_u64(wsum, red) : S_all;
  const uint64_t prod = (uint64_t)p.p_fixed * S;
  const uint64_t thr = (prod >> 24) + ((prod & 0xFFFFFFull) ? 1 : 0);
  const uint64_t before = block_exscan_u64(wsum, red);
  // the first sorted index whose inclusive mass reaches thr (index 0 when thr = 0); the list
  // provably holds it
  if (thr == 0 ? threadIdx.x == 0 : (before < thr && before + wsum >= thr)) {
    uint64_t cum = before;
#pragma unroll
    for (int e = 0; e < PER; ++e) {
      cum += K[i0 + e] >> 32;
      if (cum >= thr) {
        L.kstar = K[i0 + e];
        L.sk = cum;
        break;
      }
    }
  }
  __syncthreads();
  const uint64_t kstar = L.kstar, Sk = L.sk;
  const uint64_t tau = __umul64hi(rnd, Sk);
  // 7. the first kept id (ascending) whose inclusive cumulative weight exceeds tau
  uint64_t mine = 0;
#pragma unroll
  for (int e = 0; e < ACC_EPT; ++e)
    if (nuc_key(W[e], base + e) >= kstar) mine += W[e];
  const uint64_t below = block_exscan_u64(mine, red);
  if (threadIdx.x == 0) redi[0] = 0x7FFFFFFF;
  __syncthreads();
  if (below <= tau && below + mine > tau) {
    uint64_t cum = below;
    int pick = 0x7FFFFFFF;
#pragma unroll
    for (int e = 0; e < ACC_EPT; ++e) {
      if (nuc_key(W[e], base + e) >= kstar) {
        cum += W[e];
        if (cum > tau && pick == 0x7FFFFFFF) pick = base + e;
      }
    }
    redi[0] = pick;
  }
  __syncthreads();
  const int out = redi[0];
  __syncthreads();
  return out;
}

__device__ __forceinline__ int row_nucleus(const AcceptParams& p, const float* row, int position, int seq,
                                           float* redf, uint64_t* red, int* redi, NucList& L) {
  const int V = p.V;
  const int base = threadIdx.x * ACC_EPT;
  uint32_t W[ACC_EPT];
  float mx = -INFINITY;
  bool nan = false;
  if (threadIdx.x < NUC_FLOORS) L.cnt[threadIdx.x] = 0;   // published by block_max_f's barriers
  if (threadIdx.x < 3) L.mhi[threadIdx.x] = L.mlo[threadIdx.x] = 0;
  {
    // 1. logits (NaN -> -inf; ids >= V are -inf, hence W = 0) and the row maximum
    float l[ACC_EPT];
#pragma unroll
    for (int e = 0; e < ACC_EPT; e += 4) {
      float4 v = make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
      if (base + e + 3 < V) {
        v = __ldcg(reinterpret_cast<const float4*>(row + base + e));
      } else {
        if (base + e < V) v.x = __ldcg(row + base + e);
        if (base + e + 1 < V) v.y = __ldcg(row + base + e + 1);
        if (base + e + 2 < V) v.z = __ldcg(row + base + e + 2);
      }
      l[e] = v.x; l[e + 1] = v.y; l[e + 2] = v.z; l[e + 3] = v.w;
    }
#pragma unroll
    for (int e = 0; e < ACC_EPT; ++e) {
      if (l[e] != l[e]) {
        nan = true;
        l[e] = -INFINITY;
      }
      mx = fmaxf(mx, l[e]);
    }
    if (nan) set_error(p.err, ERR_NAN_LOGITS);
    mx = block_max_f(mx, redf);
    // 2-3. W_i = floor(exp((l_i - max) / T) * 2^24)
#pragma unroll
    for (int e = 0; e < ACC_EPT; ++e) W[e] = fixed24(exp_sd(__fdiv_rn(__fsub_rn(l[e], mx), p.temperature)));
  }
  // 6. the 64-bit draw keyed by (produced position, sequence)
  uint32_t ctr[4] = {(uint32_t)position, (uint32_t)seq, 0u, 0u};
  philox4x32_10(ctr, (uint32_t)(p.seed & 0xFFFFFFFFull), (uint32_t)(p.seed >> 32));
  const uint64_t rnd = ((uint64_t)ctr[0] << 32) | ctr[1];

  // ---- the list path: counts (and, without top-k, masses) of the weights above each floor
  {
    const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const bool topk = p.top_k > 0 && p.top_k < V;
    uint32_t c01 = 0, c23 = 0, c45 = 0, c6 = 0;   // per-thread counts, two 11-bit fields per word
    uint32_t m4 = 0, m5 = 0, m6 = 0;              // per-thread masses >= floors 4, 5, 6 (< 2^29)
#pragma unroll
    for (int e = 0; e < ACC_EPT; ++e) {
      const int b = nuc_bucket(W[e]);
      c01 += (b <= 0 ? 1u : 0u) + (b <= 1 ? 1u << 11 : 0u);
      c23 += (b <= 2 ? 1u : 0u) + (b <= 3 ? 1u << 11 : 0u);
      c45 += (b <= 4 ? 1u : 0u) + (b <= 5 ? 1u << 11 : 0u);
      c6 += b <= 6 ? 1u : 0u;
      if (!topk) {
        m4 += b <= 4 ? W[e] : 0u;
        m5 += b <= 5 ? W[e] : 0u;
        m6 += W[e];
      }
    }
    c01 = __reduce_add_sync(0xffffffffu, c01);   // warp totals <= 1024 per field
    c23 = __reduce_add_sync(0xffffffffu, c23);
    c45 = __reduce_add_sync(0xffffffffu, c45);
    c6 = __reduce_add_sync(0xffffffffu, c6);
    uint32_t mh[3] = {0, 0, 0}, ml[3] = {0, 0, 0};
    if (!topk) {
      const uint32_t m[3] = {m4, m5, m6};
#pragma unroll
      for (int i = 0; i < 3; ++i) {
        mh[i] = __reduce_add_sync(0xffffffffu, m[i] >> 12);
        ml[i] = __reduce_add_sync(0xffffffffu, m[i] & 4095u);
      }
    }
    if (lane == 0) {
      atomicAdd(&L.cnt[0], c01 & 2047u);
      atomicAdd(&L.cnt[1], c01 >> 11);
      atomicAdd(&L.cnt[2], c23 & 2047u);
      atomicAdd(&L.cnt[3], c23 >> 11);
      atomicAdd(&L.cnt[4], c45 & 2047u);
      atomicAdd(&L.cnt[5], c45 >> 11);
      atomicAdd(&L.cnt[6], c6);
      if (!topk)
#pragma unroll
        for (int i = 0; i < 3; ++i) {
          atomicAdd(&L.mhi[i], (unsigned long long)mh[i]);
          atomicAdd(&L.mlo[i], (unsigned long long)ml[i]);
        }
    }
    __syncthreads();
    int N[NUC_FLOORS];
#pragma unroll
    for (int f = 0; f < NUC_FLOORS; ++f) N[f] = (int)L.cnt[f];
    if (N[6] == 0) return 0;   // every weight 0 (all-NaN row): the lowest candidate, id 0
    uint64_t Sf[3];
#pragma unroll
    for (int i = 0; i < 3; ++i) Sf[i] = (L.mhi[i] << 12) + L.mlo[i];
    const uint64_t S_all = Sf[2];
    uint64_t thr_all = 0;
    if (!topk) {
      const uint64_t prod = (uint64_t)p.p_fixed * S_all;
      thr_all = (prod >> 24) + ((prod & 0xFFFFFFull) ? 1 : 0);
    }
    // the highest floor whose elements provably hold the candidates (top-k) or the kept prefix
    int f = -1;
#pragma unroll
    for (int i = 0; i < NUC_FLOORS; ++i) {
      const bool holds = topk ? (N[i] >= p.top_k || N[i] == N[6]) : (i >= 4 && Sf[i - 4] >= thr_all);
      if (f < 0 && N[i] <= NUC_LIST_MAX && holds) f = i;
    }
    if (f >= 0) {
      uint32_t mine = 0;
#pragma unroll
      for (int e = 0; e < ACC_EPT; ++e) mine += nuc_bucket(W[e]) <= f;
      uint32_t at = (uint32_t)block_exscan_u64(mine, red);
#pragma unroll
      for (int e = 0; e < ACC_EPT; ++e)
        if (nuc_bucket(W[e]) <= f) {
          L.w[at] = W[e];
          L.id[at] = base + e;
          ++at;
        }
      __syncthreads();
      // a kept set (or top-k) of at most 32 on the lanes of one warp when that is cheap: a
      // small top-k, or a short list; otherwise, or when it does not apply, the sorted list
      if ((topk && p.top_k <= 32) || N[f] <= 64) {
        if (w == 0) {
          const int pick = list_small(p, L, N[f], S_all, topk, rnd);
          if (lane == 0) L.pick = pick;
        }
        __syncthreads();
        const int pick = L.pick;
        if (pick >= 0) return pick;
      }
      return list_sorted_select(p, L, N[f], S_all, rnd, W, base, red, redi);
    }
  }

  // ---- the block-wide path over all ids
  Cut c;
  c.xk = 0;
  c.idk = 0x7FFFFFFF;
  c.xp = 0;
  c.idp = 0x7FFFFFFF;
  // 4. top-k candidates
  if (p.top_k > 0 && p.top_k < V) {
    c.xk = search_threshold<P_GE, true>(W, base, c, (uint64_t)p.top_k, red);
    const uint64_t above = block_sum_u64(lsum<P_GT, true>(W, base, c, c.xk), red);
    c.idk = nth_id<P_EQ>(W, base, c, c.xk, (uint64_t)p.top_k - above, red, redi);
  }
  // 5. top-p over the candidates: thr = ceil(P * S / 2^24), P <= 2^24, S < 2^40
  const uint64_t S = block_sum_u64(lsum<P_CAND, false>(W, base, c, 0), red);
  if (S == 0) return nth_id<P_CAND>(W, base, c, 0, 1, red, redi);   // all-NaN row: lowest candidate
  const uint64_t prod = (uint64_t)p.p_fixed * S;
  const uint64_t thr = (prod >> 24) + ((prod & 0xFFFFFFull) ? 1 : 0);
  c.xp = search_threshold<P_CAND_GE, false>(W, base, c, thr, red);
  const uint64_t above = block_sum_u64(lsum<P_CAND_GT, false>(W, base, c, c.xp), red);
  const uint64_t n_above = block_sum_u64(lsum<P_CAND_GT, true>(W, base, c, c.xp), red);
  uint64_t ties = thr > above ? (thr - above + c.xp - 1) / c.xp : 0;
  if (n_above == 0 && ties == 0) ties = 1;
  c.idp = ties == 0 ? -1 : nth_id<P_CAND_EQ>(W, base, c, c.xp, ties, red, redi);
  const uint64_t Sk = block_sum_u64(lsum<P_KEPT, false>(W, base, c, 0), red);
  const uint64_t tau = __umul64hi(rnd, Sk);
  // 7. the first kept id (ascending) whose inclusive cumulative weight exceeds tau
  const uint64_t mine = lsum<P_KEPT, false>(W, base, c, 0);
  const uint64_t before = block_exscan_u64(mine, red);
  if (threadIdx.x == 0) redi[0] = 0x7FFFFFFF;
  __syncthreads();
  if (before <= tau && before + mine > tau) {
    uint64_t cum = before;
    int pick = 0x7FFFFFFF;
#pragma unroll
    for (int e = 0; e < ACC_EPT; ++e) {
      if (pred<P_KEPT>(W[e], base + e, c, 0)) {
        cum += W[e];
        if (cum > tau && pick == 0x7FFFFFFF) pick = base + e;
      }
    }
    redi[0] = pick;
  }
  __syncthreads();
  const int out = redi[0];
  __syncthreads();
  return out;
}

// parent of tree row i (0 < i < q): an earlier row; anything else is flagged and read as the root
__device__ __forceinline__ int tree_parent(const int* par, int i, uint32_t* err) {
  int pi = __ldcg(par + i);
  if (pi < 0 || pi >= i) {
    set_error(err, ERR_TREE);
    pi = 0;
  }
  return pi;
}

// depth of tree row j (the root has depth 0); at most j steps since parents are earlier rows
__device__ __forceinline__ int tree_depth(const int* par, int j, uint32_t* err) {
  int d = 0;
  for (int i = j; i > 0; i = tree_parent(par, i, err)) ++d;
  return d;
}

__global__ void __launch_bounds__(ACC_THREADS) accept_kernel(const AcceptParams p) {
  __shared__ float redf[32];
  __shared__ uint64_t red[32];
  __shared__ int redi[32];
  __shared__ int s_last;
  __shared__ NucList nl;
  pdl_wait();
  pdl_trigger();
  const int j = blockIdx.x, sl = blockIdx.y, s = p.seq0 + sl;
  const float* row = p.logits + (size_t)(sl * p.q + j) * p.V;
  int t;
  if (p.temperature <= 0.f) {
    t = row_argmax(row, p.V, p.err, redf, redi);
  } else {
    // the produced token's position: one past the row's own (len + j, or len + depth(j))
    const int position = __ldcg(p.len + s) + (p.parent ? tree_depth(p.parent + sl * p.q, j, nullptr) : j) + 1;
    t = row_nucleus(p, row, position, s, redf, red, redi, nl);
  }
  if (threadIdx.x == 0) p.targets[sl * p.q + j] = t;
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) s_last = (atomicAdd(p.counters + sl, 1) == p.q - 1);
  __syncthreads();
  if (!s_last || threadIdx.x != 0) return;
  __threadfence();
  int tg[SDSAT_ATT_MAXQ];
  for (int i = 0; i < p.q; ++i) tg[i] = __ldcg(p.targets + sl * p.q + i);
  int m = 0;
  if (!p.parent) {
    const int nv = p.n_verify_dev ? min(max(__ldcg(p.n_verify_dev + sl), 0), p.q - 1) : p.n_verify;
    for (int i = 1; i <= nv; ++i) {                 // Eq. 3: prefix of matching drafts
      if (__ldcg(p.drafts + sl * p.q + i) != tg[i - 1]) break;
      m = i;
    }
    for (int i = 0; i < p.q; ++i) p.out_tokens[sl * p.q + i] = tg[i];
  } else {
    // Sec. 2.1.2: the longest branch accepted by the chain test applied along every branch
    const int* par = p.parent + sl * p.q;
    int dep[SDSAT_ATT_MAXQ], path[SDSAT_ATT_MAXQ];
    uint32_t accm = 1u;
    int best = 0;
    dep[0] = 0;
    for (int i = 1; i < p.q; ++i) {
      const int pi = tree_parent(par, i, p.err);
      dep[i] = dep[pi] + 1;
      if (((accm >> pi) & 1u) && __ldcg(p.drafts + sl * p.q + i) == tg[pi]) {
        accm |= 1u << i;
        if (dep[i] > dep[best]) best = i;
      }
    }
    m = dep[best];
    for (int d = m, i = best; d >= 0; --d) {
      path[d] = i;
      if (d > 0) i = tree_parent(par, i, nullptr);
    }
    for (int i = 0; i < p.q; ++i) {
      p.out_tokens[sl * p.q + i] = i <= m ? tg[path[i]] : -1;
      if (p.path) p.path[sl * p.q + i] = i <= m ? path[i] : -1;
    }
    // the compaction kernel's input: committed length before this step, m, the path rows
    int* w = p.tree_ws + sl * TREE_WS_STRIDE;
    w[0] = __ldcg(p.len + s);
    w[1] = m;
    for (int i = 0; i <= m; ++i) w[2 + i] = path[i];
  }
  p.accepted_len[sl] = 1 + m;
  if (p.commit) {
    const int nl = __ldcg(p.len + s) + 1 + m;
    if (nl <= p.cap) p.len[s] = nl;
    else set_error(p.err, ERR_CAPACITY);
    if (p.emitted) p.emitted[s] += 1 + m;
  }
  p.counters[sl] = 0;
}

static cudaLaunchConfig_t make_cfg(dim3 grid, dim3 block, cudaStream_t st, bool pdl, cudaLaunchAttribute* attr) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.stream = st;
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cfg;
}

cudaError_t launch_accept(const AcceptParams& p, cudaStream_t st, bool pdl) {
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg = make_cfg(dim3(p.q, p.nb), dim3(ACC_THREADS), st, pdl, attr);
  return cudaLaunchKernelEx(&cfg, accept_kernel, p);
}

// ---- RMSNorm into the GEMM operand ------------------------------------------------------
// x = h * rsqrt(mean(h^2) + eps) * g (Llama's RMSNorm, fp32), stored as bf16 hi + lo with
// hi = bf16(x), lo = bf16(x - hi), so hi + lo carries ~16 significant bits of x.  With
// tokens != null the row is first gathered from the embedding table (h = E[token]).
__device__ __forceinline__ void split_store(float v, __nv_bfloat16* hi, __nv_bfloat16* lo) {
  const __nv_bfloat16 h = __float2bfloat16_rn(v);
  *hi = h;
  *lo = __float2bfloat16_rn(v - __bfloat162float(h));
}

__global__ void __launch_bounds__(256) rmsnorm_kernel(const int* tokens, const __nv_bfloat16* E, int V, float* h,
                                                      int d, const __nv_bfloat16* g, float eps, __nv_bfloat16* xhi,
                                                      __nv_bfloat16* xlo, uint32_t* err) {
  __shared__ float red[32];
  pdl_wait();
  pdl_trigger();
  const int m = blockIdx.x;
  float* hr = h + (size_t)m * d;
  const __nv_bfloat16* er = nullptr;
  if (tokens) {
    int t = __ldcg(tokens + m);
    if (t < 0 || t >= V) {
      if (threadIdx.x == 0) set_error(err, ERR_TOKEN);
      t = 0;
    }
    er = E + (size_t)t * d;
  }
  float ss = 0.f;
  for (int i = threadIdx.x * 4; i < d; i += blockDim.x * 4) {
    float4 v;
    if (er) {
      const __nv_bfloat162* e2 = reinterpret_cast<const __nv_bfloat162*>(er + i);
      const float2 a = __bfloat1622float2(e2[0]), b = __bfloat1622float2(e2[1]);
      v = make_float4(a.x, a.y, b.x, b.y);
      *reinterpret_cast<float4*>(hr + i) = v;
    } else {
      v = __ldcg(reinterpret_cast<const float4*>(hr + i));
    }
    ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
  __syncthreads();
  if (threadIdx.x < 32) {
    float t = threadIdx.x < (blockDim.x >> 5) ? red[threadIdx.x] : 0.f;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
    if (threadIdx.x == 0) red[0] = t;
  }
  __syncthreads();
  const float inv = 1.0f / sqrtf(red[0] / (float)d + eps);
  for (int i = threadIdx.x * 4; i < d; i += blockDim.x * 4) {
    const float4 v = __ldcg(reinterpret_cast<const float4*>(hr + i));
    const float vv[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int e = 0; e < 4; ++e)
      split_store(vv[e] * inv * __bfloat162float(g[i + e]), xhi + (size_t)m * d + i + e, xlo + (size_t)m * d + i + e);
  }
}

cudaError_t launch_rmsnorm(const int* tokens, const __nv_bfloat16* E, int V, float* h, int d, int M,
                           const __nv_bfloat16* gain, float eps, __nv_bfloat16* xhi, __nv_bfloat16* xlo,
                           uint32_t* err, cudaStream_t st, bool pdl) {
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg = make_cfg(dim3(M), dim3(256), st, pdl, attr);
  return cudaLaunchKernelEx(&cfg, rmsnorm_kernel, tokens, E, V, h, d, gain, eps, xhi, xlo, err);
}

__global__ void split_kernel(const float* x, int n, __nv_bfloat16* xhi, __nv_bfloat16* xlo) {
  pdl_wait();
  pdl_trigger();
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) split_store(__ldcg(x + i), xhi + i, xlo + i);
}

cudaError_t launch_split(const float* x, int M, int K, __nv_bfloat16* xhi, __nv_bfloat16* xlo, cudaStream_t st,
                         bool pdl) {
  cudaLaunchAttribute attr[1];
  const int n = M * K;
  cudaLaunchConfig_t cfg = make_cfg(dim3((n + 255) / 256), dim3(256), st, pdl, attr);
  return cudaLaunchKernelEx(&cfg, split_kernel, x, n, xhi, xlo);
}

// ---- block input of draft step 1 (mode 1) and draft step 2 (mode 2) --------------------
// The previous block had prev_q rows per sequence.  Mode 2 builds `width` chains of k drafts
// below the root (width 1: the chain block; row 1 + w*k + i - 1 holds branch w's draft for
// position len + i, from table w).
__global__ void build_block_kernel(BuildParams b) {
  pdl_wait();
  pdl_trigger();
  const int sl = blockIdx.x, j = threadIdx.x;
  const int* prev = b.prev_out + sl * b.prev_q;
  if (b.mode == 3) {
    // pipelined blocks [x_0, r_1 .. r_k, a_1 .. a_k]: mode A (drafts known) after a mode-S
    // block or after a mode-A block that accepted all k drafts, else mode S (r_i = a_i);
    // x_0 = the newest emitted token, the drafts the k targets after it
    const int acc = __ldcg(b.prev_acc + sl);
    const bool a_mode = __ldcg(b.pipe_mode + sl) == 0 || acc == b.k + 1;
    __syncthreads();   // every thread has read the previous mode before thread 0 replaces it
    if (j == 0) {
      b.pipe_mode[sl] = a_mode ? 1 : 0;
      b.pipe_nverify[sl] = a_mode ? b.k : 0;
    }
    if (j >= b.q) return;
    int t;
    if (j == 0) {
      t = __ldcg(prev + acc - 1);
    } else if (j <= b.k && a_mode) {
      t = b.table ? __ldcg(b.table + (size_t)sl * b.table_stride + __ldcg(b.len + sl) + j) : __ldcg(prev + acc - 1 + j);
    } else {
      t = b.adaptive[(j - 1) % b.k];
    }
    b.tokens[sl * b.q + j] = t;
    return;
  }
  if (j >= b.q) return;
  int t;
  if (b.mode == 1) {
    t = (j == 0) ? __ldcg(prev + __ldcg(b.prev_acc + sl) - 1) : b.adaptive[j - 1];
  } else if (j == 0) {
    t = __ldcg(prev);
  } else {
    const int w = (j - 1) / b.k, i = (j - 1) % b.k + 1;
    if (b.table)
      t = __ldcg(b.table + ((size_t)w * b.table_batch + sl) * b.table_stride + __ldcg(b.len + sl) + i);
    else
      t = __ldcg(prev + i);
  }
  b.tokens[sl * b.q + j] = t;
}

cudaError_t launch_build_block(const BuildParams& b, cudaStream_t st, bool pdl) {
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg = make_cfg(dim3(b.nb), dim3(32), st, pdl, attr);
  return cudaLaunchKernelEx(&cfg, build_block_kernel, b);
}

// ---- tree blocks: positions and attention masks, and the commit's KV compaction ----------
// Row j of a tree block: position len + depth(j) and the mask of the block rows it attends
// (its ancestors and itself).  One thread per row.
__global__ void tree_prep_kernel(const int* parent, const int* len, int nb, int q, int* pos, uint32_t* anc,
                                 uint32_t* err) {
  pdl_wait();
  pdl_trigger();
  const int r = threadIdx.x;
  if (r >= nb * q) return;
  const int sl = r / q, j = r % q;
  const int* par = parent + sl * q;
  if (j == 0 && __ldcg(par) != -1) set_error(err, ERR_TREE);
  uint32_t m = 1u << j;
  int d = 0;
  for (int i = j; i > 0; ++d) {
    i = tree_parent(par, i, err);
    m |= 1u << i;
  }
  pos[r] = __ldcg(len + sl) + d;
  anc[r] = m;
}

cudaError_t launch_tree_prep(const int* parent, const int* len, int nb, int q, int* pos, uint32_t* anc,
                             uint32_t* err, cudaStream_t st, bool pdl) {
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg = make_cfg(dim3(1), dim3(TREE_MAX_ROWS), st, pdl, attr);
  return cudaLaunchKernelEx(&cfg, tree_prep_kernel, parent, len, nb, q, pos, anc, err);
}

// Slot len0 + i receives the K and V rows of slot len0 + n_i (i = 1..m; n_i >= i, so no
// source is overwritten before it is read).  One CTA per (layer, head) and sequence, 16-byte
// chunks.
__global__ void tree_compact_kernel(const int* ws, int H, int hd, int cap, int batch, __nv_bfloat16* kc,
                                    __nv_bfloat16* vc) {
  pdl_wait();
  pdl_trigger();
  const int l = blockIdx.x / H, h = blockIdx.x % H, s = blockIdx.y;
  const int* w = ws + s * TREE_WS_STRIDE;
  const int len0 = __ldcg(w), m = __ldcg(w + 1);
  const int chunks = hd / 8;   // 16-byte chunks per row
  const size_t off = (((size_t)l * batch + s) * H + h) * cap * hd;
  for (int x = threadIdx.x; x < 2 * m * chunks; x += blockDim.x) {
    const int which = x / (m * chunks), rem = x % (m * chunks);
    const int i = 1 + rem / chunks, ch = rem % chunks;
    const int n = __ldcg(w + 2 + i);
    if (n == i || len0 + n >= cap) continue;
    __nv_bfloat16* base = (which ? vc : kc) + off;
    const uint4 v = __ldcg(reinterpret_cast<const uint4*>(base + (size_t)(len0 + n) * hd) + ch);
    __stcg(reinterpret_cast<uint4*>(base + (size_t)(len0 + i) * hd) + ch, v);
  }
}

cudaError_t launch_tree_compact(const int* ws, int nb, int L, int H, int hd, int cap, int batch,
                                __nv_bfloat16* k, __nv_bfloat16* v, cudaStream_t st, bool pdl) {
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg = make_cfg(dim3(L * H, nb), dim3(64), st, pdl, attr);
  return cudaLaunchKernelEx(&cfg, tree_compact_kernel, ws, H, hd, cap, batch, k, v);
}

// ---- the bounded wait, run out on purpose (a test hook) ----------------------------------
// One CTA waits on an mbarrier that nothing arrives on, through the same bounded wait every
// kernel uses: after WAIT_LIMIT_NS it sets ERR_TIMEOUT and returns; nothing faults.
__global__ void wait_timeout_kernel(uint32_t* err) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();
  mbar_wait_bounded(&bar, 0, &abort_flag, err);
}

cudaError_t launch_wait_timeout(uint32_t* err, cudaStream_t st) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(1);
  cfg.blockDim = dim3(32);
  cfg.stream = st;
  return cudaLaunchKernelEx(&cfg, wait_timeout_kernel, err);
}

// ---- explicit commit / rollback, and prefill commit --------------------------------------
__global__ void commit_kernel(int* len, const int* new_len, int nb, int cap, uint32_t* err) {
  pdl_wait();
  pdl_trigger();
  const int s = threadIdx.x;
  if (s >= nb) return;
  int v = __ldcg(new_len + s);
  if (v < 0 || v > cap) {
    set_error(err, ERR_CAPACITY);
    v = v < 0 ? 0 : cap;
  }
  len[s] = v;
}

cudaError_t launch_commit(int* len, const int* new_len, int nb, int cap, uint32_t* err, cudaStream_t st,
                          bool pdl) {
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg = make_cfg(dim3(1), dim3(64), st, pdl, attr);
  return cudaLaunchKernelEx(&cfg, commit_kernel, len, new_len, nb, cap, err);
}

__global__ void add_len_kernel(int* len, int seq, int n, int cap, uint32_t* err) {
  pdl_wait();
  pdl_trigger();
  const int v = __ldcg(len + seq) + n;
  if (v > cap) set_error(err, ERR_CAPACITY);
  len[seq] = v > cap ? cap : v;
}

cudaError_t launch_add_len(int* len, int seq, int n, int cap, uint32_t* err, cudaStream_t st, bool pdl) {
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg = make_cfg(dim3(1), dim3(1), st, pdl, attr);
  return cudaLaunchKernelEx(&cfg, add_len_kernel, len, seq, n, cap, err);
}

__global__ void exp_kernel(const float* in, float* out, int n) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) out[i] = exp_sd(in[i]);
}

cudaError_t launch_exp(const float* in, float* out, int n, cudaStream_t st) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((n + 255) / 256);
  cfg.blockDim = dim3(256);
  cfg.stream = st;
  return cudaLaunchKernelEx(&cfg, exp_kernel, in, out, n);
}

}  // namespace sdsat
