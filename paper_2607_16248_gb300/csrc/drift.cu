// kvq_drift_metrics / kvq_drift_window: offline drift metrics on paired FP16
// and low-bit logits and the recovery-window rule (Sec. 4.1 "Adaptive
// recovery-window selection", Sec. 4.2 "Offline supervision and
// calibration").
//
// Per step (row) t, with p = softmax(z):
//   C(alpha)  the shortest prefix of the FP16 order (z_fp descending, lower
//             index first among equal values) whose mass reaches alpha; M_t
//             its size;
//   S         TopK(z_q, K), same order on z_q;
//   c_t       sum of p_fp over C and S;
//   d_loc     || p_fp / p_fp(U) - p_q / p_q(U) ||_2 over U = C union S;
//   y_t       d_loc > eps and c_t >= rho_c;
//   cov_t(k)  sum of p_fp over C and TopK(z_q, k), k = 1 .. k_max.
// K_b is the smallest k whose coverage averaged over the rows reaches rho_K.
//
// One cluster of 8 CTAs per row.  Each CTA stages an eighth of both logit
// rows in shared memory once (the only HBM read) and the CTAs combine their
// partial results through distributed shared memory:
//   1. maxima;
//   2. the FP16 boundary: a 2048-bin histogram of the depth (m - z) * 64
//      (count and mass per bin, the depth order is the FP16 order) and, in
//      the same pass, the normaliser S_fp = sum e^{z - m}, find the bin
//      where the prefix mass reaches alpha S_fp; that bin's elements are
//      sorted in one CTA and scanned for the exact element.  A bin with more
//      than 2048 elements is narrowed by histograms of its key range first;
//      a range of equal keys takes the lowest indices (counted per CTA in
//      index order);
//   3. the same selection by count on z_q gives the k_max-th element, then
//      the k_max best elements are gathered and sorted (the TopK order);
//   4. one pass over U: its masses (fixed point) and the sums of e_fp^2,
//      e_fp e_q, e_q^2 (double-float), from which d_loc follows.
// A mass term e = expf(z - m) (fp32, in (0, 1]) is taken as an integer
// multiple of 2^-40 (round to nearest) and every mass sum is an exact 64-bit
// integer sum: the same numbers decide every comparison, in any order, and
// no per-element fp64 arithmetic is needed.

#include <float.h>

#include "common.cuh"

namespace kvq {
namespace {

constexpr int kT = 512;              // threads per CTA
constexpr int kW = kT / 32;
constexpr int kCl = 8;               // CTAs per row (one cluster)
constexpr int kSlice = 20480;        // logits per CTA and array: vocab <= 8 * kSlice
constexpr int kBins = 2048;          // histogram bins
constexpr int kCap = 2048;           // largest boundary set sorted in one CTA
constexpr int kMaxKcov = 256;        // longest coverage curve
constexpr float kDepthScale = 64.0f; // bins per unit of depth m - z
constexpr int kSlots = 32;           // exchange slots (one per cluster exchange)
constexpr int kXw = 4;               // words per exchange
typedef unsigned long long u64;

struct Sm {
  float zf[kSlice];
  float zq[kSlice];
  uint32_t hc[kBins];               // bin counts
  uint32_t hm[3][kBins];            // bin masses: 14-bit chunks of the fixed-point terms
  u64 buf[kCap];                    // rank 0: boundary set / TopK set
  u64 xd[kSlots][kXw];              // per-CTA partials read by the peers
  uint32_t xu[kSlots][2];
  uint32_t res_u[8];                // rank 0: results of a selection
  u64 res_q[4];                     // the boundary bin's owner: its result
  uint32_t nbuf;                    // rank 0: fill count of buf
  u64 rq[kW];
  // merged histogram of this CTA's eighth of the bins, and exchange scratch
  uint32_t rc[kBins / kCl];
  u64 rm[kBins / kCl];
  u64 xin[kCl][kXw];                // values loaded from the eight CTAs
  u64 xin8[kCl][2 * kXw];           // the same for a two-slot exchange
  u64 wsel[kMaxKcov];               // coverage terms of the TopK list
  float bc[4];                      // broadcast scalars
  uint32_t ru[kW];
  float rf[kW];
};

// ---- cluster primitives (distributed shared memory) ----
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::
                   : "memory");
}
__device__ __forceinline__ uint32_t peer_addr(const void* p, uint32_t rank) {
  uint32_t a;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(a) : "r"(smem_u32(p)), "r"(rank));
  return a;
}
__device__ __forceinline__ float ld_peer_f32(uint32_t a) {
  float v;
  asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(a) : "memory");
  return v;
}
__device__ __forceinline__ u64 ld_peer_u64(uint32_t a) {
  u64 v;
  asm volatile("ld.shared::cluster.u64 %0, [%1];" : "=l"(v) : "r"(a) : "memory");
  return v;
}
__device__ __forceinline__ uint32_t ld_peer_u32(uint32_t a) {
  uint32_t v;
  asm volatile("ld.shared::cluster.u32 %0, [%1];" : "=r"(v) : "r"(a) : "memory");
  return v;
}
__device__ __forceinline__ void st_peer_u64(uint32_t a, unsigned long long v) {
  asm volatile("st.shared::cluster.u64 [%0], %1;" ::"r"(a), "l"(v) : "memory");
}
__device__ __forceinline__ void st_peer_u32(uint32_t a, uint32_t v) {
  asm volatile("st.shared::cluster.u32 [%0], %1;" ::"r"(a), "r"(v) : "memory");
}
__device__ __forceinline__ uint32_t atom_add_peer(uint32_t a, uint32_t v) {
  uint32_t old;
  asm volatile("atom.shared::cluster.add.u32 %0, [%1], %2;" : "=r"(old) : "r"(a), "r"(v) : "memory");
  return old;
}

// Order-preserving key of a float (larger float, larger key; -0 as +0) and
// back.  Every key of a non-NaN float is > 0.
__device__ __forceinline__ uint32_t fkey(float x) {
  uint32_t u = __float_as_uint(x);
  if ((u << 1) == 0u) u = 0u;
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float fval(uint32_t k) {
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7fffffffu) : ~k);
}
// A mass term e in [0, 1] as a multiple of 2^-40, rounded to nearest: e 2^20
// splits exactly into its integer part and a fraction whose 2^20 multiple
// fits a u32.
__device__ __forceinline__ u64 fix40(float e) {
  const float a = e * 1048576.0f;
  const uint32_t hi = (uint32_t)a;
  const uint32_t lo = __float2uint_rn((a - (float)hi) * 1048576.0f);
  return ((u64)hi << 20) + lo;
}
constexpr double kFix = 1099511627776.0;  // 2^40

// Double-float accumulator: an unevaluated sum hi + lo of two floats
// (error-free transformations: two-sum and the fma product residual).
struct Df {
  float hi = 0.0f, lo = 0.0f;
  __device__ __forceinline__ void add(float x) {
    const float s = hi + x;
    const float bb = s - hi;
    const float e = (hi - (s - bb)) + (x - bb);
    const float l = lo + e;
    hi = s + l;
    lo = l - (hi - s);
  }
  __device__ __forceinline__ void add(const Df& o) {
    add(o.hi);
    add(o.lo);
  }
  __device__ __forceinline__ void add_prod(float a, float b) {
    const float p = a * b;
    add(p);
    add(fmaf(a, b, -p));
  }
  __device__ __forceinline__ u64 pack() const {
    return ((u64)__float_as_uint(hi) << 32) | __float_as_uint(lo);
  }
  __device__ static Df unpack(u64 w) {
    Df d;
    d.hi = __uint_as_float((uint32_t)(w >> 32));
    d.lo = __uint_as_float((uint32_t)w);
    return d;
  }
  __device__ __forceinline__ double value() const { return (double)hi + (double)lo; }
};

// (key, index) packed so that a larger word ranks first: key descending,
// index ascending.
__device__ __forceinline__ unsigned long long pack(uint32_t k, uint32_t i) {
  return ((unsigned long long)k << 32) | (0xffffffffu - i);
}
__device__ __forceinline__ uint32_t pk_key(unsigned long long w) { return (uint32_t)(w >> 32); }
__device__ __forceinline__ uint32_t pk_idx(unsigned long long w) {
  return 0xffffffffu - (uint32_t)w;
}

// ---- block reductions (all threads get the result) ----
__device__ u64 block_sum_q(u64 v, Sm& s) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  __syncthreads();
  if ((threadIdx.x & 31) == 0) s.rq[threadIdx.x >> 5] = v;
  __syncthreads();
  u64 r = 0ull;
  for (int w = 0; w < kW; ++w) r += s.rq[w];
  return r;
}
__device__ Df block_sum_df(Df v, Sm& s) {
#pragma unroll
  for (int o = 16; o; o >>= 1) {
    Df w;
    w.hi = __shfl_xor_sync(0xffffffffu, v.hi, o);
    w.lo = __shfl_xor_sync(0xffffffffu, v.lo, o);
    // a fixed pairing order keeps every lane's result identical
    if ((threadIdx.x & o) == 0) {
      v.add(w);
    } else {
      w.add(v);
      v = w;
    }
  }
  __syncthreads();
  if ((threadIdx.x & 31) == 0) s.rq[threadIdx.x >> 5] = v.pack();
  __syncthreads();
  Df r;
  for (int w = 0; w < kW; ++w) r.add(Df::unpack(s.rq[w]));
  return r;
}
__device__ float block_max_f(float v, Sm& s) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  __syncthreads();
  if ((threadIdx.x & 31) == 0) s.rf[threadIdx.x >> 5] = v;
  __syncthreads();
  float r = -INFINITY;
  for (int w = 0; w < kW; ++w) r = fmaxf(r, s.rf[w]);
  return r;
}
__device__ uint32_t block_sum_u(uint32_t v, Sm& s) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  __syncthreads();
  if ((threadIdx.x & 31) == 0) s.ru[threadIdx.x >> 5] = v;
  __syncthreads();
  uint32_t r = 0u;
  for (int w = 0; w < kW; ++w) r += s.ru[w];
  return r;
}
__device__ uint32_t block_min_u(uint32_t v, Sm& s) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v = min(v, __shfl_xor_sync(0xffffffffu, v, o));
  __syncthreads();
  if ((threadIdx.x & 31) == 0) s.ru[threadIdx.x >> 5] = v;
  __syncthreads();
  uint32_t r = 0xffffffffu;
  for (int w = 0; w < kW; ++w) r = min(r, s.ru[w]);
  return r;
}
__device__ uint32_t block_max_u(uint32_t v, Sm& s) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v = max(v, __shfl_xor_sync(0xffffffffu, v, o));
  __syncthreads();
  if ((threadIdx.x & 31) == 0) s.ru[threadIdx.x >> 5] = v;
  __syncthreads();
  uint32_t r = 0u;
  for (int w = 0; w < kW; ++w) r = max(r, s.ru[w]);
  return r;
}

// Cluster-wide reductions of two values per CTA: each CTA publishes its
// partials in slot `slot`, and after the barrier every CTA combines all eight
// in rank order (identical results everywhere).
// Publish up to four words in slot `slot`; after the barrier threads load the
// eight CTAs' words in parallel into s.xin[rank][word].
__device__ void cluster_gather(Sm& s, int slot, u64 a, u64 b, u64 c = 0ull, u64 d = 0ull) {
  if (threadIdx.x == 0) {
    s.xd[slot][0] = a;
    s.xd[slot][1] = b;
    s.xd[slot][2] = c;
    s.xd[slot][3] = d;
  }
  cluster_sync();
  if (threadIdx.x < kXw * kCl)
    s.xin[threadIdx.x / kXw][threadIdx.x % kXw] =
        ld_peer_u64(peer_addr(&s.xd[slot][threadIdx.x % kXw], threadIdx.x / kXw));
  __syncthreads();
}
// Six words in slots `slot` and `slot + 1`, one barrier; s.xin8[rank][word].
__device__ void cluster_gather2x(Sm& s, int slot, u64 a, u64 b, u64 c, u64 d, u64 e, u64 f) {
  if (threadIdx.x == 0) {
    s.xd[slot][0] = a;
    s.xd[slot][1] = b;
    s.xd[slot][2] = c;
    s.xd[slot][3] = d;
    s.xd[slot + 1][0] = e;
    s.xd[slot + 1][1] = f;
  }
  cluster_sync();
  if (threadIdx.x < 2 * kXw * kCl) {
    const int r = threadIdx.x / (2 * kXw), w = threadIdx.x % (2 * kXw);
    s.xin8[r][w] = ld_peer_u64(peer_addr(&s.xd[slot + w / kXw][w % kXw], (uint32_t)r));
  }
  __syncthreads();
}
__device__ __forceinline__ void cluster_gather2(Sm& s, int slot, u64 a, u64 b) {
  cluster_gather(s, slot, a, b);
}
// op 0: (sum, sum); op 1: (min, max); op 2: (max, max) on float bits >= 0
__device__ void cluster_red2_u(Sm& s, int slot, uint32_t& a, uint32_t& b, int op) {
  cluster_gather2(s, slot, (u64)a, (u64)b);
  uint32_t ra = op == 1 ? 0xffffffffu : 0u, rb = 0u;
  for (int r = 0; r < kCl; ++r) {
    const uint32_t x = (uint32_t)s.xin[r][0];
    const uint32_t y = (uint32_t)s.xin[r][1];
    if (op == 0) {
      ra += x;
      rb += y;
    } else if (op == 1) {
      ra = min(ra, x);
      rb = max(rb, y);
    } else {
      ra = max(ra, x);
      rb = max(rb, y);
    }
  }
  __syncthreads();
  a = ra;
  b = rb;
}

// Bitonic sort of buf[0, n) descending (n <= kCap), padding with 0.
__device__ void sort_desc(Sm& s, int n) {
  int P = 2;
  while (P < n) P <<= 1;
  for (int i = n + threadIdx.x; i < P; i += kT) s.buf[i] = 0ull;
  __syncthreads();
  for (int k = 2; k <= P; k <<= 1)
    for (int j = k >> 1; j > 0; j >>= 1) {
      for (int i = threadIdx.x; i < P; i += kT) {
        const int ixj = i ^ j;
        if (ixj > i) {
          const unsigned long long a = s.buf[i], b = s.buf[ixj];
          const bool desc = (i & k) == 0;
          if (desc ? (a < b) : (a > b)) {
            s.buf[i] = b;
            s.buf[ixj] = a;
          }
        }
      }
      __syncthreads();
    }
}

struct Ctx {
  int n;          // logits in this CTA's slice
  uint32_t i0;    // global index of its first logit
  uint32_t rank;  // cluster rank
};

// Result of a selection: the element (key, index) at which the prefix of
// the order (key descending, index ascending) first reaches the target, and
// the prefix length.  all = the target is never reached (everything).
struct Pick {
  uint32_t key, idx, len;
  bool all;
};

// The bin where the prefix weight (count, or mass in fixed point) in bin
// order (bin 0 ranks first) reaches `target`, over the histograms of all
// eight CTAs.  CTA r merges bins [256 r, 256 r + 256) of the eight
// histograms and publishes their total; the CTA whose range holds the target
// finds the bin and publishes it.  If the total stays below the target: with
// `clamp` the last non-empty bin is taken, else false is returned (in every
// CTA alike).
// With `norm` set, each CTA's *norm holds its part of S_fp on entry and the
// target is ceil(alpha S_fp) over the cluster: *norm and target return it.
__device__ bool boundary_bin(Sm& s, const Ctx& cx, bool weighted, u64& target, int& slot, int& bin,
                             uint32_t& cnt_above, u64& w_above, uint32_t& cnt_bin,
                             bool clamp = false, u64* norm = nullptr, double alpha = 0.0) {
  constexpr int kR = kBins / kCl;  // bins per CTA range
  cluster_sync();                  // every CTA's histogram is complete
  const int t = threadIdx.x;
  __shared__ uint32_t part_c[kT];
  __shared__ u64 part_m[kT];
  {
    // thread t merges bin (t % kR) of its range from four of the CTAs
    const int b = (int)cx.rank * kR + (t % kR);
    const uint32_t r0 = (uint32_t)(t / kR) * (kCl / (kT / kR));
    uint32_t c = 0u, m0 = 0u, m1 = 0u, m2 = 0u;
#pragma unroll
    for (uint32_t r = 0; r < kCl / (kT / kR); ++r) {
      c += ld_peer_u32(peer_addr(&s.hc[b], r0 + r));
      if (weighted) {
        m0 += ld_peer_u32(peer_addr(&s.hm[0][b], r0 + r));
        m1 += ld_peer_u32(peer_addr(&s.hm[1][b], r0 + r));
        m2 += ld_peer_u32(peer_addr(&s.hm[2][b], r0 + r));
      }
    }
    part_c[t] = c;
    part_m[t] = weighted ? (u64)m0 + ((u64)m1 << 14) + ((u64)m2 << 28) : (u64)c;
  }
  __syncthreads();
  // exclusive prefix over this range's bins (warp scans, then warp totals)
  __shared__ uint32_t wtot_c[kR / 32];
  __shared__ u64 wtot_m[kR / 32];
  uint32_t c = 0u, ic = 0u;
  u64 m = 0ull, im = 0ull;
  if (t < kR) {
    c = part_c[t] + part_c[t + kR];
    m = part_m[t] + part_m[t + kR];
    s.rc[t] = c;
    s.rm[t] = m;
    ic = c;
    im = m;
    const int l = t & 31;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t tc = __shfl_up_sync(0xffffffffu, ic, o);
      const u64 tm = __shfl_up_sync(0xffffffffu, im, o);
      if (l >= o) {
        ic += tc;
        im += tm;
      }
    }
    if (l == 31) {
      wtot_c[t >> 5] = ic;
      wtot_m[t >> 5] = im;
    }
  }
  __syncthreads();
  uint32_t tot_c = 0u;
  u64 tot_m = 0ull;
  for (int w = 0; w < kR / 32; ++w) {
    tot_c += wtot_c[w];
    tot_m += wtot_m[w];
  }
  uint32_t ex_c = ic - c;
  u64 ex_m = im - m;
  if (t < kR)
    for (int w = 0; w < (t >> 5); ++w) {
      ex_c += wtot_c[w];
      ex_m += wtot_m[w];
    }
  // range totals of all eight CTAs (and their S_fp parts), in rank order
  cluster_gather(s, slot++, (u64)tot_c, tot_m, norm ? *norm : 0ull);
  if (norm) {
    u64 sf = 0ull;
    for (int r = 0; r < kCl; ++r) sf += s.xin[r][2];
    *norm = sf;
    // prefix mass >= alpha S  <=>  prefix >= ceil(alpha S) in fixed point
    target = (u64)ceil(alpha * (double)sf);
  }
  u64 pre_m[kCl + 1];
  uint32_t pre_c[kCl + 1];
  pre_m[0] = 0ull;
  pre_c[0] = 0u;
  int owner = -1, last = -1;
  for (int r = 0; r < kCl; ++r) {
    pre_c[r + 1] = pre_c[r] + (uint32_t)s.xin[r][0];
    pre_m[r + 1] = pre_m[r] + s.xin[r][1];
    if (owner < 0 && pre_m[r] < target && target <= pre_m[r + 1] && s.xin[r][0] > 0ull) owner = r;
    if (s.xin[r][0] > 0ull) last = r;
  }
  __syncthreads();
  bool use_last = false;
  if (owner < 0) {
    if (!clamp || last < 0) {
      cluster_sync();  // peers finished reading this CTA's histogram (all return alike)
      return false;
    }
    owner = last;
    use_last = true;
  }
  if ((int)cx.rank == owner && t < kR) {
    const u64 wa = pre_m[owner] + ex_m;
    bool hit;
    if (use_last) {
      // the last non-empty bin of the range: no later bin has a count
      hit = c > 0u && ex_c + c == tot_c;
    } else {
      hit = c > 0u && wa < target && target <= wa + m;
    }
    if (hit) {
      s.res_q[0] = (u64)(owner * kR + t);
      s.res_q[1] = (u64)(pre_c[owner] + ex_c);
      s.res_q[2] = wa;
      s.res_q[3] = (u64)c;
    }
  }
  cluster_sync();
  if (t < 4) s.xin[t][0] = ld_peer_u64(peer_addr(&s.res_q[t], (uint32_t)owner));
  __syncthreads();
  bin = (int)s.xin[0][0];
  cnt_above = (uint32_t)s.xin[1][0];
  w_above = s.xin[2][0];
  cnt_bin = (uint32_t)s.xin[3][0];
  cluster_sync();  // every CTA read the owner's result; histograms may be rewritten
  return true;
}

// The n-th set element (1-based) in index order among this CTA's elements
// whose key equals `key` (array a), as a global index; the caller knows it is
// here.
__device__ uint32_t nth_tie(Sm& s, const Ctx& cx, const float* a, uint32_t key, uint32_t nth) {
  __shared__ uint32_t base_s, ans_s;
  if (threadIdx.x == 0) {
    base_s = 0u;
    ans_s = 0xffffffffu;
  }
  __syncthreads();
  for (int t0 = 0; t0 < cx.n; t0 += kT) {
    const int i = t0 + threadIdx.x;
    const bool hit = i < cx.n && fkey(a[i]) == key;
    const uint32_t bal = __ballot_sync(0xffffffffu, hit);
    const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
    if (l == 0) s.ru[w] = __popc(bal);
    __syncthreads();
    uint32_t before = base_s;
    for (int v = 0; v < w; ++v) before += s.ru[v];
    const uint32_t rank_in = before + __popc(bal & ((1u << l) - 1u)) + 1u;
    if (hit && rank_in == nth) ans_s = cx.i0 + (uint32_t)i;
    __syncthreads();
    if (threadIdx.x == 0) {
      uint32_t tot = 0u;
      for (int v = 0; v < kW; ++v) tot += s.ru[v];
      base_s += tot;
    }
    __syncthreads();
  }
  return ans_s;
}

// The elements i of this CTA's slice with hit(i), as packed (key(i), index)
// words, appended to rank 0's buf: compacted in this CTA's histogram area
// (free once a selection's bin is known), then one remote reservation on
// rank 0's fill count and parallel remote stores.  Rank 0's nbuf must be
// zero, and visible through a cluster barrier, before the call.
template <typename Hit, typename Key>
__device__ void gather_to_rank0(Sm& s, const Ctx& cx, const Hit& hit, const Key& key) {
  __shared__ uint32_t lcount, lbase;
  u64* loc = reinterpret_cast<u64*>(&s.hm[0][0]);  // 3 * kBins u32 >= kCap u64
  if (threadIdx.x == 0) lcount = 0u;
  __syncthreads();
  const int l = threadIdx.x & 31;
  for (int t0 = 0; t0 < cx.n; t0 += kT) {
    const int i = t0 + threadIdx.x;
    const bool h = i < cx.n && hit(i);
    const uint32_t bal = __ballot_sync(0xffffffffu, h);
    if (bal == 0u) continue;
    uint32_t base = 0u;
    if (l == 0) base = atomicAdd(&lcount, (uint32_t)__popc(bal));
    base = __shfl_sync(0xffffffffu, base, 0);
    if (h) {
      const uint32_t pos = base + __popc(bal & ((1u << l) - 1u));
      if (pos < (uint32_t)kCap) loc[pos] = pack(key(i), cx.i0 + (uint32_t)i);
    }
  }
  __syncthreads();
  const uint32_t n = min(lcount, (uint32_t)kCap);
  if (threadIdx.x == 0) lbase = n ? atom_add_peer(peer_addr(&s.nbuf, 0), n) : 0u;
  __syncthreads();
  for (uint32_t j = threadIdx.x; j < n; j += kT) {
    const uint32_t pos = lbase + j;
    if (pos < (uint32_t)kCap) st_peer_u64(peer_addr(&s.buf[pos], 0), loc[j]);
  }
}

__device__ void clear_hist(Sm& s) {
  for (int i = threadIdx.x; i < kBins; i += kT) {
    s.hc[i] = 0u;
    s.hm[0][i] = 0u;
    s.hm[1][i] = 0u;
    s.hm[2][i] = 0u;
  }
  __syncthreads();
}
// Count one element in bin b and (weighted) its mass term in three 14-bit
// chunks: each chunk's sum over a CTA stays below 2^28.
__device__ __forceinline__ u64 add_hist(Sm& s, int b, bool weighted, float z, float m) {
  atomicAdd(&s.hc[b], 1u);
  if (!weighted) return 0ull;
  const u64 q = fix40(expf(z - m));
  atomicAdd(&s.hm[0][b], (uint32_t)(q & 0x3fffu));
  atomicAdd(&s.hm[1][b], (uint32_t)((q >> 14) & 0x3fffu));
  atomicAdd(&s.hm[2][b], (uint32_t)(q >> 28));
  return q;
}

// Selection over array a (maximum m): the first element of the order at
// which the prefix weight reaches target.  `slot` counts exchange slots.
__device__ Pick select(Sm& s, const Ctx& cx, const float* a, float m, bool weighted,
                       u64 target, int& slot, u64* norm = nullptr, double alpha = 0.0) {
  Pick pk;
  pk.all = false;
  // ---- round 0: depth bins ----
  clear_hist(s);
  u64 part = 0ull;
  for (int i = threadIdx.x; i < cx.n; i += kT) {
    const float z = a[i];
    const float t = (m - z) * kDepthScale;
    const int b = t < (float)(kBins - 1) ? (int)t : kBins - 1;
    part += add_hist(s, b, weighted, z, m);
  }
  if (norm) *norm = block_sum_q(part, s);
  int bin;
  uint32_t cnt_above, n_set;
  u64 w_above;
  if (!boundary_bin(s, cx, weighted, target, slot, bin, cnt_above, w_above, n_set, false, norm,
                    alpha)) {
    pk.all = true;
    pk.key = 0u;
    pk.idx = 0xffffffffu;
    pk.len = 0u;
    return pk;
  }
  // the set: elements of the bin, then (if too large) narrower key ranges
  bool by_bin = true;
  uint32_t klo = 0u, khi = 0u;
  auto in_set = [&](float z) -> bool {
    if (by_bin) {
      const float t = (m - z) * kDepthScale;
      const int b = t < (float)(kBins - 1) ? (int)t : kBins - 1;
      return b == bin;
    }
    const uint32_t k = fkey(z);
    return k >= klo && k <= khi;
  };
  for (int round = 0; n_set > (uint32_t)kCap; ++round) {
    // key range of the set
    uint32_t lo = 0xffffffffu, hi = 0u;
    for (int i = threadIdx.x; i < cx.n; i += kT)
      if (in_set(a[i])) {
        const uint32_t k = fkey(a[i]);
        lo = min(lo, k);
        hi = max(hi, k);
      }
    lo = block_min_u(lo, s);
    hi = block_max_u(hi, s);
    cluster_red2_u(s, slot++, lo, hi, 1);
    klo = lo;
    khi = hi;
    by_bin = false;
    if (klo == khi || round >= 3) break;  // equal keys: ties
    // sub-bins of the key range, largest key first
    const unsigned long long span = (unsigned long long)(khi - klo) + 1ull;
    clear_hist(s);
    for (int i = threadIdx.x; i < cx.n; i += kT) {
      const uint32_t k = fkey(a[i]);
      if (k < klo || k > khi) continue;
      const int sb = (int)(((unsigned long long)(khi - k) * kBins) / span);
      add_hist(s, sb, weighted, a[i], m);
    }
    int sbin;
    uint32_t ca, cb;
    u64 wa;
    // (rounding can leave the narrowed set below the target: its last
    // non-empty sub-bin is taken)
    u64 rel = target - w_above;
    boundary_bin(s, cx, weighted, rel, slot, sbin, ca, wa, cb, true);
    cnt_above += ca;
    w_above += wa;
    n_set = cb;
    // the new set is the sub-bin's key range: [klo', khi'] from its keys
    const uint32_t olo = klo, ohi = khi;
    uint32_t lo2 = 0xffffffffu, hi2 = 0u;
    for (int i = threadIdx.x; i < cx.n; i += kT) {
      const uint32_t k = fkey(a[i]);
      if (k < olo || k > ohi) continue;
      const int sb = (int)(((unsigned long long)(ohi - k) * kBins) / span);
      if (sb == sbin) {
        lo2 = min(lo2, k);
        hi2 = max(hi2, k);
      }
    }
    lo2 = block_min_u(lo2, s);
    hi2 = block_max_u(hi2, s);
    cluster_red2_u(s, slot++, lo2, hi2, 1);
    klo = lo2;
    khi = hi2;
  }

  if (n_set > (uint32_t)kCap) {
    // all keys equal (klo == khi): the lowest indices come first
    const u64 wt = weighted ? fix40(expf(fval(klo) - m)) : 1ull;
    const u64 rest = target > w_above ? target - w_above : 0ull;
    const u64 need_q = wt == 0ull ? (u64)n_set : (rest + wt - 1ull) / wt;
    const uint32_t need = need_q < 1ull ? 1u : (need_q > (u64)n_set ? n_set : (uint32_t)need_q);
    // ties per CTA, in rank (index) order
    uint32_t mine = 0u;
    for (int i = threadIdx.x; i < cx.n; i += kT) mine += fkey(a[i]) == klo;
    mine = block_sum_u(mine, s);
    cluster_gather2(s, slot++, (u64)mine, 0ull);
    uint32_t before = 0u;
    for (uint32_t r = 0; r < cx.rank; ++r) before += (uint32_t)s.xin[r][0];
    __syncthreads();
    if (cluster_rank() == 0 && threadIdx.x == 0) s.res_u[0] = 0xffffffffu;
    cluster_sync();
    if (need > before && need <= before + mine) {
      const uint32_t gi = nth_tie(s, cx, a, klo, need - before);
      if (threadIdx.x == 0) st_peer_u32(peer_addr(&s.res_u[0], 0), gi);
    }
    cluster_sync();
    if (threadIdx.x == 0) s.xin[0][0] = ld_peer_u32(peer_addr(&s.res_u[0], 0));
    __syncthreads();
    pk.key = klo;
    pk.idx = (uint32_t)s.xin[0][0];
    pk.len = cnt_above + need;
    cluster_sync();  // everyone has read rank 0's result
    return pk;
  }

  // ---- gather the set into rank 0, sort, scan ----
  if (cx.rank == 0 && threadIdx.x == 0) s.nbuf = 0u;
  cluster_sync();
  gather_to_rank0(s, cx, [&](int i) { return in_set(a[i]); }, [&](int i) { return fkey(a[i]); });
  cluster_sync();
  if (cx.rank == 0) {
    const int n = (int)min(s.nbuf, (uint32_t)kCap);
    sort_desc(s, n);
    if (threadIdx.x < 32) {
      // first element whose prefix weight (above + own) reaches the target
      const int l = threadIdx.x;
      u64 run = w_above;
      int hit = -1;
      for (int j0 = 0; j0 < n && hit < 0; j0 += 32) {
        const int j = j0 + l;
        u64 w = 0ull;
        if (j < n) w = weighted ? fix40(expf(fval(pk_key(s.buf[j])) - m)) : 1ull;
        u64 inc = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const u64 t = __shfl_up_sync(0xffffffffu, inc, o);
          if (l >= o) inc += t;
        }
        const bool ok = j < n && run + inc >= target;
        const uint32_t bal = __ballot_sync(0xffffffffu, ok);
        if (bal) hit = j0 + __ffs(bal) - 1;
        run += __shfl_sync(0xffffffffu, inc, 31);
      }
      if (hit < 0) hit = n > 0 ? n - 1 : 0;  // rounding: the whole set
      if (l == 0) {
        s.res_u[0] = pk_key(s.buf[hit]);
        s.res_u[1] = pk_idx(s.buf[hit]);
        s.res_u[2] = cnt_above + (uint32_t)hit + 1u;
      }
    }
  }
  cluster_sync();
  if (threadIdx.x < 3) s.xin[threadIdx.x][0] = ld_peer_u32(peer_addr(&s.res_u[threadIdx.x], 0));
  __syncthreads();
  pk.key = (uint32_t)s.xin[0][0];
  pk.idx = (uint32_t)s.xin[1][0];
  pk.len = (uint32_t)s.xin[2][0];
  cluster_sync();  // everyone has read rank 0's result
  return pk;
}

__device__ __forceinline__ bool ranks_in(uint32_t k, uint32_t i, const Pick& p) {
  return p.all || k > p.key || (k == p.key && i <= p.idx);
}

__global__ void __cluster_dims__(kCl, 1, 1) __launch_bounds__(kT, 1)
    drift_kernel(const float* __restrict__ z_fp, const float* __restrict__ z_q, int vocab,
                 kvq_drift_params p, int32_t* __restrict__ m_t, float* __restrict__ c_t,
                 float* __restrict__ d_loc, uint8_t* __restrict__ y_t, float* __restrict__ cov) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  Sm& s = *reinterpret_cast<Sm*>(smem_raw);
  const int row = blockIdx.y;
  Ctx cx;
  cx.rank = cluster_rank();
  const int sl = ((vocab + kCl - 1) / kCl + 3) & ~3;
  cx.i0 = (uint32_t)(cx.rank * sl);
  cx.n = max(0, min(vocab - (int)cx.i0, sl));
  const float* gf = z_fp + (long long)row * vocab + cx.i0;
  const float* gq = z_q + (long long)row * vocab + cx.i0;
  int slot = 0;

  // ---- stage the slices (one HBM read) and the maxima ----
  float mf = -INFINITY, mq = -INFINITY;
  const bool vec = ((reinterpret_cast<uintptr_t>(gf) | reinterpret_cast<uintptr_t>(gq)) & 15u) == 0;
  if (vec) {
    const int n4 = cx.n >> 2;
    for (int i = threadIdx.x; i < n4; i += kT) {
      const float4 a = __ldg(reinterpret_cast<const float4*>(gf) + i);
      const float4 b = __ldg(reinterpret_cast<const float4*>(gq) + i);
      reinterpret_cast<float4*>(s.zf)[i] = a;
      reinterpret_cast<float4*>(s.zq)[i] = b;
      mf = fmaxf(mf, fmaxf(fmaxf(a.x, a.y), fmaxf(a.z, a.w)));
      mq = fmaxf(mq, fmaxf(fmaxf(b.x, b.y), fmaxf(b.z, b.w)));
    }
    for (int i = 4 * n4 + threadIdx.x; i < cx.n; i += kT) {
      s.zf[i] = gf[i];
      s.zq[i] = gq[i];
      mf = fmaxf(mf, s.zf[i]);
      mq = fmaxf(mq, s.zq[i]);
    }
  } else {
    for (int i = threadIdx.x; i < cx.n; i += kT) {
      s.zf[i] = gf[i];
      s.zq[i] = gq[i];
      mf = fmaxf(mf, s.zf[i]);
      mq = fmaxf(mq, s.zq[i]);
    }
  }
  mf = block_max_f(mf, s);
  mq = block_max_f(mq, s);
  {
    // maxima as order keys (max of keys = key of the max)
    uint32_t a = fkey(mf), b = fkey(mq);
    cluster_red2_u(s, slot++, a, b, 2);
    mf = fval(a);
    mq = fval(b);
  }

  // ---- C(alpha) (with S_fp) and TopK(z_q, k_max) boundaries ----
  u64 sf = 0ull;
  const Pick pf = select(s, cx, s.zf, mf, true, 0ull, slot, &sf, (double)p.alpha);
  const Pick pq = select(s, cx, s.zq, mq, false, (u64)p.k_max, slot);

  // ---- the k_max best of z_q, sorted, in rank 0 ----
  if (cx.rank == 0 && threadIdx.x == 0) s.nbuf = 0u;
  cluster_sync();
  gather_to_rank0(
      s, cx, [&](int i) { return ranks_in(fkey(s.zq[i]), cx.i0 + (uint32_t)i, pq); },
      [&](int i) { return fkey(s.zq[i]); });
  cluster_sync();
  if (cx.rank == 0) {
    sort_desc(s, (int)min(s.nbuf, (uint32_t)kCap));
    if (threadIdx.x == 0) {
      const unsigned long long w = s.buf[p.window - 1];  // the K-th of TopK(z_q)
      s.res_u[4] = pk_key(w);
      s.res_u[5] = pk_idx(w);
    }
  }
  cluster_sync();
  if (threadIdx.x < 2) s.xin[threadIdx.x][0] = ld_peer_u32(peer_addr(&s.res_u[4 + threadIdx.x], 0));
  __syncthreads();
  Pick ps;
  ps.all = false;
  ps.key = (uint32_t)s.xin[0][0];
  ps.idx = (uint32_t)s.xin[1][0];
  ps.len = (uint32_t)p.window;
  __syncthreads();

  // ---- one pass over U = C union S ----
  // masses A = e_fp(U), B = e_q(U), c = e_fp(C and S) in fixed point; the
  // sums of e_fp^2, e_fp e_q, e_q^2 in double-float for
  //   d_loc^2 = Saa / A^2 - 2 Sab / (A B) + Sbb / B^2.
  // U is sparse: each warp queues its members (local index, bit 31 = in C
  // and S) in its own 64 entries of buf past the TopK list and works on them
  // 32 at a time, so the exponentials and products run on full warps.
  u64 A = 0ull, B = 0ull, Cs = 0ull;
  Df saa, sab, sbb;
  {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    uint32_t* uq = reinterpret_cast<uint32_t*>(&s.buf[kMaxKcov]) + warp * 64;
    auto member = [&](uint32_t e) {
      const int i = (int)(e & 0x7fffffffu);
      const float a = expf(s.zf[i] - mf), b = expf(s.zq[i] - mq);
      const u64 qa = fix40(a);
      A += qa;
      B += fix40(b);
      if (e >> 31) Cs += qa;
      saa.add_prod(a, a);
      sab.add_prod(a, b);
      sbb.add_prod(b, b);
    };
    int qn = 0;
    for (int t0 = warp * 32; t0 < cx.n; t0 += kT) {
      const int i = t0 + lane;
      bool inc = false, ins = false;
      if (i < cx.n) {
        const uint32_t gi = cx.i0 + (uint32_t)i;
        inc = ranks_in(fkey(s.zf[i]), gi, pf);
        ins = ranks_in(fkey(s.zq[i]), gi, ps);
      }
      const bool mem = inc || ins;
      const uint32_t bal = __ballot_sync(0xffffffffu, mem);
      if (mem) uq[qn + __popc(bal & ((1u << lane) - 1u))] = (uint32_t)i | (inc && ins ? 0x80000000u : 0u);
      qn += __popc(bal);
      __syncwarp();
      if (qn >= 32) {
        member(uq[lane]);
        __syncwarp();
        if (lane < qn - 32) uq[lane] = uq[32 + lane];  // the rest (< 32) to the front
        qn -= 32;
        __syncwarp();
      }
    }
    if (lane < qn) member(uq[lane]);
  }
  // per-warp sums (a fixed pairing order), then thread 0 adds the warps
  {
#pragma unroll
    for (int o = 16; o; o >>= 1) {
      A += __shfl_xor_sync(0xffffffffu, A, o);
      B += __shfl_xor_sync(0xffffffffu, B, o);
      Cs += __shfl_xor_sync(0xffffffffu, Cs, o);
      Df* acc[3] = {&saa, &sab, &sbb};
#pragma unroll
      for (int k = 0; k < 3; ++k) {
        Df w;
        w.hi = __shfl_xor_sync(0xffffffffu, acc[k]->hi, o);
        w.lo = __shfl_xor_sync(0xffffffffu, acc[k]->lo, o);
        if ((threadIdx.x & o) == 0) {
          acc[k]->add(w);
        } else {
          w.add(*acc[k]);
          *acc[k] = w;
        }
      }
    }
    u64* wpart = reinterpret_cast<u64*>(s.wsel);  // [kW][6] (wsel is free until the outputs)
    if ((threadIdx.x & 31) == 0) {
      u64* w = wpart + (threadIdx.x >> 5) * 6;
      w[0] = A;
      w[1] = B;
      w[2] = Cs;
      w[3] = saa.pack();
      w[4] = sab.pack();
      w[5] = sbb.pack();
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      A = B = Cs = 0ull;
      Df ta, tb, tc;
      for (int w = 0; w < kW; ++w) {
        A += wpart[w * 6];
        B += wpart[w * 6 + 1];
        Cs += wpart[w * 6 + 2];
        ta.add(Df::unpack(wpart[w * 6 + 3]));
        tb.add(Df::unpack(wpart[w * 6 + 4]));
        tc.add(Df::unpack(wpart[w * 6 + 5]));
      }
      saa = ta;
      sab = tb;
      sbb = tc;
    }
    __syncthreads();
  }
  // one exchange of the six CTA totals (thread 0's values are published)
  cluster_gather2x(s, slot, A, B, Cs, saa.pack(), sab.pack(), sbb.pack());
  slot += 2;
  u64 c_sum = 0ull;
  double Dsum = 0.0;
  if (threadIdx.x == 0) {
    A = B = 0ull;
    Df taa, tab, tbb;
    for (int r = 0; r < kCl; ++r) {
      A += s.xin8[r][0];
      B += s.xin8[r][1];
      c_sum += s.xin8[r][2];
      taa.add(Df::unpack(s.xin8[r][3]));
      tab.add(Df::unpack(s.xin8[r][4]));
      tbb.add(Df::unpack(s.xin8[r][5]));
    }
    const double ia = kFix / (double)A, ib = kFix / (double)B;
    Dsum = taa.value() * ia * ia - 2.0 * tab.value() * ia * ib + tbb.value() * ib * ib;
    if (Dsum < 0.0) Dsum = 0.0;  // rounding of an exact zero
  }

  // ---- outputs (rank 0) ----
  if (cx.rank == 0) {
    if (threadIdx.x == 0) {
      const double c = (double)c_sum / (double)sf;
      const double d = sqrt(Dsum);
      m_t[row] = pf.all ? vocab : (int32_t)pf.len;
      c_t[row] = (float)c;
      d_loc[row] = (float)d;
      y_t[row] = (uint8_t)(d > (double)p.eps && c >= (double)p.rho_c);
    }
    // coverage curve: prefix sums of p_fp over TopK(z_q, k) within C; the
    // FP16 logits of the list come from the CTAs that hold them
    const int sl = ((vocab + kCl - 1) / kCl + 3) & ~3;
    if (threadIdx.x < p.k_max) {
      const uint32_t gi = pk_idx(s.buf[threadIdx.x]);
      u64 w = 0ull;
      if (gi < (uint32_t)vocab) {
        const uint32_t owner = gi / (uint32_t)sl;
        const float zf = ld_peer_f32(peer_addr(&s.zf[gi - owner * (uint32_t)sl], owner));
        if (ranks_in(fkey(zf), gi, pf)) w = fix40(expf(zf - mf));
      }
      s.wsel[threadIdx.x] = w;
    }
    if (threadIdx.x == 0) s.bc[2] = (float)(1.0 / (double)sf);
    __syncthreads();
    if (threadIdx.x < 32) {
      const int l = threadIdx.x;
      const float inv = s.bc[2];
      u64 run = 0ull;
      for (int j0 = 0; j0 < p.k_max; j0 += 32) {
        const int j = j0 + l;
        u64 inc = j < p.k_max ? s.wsel[j] : 0ull;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const u64 t = __shfl_up_sync(0xffffffffu, inc, o);
          if (l >= o) inc += t;
        }
        if (j < p.k_max) cov[(long long)row * p.k_max + j] = (float)(run + inc) * inv;
        run += __shfl_sync(0xffffffffu, inc, 31);
      }
    }
  }
  cluster_sync();  // no CTA leaves while a peer may read its shared memory
}

// K_b: column means of cov over the rows (fixed order, fp64) and the smallest
// k whose mean reaches rho_K (0 if none).
__global__ void __launch_bounds__(256) drift_window_kernel(const float* __restrict__ cov, int rows,
                                                           int k_max, float rho_k,
                                                           float* __restrict__ mean_cov,
                                                           int32_t* __restrict__ k_b) {
  __shared__ int best[8];
  int mine = 0x7fffffff;
  for (int k = threadIdx.x; k < k_max; k += blockDim.x) {
    double sum = 0.0;
    for (int r = 0; r < rows; ++r) sum += (double)cov[(long long)r * k_max + k];
    const double mean = sum / rows;
    mean_cov[k] = (float)mean;
    if (mean >= (double)rho_k) mine = min(mine, k + 1);
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) mine = min(mine, __shfl_xor_sync(0xffffffffu, mine, o));
  if ((threadIdx.x & 31) == 0) best[threadIdx.x >> 5] = mine;
  __syncthreads();
  if (threadIdx.x == 0) {
    int b = 0x7fffffff;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) b = min(b, best[w]);
    *k_b = b == 0x7fffffff ? 0 : b;
  }
}

}  // namespace

int drift_max_vocab() { return kCl * kSlice; }
int drift_max_kcov() { return kMaxKcov; }
int drift_cap() { return kCap; }

cudaError_t launch_drift(const float* z_fp, const float* z_q, int rows, int vocab,
                         const kvq_drift_params& p, int32_t* m_t, float* c_t, float* d_loc,
                         uint8_t* y_t, float* cov, cudaStream_t st) {
  const size_t smem = sizeof(Sm);
  cudaError_t e = cudaFuncSetAttribute(drift_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  drift_kernel<<<dim3(kCl, rows), kT, smem, st>>>(z_fp, z_q, vocab, p, m_t, c_t, d_loc, y_t, cov);
  return cudaGetLastError();
}

cudaError_t launch_drift_window(const float* cov, int rows, int k_max, float rho_k,
                                float* mean_cov, int32_t* k_b, cudaStream_t st) {
  drift_window_kernel<<<1, 256, 0, st>>>(cov, rows, k_max, rho_k, mean_cov, k_b);
  return cudaGetLastError();
}

}  // namespace kvq
