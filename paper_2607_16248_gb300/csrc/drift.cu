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
//   1. maxima, then the FP16 normaliser S_fp = sum e^{z - m} (fp64);
//   2. the FP16 boundary: a 2048-bin histogram of the depth (m - z) * 64
//      (count and mass per bin, the depth order is the FP16 order) finds the
//      bin where the prefix mass reaches alpha S_fp; that bin's elements are
//      sorted in one CTA and scanned for the exact element.  A bin with more
//      than 2048 elements is narrowed by histograms of its key range first;
//      a range of equal keys takes the lowest indices (counted per CTA in
//      index order);
//   3. the same selection by count on z_q gives the k_max-th element, then
//      the k_max best elements are gathered and sorted (the TopK order);
//   4. the sums over U (fp64), then d_loc from the renormalised vectors.
// Weights are e = expf(z - m) in fp32 everywhere, summed in fp64, so every
// decision between two elements uses the same numbers.

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
constexpr int kSlots = 64;           // exchange slots (one per cluster reduction)

struct Sm {
  float zf[kSlice];
  float zq[kSlice];
  uint32_t hc[kBins];
  float hm[kBins];
  unsigned long long buf[kCap];     // rank 0: boundary set / TopK set
  double xd[kSlots][2];             // per-CTA partials read by the peers
  uint32_t xu[kSlots][2];
  double res_d[4];                  // rank 0: results of a selection
  uint32_t res_u[8];
  uint32_t nbuf;                    // rank 0: fill count of buf
  double rd[kW];
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
__device__ __forceinline__ double ld_peer_f64(uint32_t a) {
  double v;
  asm volatile("ld.shared::cluster.f64 %0, [%1];" : "=d"(v) : "r"(a) : "memory");
  return v;
}
__device__ __forceinline__ float ld_peer_f32(uint32_t a) {
  float v;
  asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(a) : "memory");
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
__device__ double block_sum_d(double v, Sm& s) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  __syncthreads();
  if ((threadIdx.x & 31) == 0) s.rd[threadIdx.x >> 5] = v;
  __syncthreads();
  double r = 0.0;
  for (int w = 0; w < kW; ++w) r += s.rd[w];  // fixed order
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
__device__ void cluster_sum2_d(Sm& s, int slot, double& a, double& b) {
  if (threadIdx.x == 0) {
    s.xd[slot][0] = a;
    s.xd[slot][1] = b;
  }
  cluster_sync();
  double ra = 0.0, rb = 0.0;
  for (uint32_t r = 0; r < kCl; ++r) {
    ra += ld_peer_f64(peer_addr(&s.xd[slot][0], r));
    rb += ld_peer_f64(peer_addr(&s.xd[slot][1], r));
  }
  a = ra;
  b = rb;
}
// op 0: (sum, sum); op 1: (min, max); op 2: (max, max) on float bits >= 0
__device__ void cluster_red2_u(Sm& s, int slot, uint32_t& a, uint32_t& b, int op) {
  if (threadIdx.x == 0) {
    s.xu[slot][0] = a;
    s.xu[slot][1] = b;
  }
  cluster_sync();
  uint32_t ra = op == 1 ? 0xffffffffu : 0u, rb = 0u;
  for (uint32_t r = 0; r < kCl; ++r) {
    const uint32_t x = ld_peer_u32(peer_addr(&s.xu[slot][0], r));
    const uint32_t y = ld_peer_u32(peer_addr(&s.xu[slot][1], r));
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

// Weight of a logit in a selection: its FP16 mass term (weighted) or 1.
__device__ __forceinline__ float weight(float z, float m, bool weighted) {
  return weighted ? expf(z - m) : 1.0f;
}

// Result of a selection: the element (key, index) at which the prefix of
// the order (key descending, index ascending) first reaches the target, and
// the prefix length.  all = the target is never reached (everything).
struct Pick {
  uint32_t key, idx, len;
  bool all;
};

// Exclusive prefix over the histogram in bin order (bin 0 ranks first) of
// the cluster-wide counts / masses; finds the bin where the prefix weight
// reaches `target` (count or mass).  Histograms of all CTAs are reduced in
// rank order.  If the total stays below the target: with `clamp` the last
// non-empty bin is taken, else false is returned.
__device__ bool boundary_bin(Sm& s, bool weighted, double target, int& bin, uint32_t& cnt_above,
                             double& w_above, uint32_t& cnt_bin, bool clamp = false) {
  cluster_sync();  // every CTA's histogram is complete
  const int b0 = threadIdx.x * (kBins / kT);
  uint32_t c[kBins / kT];
  double m[kBins / kT];
  uint32_t csum = 0u;
  double msum = 0.0;
#pragma unroll
  for (int j = 0; j < kBins / kT; ++j) {
    c[j] = 0u;
    m[j] = 0.0;
    for (uint32_t r = 0; r < kCl; ++r) {
      c[j] += ld_peer_u32(peer_addr(&s.hc[b0 + j], r));
      if (weighted) m[j] += (double)ld_peer_f32(peer_addr(&s.hm[b0 + j], r));
    }
    if (!weighted) m[j] = (double)c[j];
    csum += c[j];
    msum += m[j];
  }
  // block exclusive scan of (csum, msum) over threads, in thread order
  __shared__ double sc_m[kT];
  __shared__ uint32_t sc_c[kT];
  __shared__ int found_bin, last_bin;
  __shared__ uint32_t found_ca, found_cb;
  __shared__ double found_wa;
  sc_m[threadIdx.x] = msum;
  sc_c[threadIdx.x] = csum;
  if (threadIdx.x == 0) {
    found_bin = -1;
    last_bin = -1;
  }
  __syncthreads();
  for (int o = 1; o < kT; o <<= 1) {
    const double tm = threadIdx.x >= o ? sc_m[threadIdx.x - o] : 0.0;
    const uint32_t tc = threadIdx.x >= o ? sc_c[threadIdx.x - o] : 0u;
    __syncthreads();
    sc_m[threadIdx.x] += tm;
    sc_c[threadIdx.x] += tc;
    __syncthreads();
  }
  const double wa0 = sc_m[threadIdx.x] - msum;  // exclusive prefix of this thread
  const uint32_t ca0 = sc_c[threadIdx.x] - csum;
  double wa = wa0;
  uint32_t ca = ca0;
  int last = -1;
#pragma unroll
  for (int j = 0; j < kBins / kT; ++j) {
    if (wa < target && target <= wa + m[j] && c[j] > 0u) {
      found_bin = b0 + j;
      found_wa = wa;
      found_ca = ca;
      found_cb = c[j];
    }
    if (c[j] > 0u) last = b0 + j;
    wa += m[j];
    ca += c[j];
  }
  if (last >= 0) atomicMax(&last_bin, last);
  __syncthreads();
  if (clamp && found_bin < 0 && last_bin >= b0 && last_bin < b0 + kBins / kT) {
    // the last non-empty bin: everything before it ranks above
    wa = wa0;
    ca = ca0;
    for (int j = 0; j < kBins / kT; ++j) {
      if (b0 + j == last_bin) {
        found_bin = last_bin;
        found_wa = wa;
        found_ca = ca;
        found_cb = c[j];
      }
      wa += m[j];
      ca += c[j];
    }
  }
  cluster_sync();  // peers finished reading this CTA's histogram
  __syncthreads();
  bin = found_bin;
  if (bin < 0) return false;
  cnt_above = found_ca;
  w_above = found_wa;
  cnt_bin = found_cb;
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

// Selection over array a (maximum m): the first element of the order at
// which the prefix weight reaches target.  `slot` counts exchange slots.
__device__ Pick select(Sm& s, const Ctx& cx, const float* a, float m, bool weighted,
                       double target, int& slot) {
  Pick pk;
  pk.all = false;
  // ---- round 0: depth bins ----
  for (int i = threadIdx.x; i < kBins; i += kT) {
    s.hc[i] = 0u;
    s.hm[i] = 0.0f;
  }
  __syncthreads();
  for (int i = threadIdx.x; i < cx.n; i += kT) {
    const float z = a[i];
    const float t = (m - z) * kDepthScale;
    const int b = t < (float)(kBins - 1) ? (int)t : kBins - 1;
    atomicAdd(&s.hc[b], 1u);
    if (weighted) atomicAdd(&s.hm[b], weight(z, m, true));
  }
  int bin;
  uint32_t cnt_above, n_set;
  double w_above;
  if (!boundary_bin(s, weighted, target, bin, cnt_above, w_above, n_set)) {
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
    for (int i = threadIdx.x; i < kBins; i += kT) {
      s.hc[i] = 0u;
      s.hm[i] = 0.0f;
    }
    __syncthreads();
    for (int i = threadIdx.x; i < cx.n; i += kT) {
      const uint32_t k = fkey(a[i]);
      if (k < klo || k > khi) continue;
      const int sb = (int)(((unsigned long long)(khi - k) * kBins) / span);
      atomicAdd(&s.hc[sb], 1u);
      if (weighted) atomicAdd(&s.hm[sb], weight(a[i], m, true));
    }
    int sbin;
    uint32_t ca, cb;
    double wa;
    // (rounding can leave the narrowed set below the target: its last
    // non-empty sub-bin is taken)
    boundary_bin(s, weighted, target - w_above, sbin, ca, wa, cb, true);
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
    const float zt = fval(klo);
    const double wt = (double)weight(zt, m, weighted);
    double need_d = weighted ? ceil((target - w_above) / wt) : (target - w_above);
    uint32_t need = need_d < 1.0 ? 1u : (need_d > (double)n_set ? n_set : (uint32_t)need_d);
    // ties per CTA, in rank (index) order
    uint32_t mine = 0u;
    for (int i = threadIdx.x; i < cx.n; i += kT) mine += fkey(a[i]) == klo;
    mine = block_sum_u(mine, s);
    if (threadIdx.x == 0) s.xu[slot][0] = mine;
    cluster_sync();
    uint32_t before = 0u;
    for (uint32_t r = 0; r < cx.rank; ++r) before += ld_peer_u32(peer_addr(&s.xu[slot][0], r));
    ++slot;
    if (cluster_rank() == 0 && threadIdx.x == 0) s.res_u[0] = 0xffffffffu;
    cluster_sync();
    if (need > before && need <= before + mine) {
      const uint32_t gi = nth_tie(s, cx, a, klo, need - before);
      if (threadIdx.x == 0) st_peer_u32(peer_addr(&s.res_u[0], 0), gi);
    }
    cluster_sync();
    pk.key = klo;
    pk.idx = ld_peer_u32(peer_addr(&s.res_u[0], 0));
    pk.len = cnt_above + need;
    cluster_sync();  // everyone has read rank 0's result
    return pk;
  }

  // ---- gather the set into rank 0, sort, scan ----
  if (cx.rank == 0 && threadIdx.x == 0) s.nbuf = 0u;
  cluster_sync();
  const uint32_t nb0 = peer_addr(&s.nbuf, 0);
  for (int t0 = 0; t0 < cx.n; t0 += kT) {
    const int i = t0 + threadIdx.x;
    const bool hit = i < cx.n && in_set(a[i]);
    const uint32_t bal = __ballot_sync(0xffffffffu, hit);
    if (bal == 0u) continue;
    const int l = threadIdx.x & 31;
    uint32_t base = 0u;
    if (l == 0) base = atom_add_peer(nb0, __popc(bal));
    base = __shfl_sync(0xffffffffu, base, 0);
    if (hit) {
      const uint32_t pos = base + __popc(bal & ((1u << l) - 1u));
      if (pos < (uint32_t)kCap)
        st_peer_u64(peer_addr(&s.buf[pos], 0), pack(fkey(a[i]), cx.i0 + (uint32_t)i));
    }
  }
  cluster_sync();
  if (cx.rank == 0) {
    const int n = (int)min(s.nbuf, (uint32_t)kCap);
    sort_desc(s, n);
    if (threadIdx.x < 32) {
      // first element whose prefix weight (above + own) reaches the target
      const int l = threadIdx.x;
      double run = w_above;
      int hit = -1;
      for (int j0 = 0; j0 < n && hit < 0; j0 += 32) {
        const int j = j0 + l;
        double w = 0.0;
        if (j < n) w = (double)weight(fval(pk_key(s.buf[j])), m, weighted);
        double inc = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const double t = __shfl_up_sync(0xffffffffu, inc, o);
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
  pk.key = ld_peer_u32(peer_addr(&s.res_u[0], 0));
  pk.idx = ld_peer_u32(peer_addr(&s.res_u[1], 0));
  pk.len = ld_peer_u32(peer_addr(&s.res_u[2], 0));
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

  // ---- FP16 normaliser ----
  double sf = 0.0, dummy = 0.0;
  for (int i = threadIdx.x; i < cx.n; i += kT) sf += (double)expf(s.zf[i] - mf);
  sf = block_sum_d(sf, s);
  cluster_sum2_d(s, slot++, sf, dummy);

  // ---- C(alpha) and TopK(z_q, k_max) boundaries ----
  const Pick pf = select(s, cx, s.zf, mf, true, (double)p.alpha * sf, slot);
  const Pick pq = select(s, cx, s.zq, mq, false, (double)p.k_max, slot);

  // ---- the k_max best of z_q, sorted, in rank 0 ----
  if (cx.rank == 0 && threadIdx.x == 0) s.nbuf = 0u;
  cluster_sync();
  {
    const uint32_t nb0 = peer_addr(&s.nbuf, 0);
    for (int t0 = 0; t0 < cx.n; t0 += kT) {
      const int i = t0 + threadIdx.x;
      const bool hit = i < cx.n && ranks_in(fkey(s.zq[i]), cx.i0 + (uint32_t)i, pq);
      const uint32_t bal = __ballot_sync(0xffffffffu, hit);
      if (bal == 0u) continue;
      const int l = threadIdx.x & 31;
      uint32_t base = 0u;
      if (l == 0) base = atom_add_peer(nb0, __popc(bal));
      base = __shfl_sync(0xffffffffu, base, 0);
      if (hit) {
        const uint32_t pos = base + __popc(bal & ((1u << l) - 1u));
        if (pos < (uint32_t)kCap)
          st_peer_u64(peer_addr(&s.buf[pos], 0), pack(fkey(s.zq[i]), cx.i0 + (uint32_t)i));
      }
    }
  }
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
  Pick ps;
  ps.all = false;
  ps.key = ld_peer_u32(peer_addr(&s.res_u[4], 0));
  ps.idx = ld_peer_u32(peer_addr(&s.res_u[5], 0));
  ps.len = (uint32_t)p.window;

  // ---- sums over U = C union S ----
  double A = 0.0, B = 0.0, Cs = 0.0;
  for (int i = threadIdx.x; i < cx.n; i += kT) {
    const uint32_t gi = cx.i0 + (uint32_t)i;
    const bool inc = ranks_in(fkey(s.zf[i]), gi, pf);
    const bool ins = ranks_in(fkey(s.zq[i]), gi, ps);
    if (inc || ins) {
      const double ef = (double)expf(s.zf[i] - mf);
      A += ef;
      B += (double)expf(s.zq[i] - mq);
      if (inc && ins) Cs += ef;
    }
  }
  A = block_sum_d(A, s);
  B = block_sum_d(B, s);
  Cs = block_sum_d(Cs, s);
  cluster_sum2_d(s, slot++, A, B);
  double c_sum = Cs;
  cluster_sum2_d(s, slot++, c_sum, dummy);
  double D = 0.0;
  for (int i = threadIdx.x; i < cx.n; i += kT) {
    const uint32_t gi = cx.i0 + (uint32_t)i;
    if (ranks_in(fkey(s.zf[i]), gi, pf) || ranks_in(fkey(s.zq[i]), gi, ps)) {
      const double d = (double)expf(s.zf[i] - mf) / A - (double)expf(s.zq[i] - mq) / B;
      D += d * d;
    }
  }
  D = block_sum_d(D, s);
  cluster_sum2_d(s, slot++, D, dummy);

  // ---- outputs (rank 0) ----
  if (cx.rank == 0) {
    const double c = c_sum / sf;
    const double d = sqrt(D);
    if (threadIdx.x == 0) {
      m_t[row] = pf.all ? vocab : (int32_t)pf.len;
      c_t[row] = (float)c;
      d_loc[row] = (float)d;
      y_t[row] = (uint8_t)(d > (double)p.eps && c >= (double)p.rho_c);
    }
    if (threadIdx.x < 32) {
      // coverage curve: prefix sums of p_fp over TopK(z_q, k) within C
      const int l = threadIdx.x;
      double run = 0.0;
      for (int j0 = 0; j0 < p.k_max; j0 += 32) {
        const int j = j0 + l;
        double w = 0.0;
        if (j < p.k_max) {
          const uint32_t gi = pk_idx(s.buf[j]);
          if (gi < (uint32_t)vocab) {
            const float zf = z_fp[(long long)row * vocab + gi];
            if (ranks_in(fkey(zf), gi, pf)) w = (double)expf(zf - mf);
          }
        }
        double inc = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const double t = __shfl_up_sync(0xffffffffu, inc, o);
          if (l >= o) inc += t;
        }
        if (j < p.k_max) cov[(long long)row * p.k_max + j] = (float)((run + inc) / sf);
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
