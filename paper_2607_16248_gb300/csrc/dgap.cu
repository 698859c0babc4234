// dgap_restore: the DGAP local-distribution-restoration epilogue
// (Sec. 4.1-4.3 of the paper) on one decode step's logits [batch][vocab].
//
// One launch, grid (n_chunks, batch), 256 threads.  Each CTA scans a 4096-logit
// chunk of one row once: running max m, S1 = sum e^{z-m}, S2 = sum (z-m) e^{z-m}
// and the chunk's K+1 best (value descending, index ascending) candidates.
// The last CTA of a row to finish (atomic ticket, no waiting) merges the
// chunks, forms the window S = TopK(z, K) and z_(K), the features phi,
// runs the detector r = sigmoid(f) (Eq. 6), and when f > logit(tau) the
// candidate features xi, the corrector Delta = g(xi, phi) (Eq. 12) and the
// sparse merge z[S_k] += Delta_k in place (Eq. 13).  Non-selected logits and
// ungated rows are never written.
//
// The last CTA is latency-bound: every global read it makes is issued in one
// round (chunk statistics and candidate lists into shared memory, the
// corrector's first-layer weights by one bulk copy started as soon as the CTA
// knows it is last, so the copy overlaps the merge and the detector).
//
// Candidates are ranked by an order-preserving uint32 key of the float
// (-0 folded onto +0) and then by the lower index.

#include <limits.h>
#include <stddef.h>

#include "common.cuh"

namespace kvq {
namespace {

constexpr int kT = 256;
constexpr int kWarpsD = kT / 32;
constexpr int kPer = 16;
constexpr int kChunk = kT * kPer;
constexpr int kMaxChunks = kT;  // one candidate list per finalize thread
constexpr int kMaxIn = 5 * kMaxK + 8;  // corrector input width

struct DWs {
  float4* stats;   // [B][n_chunks] (m, S1, S2, -)
  uint2* cand;     // [B][n_chunks][K+1] (key, index)
  unsigned* tk;    // [B]
};

__host__ __device__ inline size_t a256(size_t x) { return (x + 255) / 256 * 256; }

__host__ __device__ inline DWs carve(void* base, int batch, int n_chunks, int K) {
  DWs w;
  char* p = static_cast<char*>(base);
  w.stats = reinterpret_cast<float4*>(p);
  p += a256((size_t)batch * n_chunks * sizeof(float4));
  w.cand = reinterpret_cast<uint2*>(p);
  p += a256((size_t)batch * n_chunks * (K + 1) * sizeof(uint2));
  w.tk = reinterpret_cast<unsigned*>(p);
  return w;
}

__device__ __forceinline__ uint32_t order_key(float x) {
  uint32_t u = __float_as_uint(x);
  if ((u << 1) == 0u) u = 0u;  // -0 ranks with +0
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float key_value(uint32_t k) {
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7fffffffu) : ~k);
}
// (ka, ia) ranks before (kb, ib)?
__device__ __forceinline__ bool before(uint32_t ka, int ia, uint32_t kb, int ib) {
  return ka > kb || (ka == kb && ia < ib);
}

__device__ __forceinline__ float wsum(float v) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float wmax(float v) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// Block-wide reductions over 256 threads (all threads get the result).
__device__ float block_sum(float v, float* red) {
  v = wsum(v);
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  __syncthreads();
  if (l == 0) red[w] = v;
  __syncthreads();
  float r = l < kWarpsD ? red[l] : 0.0f;
  return wsum(r);
}
__device__ float block_max(float v, float* red) {
  v = wmax(v);
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  __syncthreads();
  if (l == 0) red[w] = v;
  __syncthreads();
  float r = l < kWarpsD ? red[l] : -INFINITY;
  return wmax(r);
}

// ---------------------------------------------------------------------------
// Block-wide top-n selection (256 threads).  Keys are order-preserving uint32
// (larger is better; 0 marks padding); ties rank by the lower index.
// ---------------------------------------------------------------------------

struct Sel {
  unsigned hist[kT];   // one 8-bit digit's histogram
  unsigned digit;      // the digit holding the n-th element
  unsigned above;      // elements in higher digits
  unsigned at;         // elements in that digit
  unsigned pos;        // collection counter
};

// Key of the n-th largest key among the elements i < N with act(i) (which
// must number at least n), and how many elements with that key belong to the
// n largest: four passes of an 8-bit radix histogram, most significant first.
template <typename KeyF, typename ActF>
__device__ void radix_nth(int N, int n, const KeyF& key, const ActF& act, Sel& ss, uint32_t& T,
                          int& need, int& n_at) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  uint32_t prefix = 0u, mask = 0u;
  unsigned rem = (unsigned)n;
  for (int shift = 24; shift >= 0; shift -= 8) {
    ss.hist[tid] = 0u;
    __syncthreads();
    for (int i = tid; i < N; i += kT) {
      if (!act(i)) continue;
      const uint32_t k = key(i);
      if ((k & mask) == prefix) atomicAdd(&ss.hist[(k >> shift) & 255u], 1u);
    }
    __syncthreads();
    if (warp == 0) {
      // lane l takes digits 255 - 8 l .. 248 - 8 l, largest first
      unsigned c[8], sum = 0u;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        c[j] = ss.hist[255 - 8 * lane - j];
        sum += c[j];
      }
      unsigned inc = sum;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const unsigned t = __shfl_up_sync(0xffffffffu, inc, o);
        if (lane >= o) inc += t;
      }
      unsigned acc = inc - sum;
      if (acc < rem && rem <= inc) {
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          if (acc < rem && rem <= acc + c[j]) {
            ss.digit = 255u - 8u * lane - j;
            ss.above = acc;
            ss.at = c[j];
          }
          acc += c[j];
        }
      }
    }
    __syncthreads();
    prefix |= ss.digit << shift;
    mask |= 255u << shift;
    rem -= ss.above;
    n_at = (int)ss.at;
  }
  T = prefix;
  need = (int)rem;
}

// The n best of N elements (get(i, key, index)), sorted best first into
// ok / oi; tk / ti hold n entries of scratch.
template <typename GetF>
__device__ void block_select(int N, int n, const GetF& get, Sel& ss, uint32_t* ok, int* oi,
                             uint32_t* tk, int* ti) {
  const int tid = threadIdx.x;
  uint32_t T;
  int need, n_at;
  radix_nth(N, n, [&](int i) { uint32_t k; int x; get(i, k, x); return k; },
            [](int) { return true; }, ss, T, need, n_at);
  // Ties at T: the `need` lowest indices (largest ~index), unless all are taken.
  uint32_t TI = 0u;
  if (need < n_at) {
    int need2, n_at2;
    radix_nth(N, need, [&](int i) { uint32_t k; int x; get(i, k, x); return ~(uint32_t)x; },
              [&](int i) { uint32_t k; int x; get(i, k, x); return k == T; }, ss, TI, need2,
              n_at2);
  }
  if (tid == 0) ss.pos = 0u;
  __syncthreads();
  const int lane = tid & 31;
  for (int b0 = 0; b0 < N; b0 += kT) {
    const int i = b0 + tid;
    uint32_t k = 0u;
    int x = 0;
    bool take = false;
    if (i < N) {
      get(i, k, x);
      take = k > T || (k == T && ~(uint32_t)x >= TI);
    }
    const unsigned m = __ballot_sync(0xffffffffu, take);
    if (m) {
      unsigned p0 = 0u;
      if (lane == __ffs(m) - 1) p0 = atomicAdd(&ss.pos, (unsigned)__popc(m));
      p0 = __shfl_sync(0xffffffffu, p0, __ffs(m) - 1);
      const unsigned p = p0 + __popc(m & ((1u << lane) - 1u));
      if (take && p < (unsigned)n) {
        tk[p] = k;
        ti[p] = x;
      }
    }
  }
  __syncthreads();
  if (tid < n) {  // rank sort (duplicates only among padding entries)
    const uint32_t k = tk[tid];
    const int x = ti[tid];
    int r = 0;
    for (int j = 0; j < n; ++j)
      r += before(tk[j], ti[j], k, x) || (tk[j] == k && ti[j] == x && j < tid);
    ok[r] = k;
    oi[r] = x;
  }
  __syncthreads();
}

// Largest key of lane rank q - 1 in the warp (keys sorted descending across
// lanes by a bitonic network of shuffles).
__device__ __forceinline__ uint32_t warp_kth_key(uint32_t k, int q) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int size = 2; size <= 32; size <<= 1)
#pragma unroll
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      const uint32_t o = __shfl_xor_sync(0xffffffffu, k, stride);
      const bool lower = (lane & stride) == 0;          // keeps the larger when descending
      const bool desc = (lane & size) == 0 || size == 32;
      k = (lower == desc) ? max(k, o) : min(k, o);
    }
  return __shfl_sync(0xffffffffu, k, q - 1);
}

constexpr int kSurvivors = 1024;  // candidates kept for the exact ranking

// The n best of the elements held in registers whose key is at least T0, a
// lower bound on the n-th best key (so they contain the n best), sorted best
// first into ok / oi: packed into sv as (key, ~index) words, whose order is
// the ranking order, and ranked exactly.  With more than kSurvivors of them
// (heavy ties) every thread calls fallback() instead.
template <int E, typename Fallback>
__device__ void select_above(const uint32_t (&k)[E], const int (&x)[E], int n, uint32_t T0,
                             Sel& ss, unsigned long long* sv, uint32_t* ok, int* oi,
                             const Fallback& fallback) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  int c = 0;
#pragma unroll
  for (int i = 0; i < E; ++i) c += k[i] >= T0;
  int inc = c;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int t = __shfl_up_sync(0xffffffffu, inc, o);
    if (lane >= o) inc += t;
  }
  if (lane == 31) ss.hist[kWarpsD + warp] = (unsigned)inc;
  __syncthreads();
  int off = inc - c, S = 0;
#pragma unroll
  for (int w = 0; w < kWarpsD; ++w) {
    const int cw = (int)ss.hist[kWarpsD + w];
    off += w < warp ? cw : 0;
    S += cw;
  }
  if (S > kSurvivors) {
    __syncthreads();
    fallback();
    return;
  }
#pragma unroll
  for (int i = 0; i < E; ++i)
    if (k[i] >= T0) sv[off++] = ((unsigned long long)k[i] << 32) | (uint32_t)~x[i];
  __syncthreads();
  for (int t = tid; t < S; t += kT) {
    const unsigned long long me = sv[t];
    int r = 0;
#pragma unroll 8
    for (int j = 0; j < S; ++j) {
      const unsigned long long o = sv[j];
      r += (o > me) || (o == me && j < t);
    }
    if (r < n) {
      ok[r] = (uint32_t)(me >> 32);
      oi[r] = (int)~(uint32_t)me;
    }
  }
  __syncthreads();
}

// The n best (n <= 72) of the elements the CTA's threads hold in registers
// (E per thread; key 0 marks padding), sorted best first into ok / oi.
// Every warp's q = ceil(n / 8)-th largest per-thread maximum bounds the n-th
// best key from below (8 q >= n elements reach it); select_above does the
// rest.
template <int E, typename Fallback>
__device__ void select_top(const uint32_t (&k)[E], const int (&x)[E], int n, Sel& ss,
                           unsigned long long* sv, uint32_t* ok, int* oi,
                           const Fallback& fallback) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  uint32_t mk = 0u;
#pragma unroll
  for (int i = 0; i < E; ++i) mk = max(mk, k[i]);
  const uint32_t wq = warp_kth_key(mk, (n + kWarpsD - 1) / kWarpsD);
  if (lane == 0) ss.hist[warp] = wq;
  __syncthreads();
  uint32_t T0 = ss.hist[0];
#pragma unroll
  for (int w = 1; w < kWarpsD; ++w) T0 = min(T0, ss.hist[w]);
  select_above(k, x, n, T0, ss, sv, ok, oi, fallback);
}

constexpr int kCandReg = 16;                // candidates of a row per thread (finalize)
constexpr size_t kW1StageMax = 168 * 1024;  // largest staged corrector W1 (256 x 168)

// The union comes last: a launch that does not stage W1 (grids of more
// CTAs than SMs, where one ~190 KB CTA per SM would run in waves) stops the
// shared memory after its chunk-phase part (kSmemNoW1 bytes).
struct Smem {
  uint64_t w1_bar;
  Sel sel;
  unsigned long long sv[kSurvivors];    // select_top: candidates above the bound
  unsigned long long su[kMaxK + 1 + kMaxChunks];  // finalize: leaders of every list
  uint32_t t0;                          // finalize: lower bound on the window's keys
  uint32_t wk[kWarpsD][kMaxK + 1];
  int wi[kWarpsD][kMaxK + 1];
  uint32_t fk[kMaxK + 1];
  int fi[kMaxK + 1];
  float zt[kMaxK];
  alignas(16) float x[kMaxIn];
  float hb[kMaxHidden];
  float phi[8];
  float red[32];
  float f;
  int last;
  union alignas(16) {
    struct {
      uint32_t sk[kChunk];
      int si[kChunk];
    } srt;                              // chunk phase: the chunk's keys
    float w1[kW1StageMax / 4];          // finalize: corrector W1 (bulk copy)
  } u;
};
constexpr size_t kSmemNoW1 = offsetof(Smem, u) + sizeof(static_cast<Smem*>(nullptr)->u.srt);

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
// Whether the corrector's W1 is copied to shared memory in one bulk copy
// (decided by the host, passed to the kernel): when it fits and the grid
// runs in one wave of one CTA per SM.  Otherwise the finalizing CTA reads it
// through L1 (prefetched when the CTA learns it is last).
inline bool stage_w1(const DgapDims& d, const dgap_params& p, int sm_count) {
  const size_t bytes = (size_t)d.hidden * (5 * d.K + 8) * sizeof(float);
  return bytes <= kW1StageMax && bytes % 16 == 0 &&
         (reinterpret_cast<uintptr_t>(p.cor_w1) & 15) == 0 &&
         (long long)d.n_chunks * d.batch <= sm_count;
}

__device__ void finalize_row(const DgapDims& d, const dgap_params& p, float* logits, int row,
                             int32_t* topk_idx, float* topk_val, float* risk, uint8_t* gate,
                             int32_t* next_token, float* features, const DWs& ws, Smem& sm,
                             int w1_staged) {
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int K = d.K, K1 = d.K + 1, nc = d.n_chunks;
  const int nin = 5 * K + 8;
  const float4* st = ws.stats + (size_t)row * nc;

  // The corrector's first layer, fetched while the window is formed (only
  // used when the row is gated; always awaited before the CTA exits).
  const bool w1s = w1_staged != 0;
  const uint32_t w1_bytes = (uint32_t)((size_t)d.hidden * nin * sizeof(float));
  const bool w1v = (nin & 3) == 0 && (reinterpret_cast<uintptr_t>(p.cor_w1) & 15) == 0;
  if (!w1s && w1v)  // every 128-byte line of W1 into L1 while the window is formed
    for (uint32_t o = (uint32_t)tid * 128u; o < w1_bytes; o += (uint32_t)kT * 128u)
      asm volatile("prefetch.global.L1 [%0];" ::"l"(reinterpret_cast<const char*>(p.cor_w1) + o));
  if (w1s && tid == 0) {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // chunk-phase writes first
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_u32(&sm.w1_bar)) : "memory");
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(&sm.w1_bar)),
                 "r"(w1_bytes)
                 : "memory");
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
            smem_u32(sm.u.w1)),
        "l"(p.cor_w1), "r"(w1_bytes), "r"(smem_u32(&sm.w1_bar))
        : "memory");
  }

  // This thread's detector unit (j = tid), loaded with the first round.
  float dw[8], db1 = 0.0f, dw2 = 0.0f;
  if (tid < d.hidden) {
#pragma unroll
    for (int i = 0; i < 8; ++i) dw[i] = __ldg(p.det_w1 + tid * 8 + i);
    db1 = __ldg(p.det_b1 + tid);
    dw2 = __ldg(p.det_w2 + tid);
  }

  // The corrector's output-layer weights of this thread (output k = tid / 8,
  // every eighth hidden unit from tid mod 8), when that layer is one pass of
  // at most 256 units, and its hidden bias: fetched with the first round of
  // loads, used only if the row is gated.
  constexpr int kW2Reg = 32;
  const bool w2r = K <= kT / 8 && d.hidden <= 8 * kW2Reg;
  float w2v[kW2Reg];
  if (w2r) {
    const int k = tid >> 3, s8 = tid & 7;
#pragma unroll
    for (int i = 0; i < kW2Reg; ++i) {
      const int j = s8 + 8 * i;
      w2v[i] = (k < K && j < d.hidden) ? __ldg(p.cor_w2 + (size_t)k * d.hidden + j) : 0.0f;
    }
  }
  const float cb1 = tid < d.hidden ? __ldg(p.cor_b1 + tid) : 0.0f;
  // Chunk statistics and candidate lists in one round of loads.
  const uint2* cand = ws.cand + (size_t)row * nc * K1;
  const int n_cand = nc * K1;
  uint32_t ck[kCandReg];
  int cx[kCandReg];
#pragma unroll
  for (int e = 0; e < kCandReg; ++e) {
    const int i = tid + e * kT;
    const uint2 v = i < n_cand ? __ldcg(&cand[i]) : make_uint2(0u, (uint32_t)INT_MAX);
    ck[e] = v.x;
    cx[e] = (int)v.y;
  }
  // The lists are sorted best first, so the first r0 = ceil(K1 / nc)
  // entries of every list (r0 nc >= K1 of them, all at or above their own
  // K1-th best) bound the K1-th best overall from below by their K1-th best.
  // They are loaded with this round and ranked directly, which spares
  // select_top's shuffle network and one barrier; either bound leaves a few
  // dozen candidates on such lists.
  const int r0 = (K1 + nc - 1) / nc, m_u = r0 * nc;  // m_u <= K1 + nc - 1 <= 2 kT
  uint2 uv[2];
#pragma unroll
  for (int e = 0; e < 2; ++e) {
    const int t = tid + e * kT;
    uv[e] = t < m_u ? __ldcg(&cand[(t / r0) * K1 + t % r0]) : make_uint2(0u, 0u);
  }
  float4 sv[(kMaxChunks + kT - 1) / kT];
#pragma unroll
  for (int j = 0; j < (kMaxChunks + kT - 1) / kT; ++j) {
    const int c = tid + j * kT;
    sv[j] = c < nc ? __ldcg(&st[c]) : make_float4(-INFINITY, 0.0f, 0.0f, 0.0f);
  }
#pragma unroll
  for (int e = 0; e < 2; ++e) {
    const int t = tid + e * kT;
    if (t < m_u) sm.su[t] = ((unsigned long long)uv[e].x << 32) | (uint32_t)~uv[e].y;
  }
  float mloc = -INFINITY;
#pragma unroll
  for (int j = 0; j < (kMaxChunks + kT - 1) / kT; ++j) mloc = fmaxf(mloc, sv[j].x);
  const float M = block_max(mloc, sm.red);  // also publishes su
  {
    // rank of each leader, P = 8, 4, 2 or 1 consecutive lanes per leader
    // (each over every P-th other leader, summed by shuffles); the one of
    // rank K1 - 1 gives the bound
    const int P = m_u <= kT / 8 ? 8 : m_u <= kT / 4 ? 4 : m_u <= kT / 2 ? 2 : 1;
    for (int base = 0; base < m_u * P; base += kT) {
      const int w = base + tid, t = w / P, part = w % P;
      const unsigned long long me = t < m_u ? sm.su[t] : 0ull;
      int r = 0;
      if (t < m_u)
        for (int j = part; j < m_u; j += P) {
          const unsigned long long o = sm.su[j];
          r += (o > me) || (o == me && j < t);
        }
      for (int o = 1; o < P; o <<= 1) r += __shfl_xor_sync(0xffffffffu, r, o);
      if (t < m_u && part == 0 && r == K1 - 1) sm.t0 = (uint32_t)(me >> 32);
    }
  }
  float s1 = 0.0f, s2 = 0.0f;
#pragma unroll
  for (int j = 0; j < (kMaxChunks + kT - 1) / kT; ++j) {
    const float4 v = sv[j];
    if (v.y > 0.0f) {
      const float e = expf(v.x - M);
      s1 += v.y * e;
      s2 += (v.z + (v.x - M) * v.y) * e;
    }
  }
  const float S1 = block_sum(s1, sm.red);
  const float S2 = block_sum(s2, sm.red);

  // The window: the K + 1 best of all chunk candidates (the registers hold
  // the first kCandReg * 256; a longer list goes the radix way).
  auto from_global = [&]() {
    block_select(n_cand, K1, [&](int i, uint32_t& k, int& x) {
      const uint2 v = __ldcg(&cand[i]);
      k = v.x;
      x = (int)v.y;
    }, sm.sel, sm.fk, sm.fi, &sm.wk[0][0], &sm.wi[0][0]);
  };
  if (n_cand > kCandReg * kT) from_global();
  else select_above(ck, cx, K1, sm.t0, sm.sel, sm.sv, sm.fk, sm.fi, from_global);

  // Features phi (Sec. 4.2): warp 0, lanes over the window.
  if (warp == 0) {
    const float z0 = key_value(sm.fk[0]);
    float mass_e = 0.0f, wsum_e = 0.0f, sum = 0.0f, min_gap = INFINITY;
    for (int k = lane; k < K; k += 32) {
      const float zk = key_value(sm.fk[k]);
      const float e = expf(zk - M);
      mass_e += e;
      wsum_e += e * (zk - M);
      sum += zk;
      if (k + 1 < K) min_gap = fminf(min_gap, zk - key_value(sm.fk[k + 1]));
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) {  // four independent reductions, interleaved
      mass_e += __shfl_xor_sync(0xffffffffu, mass_e, o);
      wsum_e += __shfl_xor_sync(0xffffffffu, wsum_e, o);
      sum += __shfl_xor_sync(0xffffffffu, sum, o);
      min_gap = fminf(min_gap, __shfl_xor_sync(0xffffffffu, min_gap, o));
    }
    const float mean = sum / (float)K;
    float var = 0.0f;
    for (int k = lane; k < K; k += 32) {
      const float dz = key_value(sm.fk[k]) - mean;
      var += dz * dz;
    }
    var = wsum(var) / (float)K;
    if (lane == 0) {
      sm.phi[0] = logf(S1) - S2 / S1;
      sm.phi[1] = mass_e / S1;
      sm.phi[2] = expf(z0 - M) / S1;
      sm.phi[3] = z0 - key_value(sm.fk[1]);
      sm.phi[4] = (z0 - key_value(sm.fk[K - 1])) / (float)(K - 1);
      sm.phi[5] = min_gap;
      sm.phi[6] = sqrtf(var);
      sm.phi[7] = logf(mass_e) - wsum_e / mass_e;
    }
  }
  for (int k = tid; k < K; k += kT) sm.zt[k] = key_value(sm.fk[k]);
  __syncthreads();

  // Detector f = w2 . relu(W1 phi + b1) + b2 (Eq. 6).
  float part = 0.0f;
  if (tid < d.hidden) {
    float a = db1;
#pragma unroll
    for (int i = 0; i < 8; ++i) a = fmaf(dw[i], sm.phi[i], a);
    part = dw2 * fmaxf(a, 0.0f);
  }
  for (int j = tid + kT; j < d.hidden; j += kT) {
    float a = p.det_b1[j];
#pragma unroll
    for (int i = 0; i < 8; ++i) a = fmaf(p.det_w1[j * 8 + i], sm.phi[i], a);
    part = fmaf(p.det_w2[j], fmaxf(a, 0.0f), part);
  }
  const float f = block_sum(part, sm.red) + p.det_b2[0];
  const bool gated = f > d.logit_tau;

  bool w1_ok = true;
  if (w1s) {  // every thread observes the copy's completion (bounded wait)
    const long long t0 = clock64();
    uint32_t done = 0;
    while (!done) {
      asm volatile(
          "{\n .reg .pred q;\n mbarrier.try_wait.parity.shared::cta.b64 q, [%1], 0;\n"
          " selp.u32 %0, 1, 0, q;\n}"
          : "=r"(done)
          : "r"(smem_u32(&sm.w1_bar))
          : "memory");
      if (!done && clock64() - t0 > 4000000000LL) break;
    }
    w1_ok = __syncthreads_and(done != 0);
  }

  if (gated) {
    // Candidate features xi (Sec. 4.3), rank-major, then phi.
    const float lse = M + logf(S1);
    const float z0 = sm.zt[0];
    for (int k = tid; k < K; k += kT) {
      const float zk = sm.zt[k];
      const float znext = k + 1 < K ? sm.zt[k + 1] : key_value(sm.fk[K]);
      sm.x[5 * k + 0] = zk - z0;
      sm.x[5 * k + 1] = zk - lse;
      sm.x[5 * k + 2] = (float)k / (float)(K - 1);
      sm.x[5 * k + 3] = k == 0 ? 0.0f : sm.zt[k - 1] - zk;
      sm.x[5 * k + 4] = zk - znext;
    }
    if (tid < 8) sm.x[5 * K + tid] = sm.phi[tid];
    __syncthreads();
    // Hidden layer: one thread per hidden unit (W1 from shared memory when
    // staged, else through L1).
    const float* w1 = (w1s && w1_ok) ? sm.u.w1 : p.cor_w1;
    if (w1v && (!w1s || w1_ok)) {
      // rows of float4s (shared memory when staged, else global memory
      // through L1), four accumulators.  With an even number n4
      // of float4s per row, thread j starts at column j mod 8: the float4 at
      // column c of row j lies in 16-byte bank group (j n4 + c) mod 8, so the
      // eight rows a quarter-warp reads fall in groups j (n4 + 1) mod 8, all
      // different (n4 + 1 odd), and so do the eight inputs it reads.
      const float4* xv = reinterpret_cast<const float4*>(sm.x);
      const int n4 = nin / 4;
      const auto rows = [&](auto load) {
        for (int j = tid; j < d.hidden; j += kT) {
          const float4* wr = reinterpret_cast<const float4*>(w1 + (size_t)j * nin);
          float4 a = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
          int c = (n4 & 1) ? 0 : (j & 7) % n4;
#pragma unroll 6
          for (int t = 0; t < n4; ++t) {
            const float4 w = load(wr + c), xx = xv[c];
            c = c + 1 == n4 ? 0 : c + 1;
            a.x = fmaf(w.x, xx.x, a.x);
            a.y = fmaf(w.y, xx.y, a.y);
            a.z = fmaf(w.z, xx.z, a.z);
            a.w = fmaf(w.w, xx.w, a.w);
          }
          const float b1 = j == tid ? cb1 : __ldg(p.cor_b1 + j);
          sm.hb[j] = fmaxf((a.x + a.y) + (a.z + a.w) + b1, 0.0f);
        }
      };
      if (w1s) rows([](const float4* q) { return *q; });
      else rows([](const float4* q) { return __ldg(q); });
    } else
    for (int j = tid; j < d.hidden; j += kT) {
      const float* wrow = w1 + (size_t)j * nin;
      float a0 = 0.0f, a1 = 0.0f;
      int i = j % nin;
      for (int c = 0; c + 1 < nin; c += 2) {
        a0 = fmaf(wrow[i], sm.x[i], a0);
        i = i + 1 == nin ? 0 : i + 1;
        a1 = fmaf(wrow[i], sm.x[i], a1);
        i = i + 1 == nin ? 0 : i + 1;
      }
      if (nin & 1) a0 = fmaf(wrow[i], sm.x[i], a0);
      sm.hb[j] = fmaxf(a0 + a1 + p.cor_b1[j], 0.0f);
    }
    __syncthreads();
    // Output layer Delta_k: eight threads per output, each over every eighth
    // hidden unit (rows prefetched into L1 above), then the sparse merge
    // (Eq. 13).
    for (int k0 = 0; k0 < K; k0 += kT / 8) {
      const int k = k0 + (tid >> 3), s8 = tid & 7;
      float a = 0.0f;
      if (w2r) {
#pragma unroll
        for (int i = 0; i < kW2Reg; ++i)
          if (s8 + 8 * i < d.hidden) a = fmaf(w2v[i], sm.hb[s8 + 8 * i], a);
      } else if (k < K) {
        const float* wrow = p.cor_w2 + (size_t)k * d.hidden;
#pragma unroll 8
        for (int j = s8; j < d.hidden; j += 8) a = fmaf(__ldg(wrow + j), sm.hb[j], a);
      }
      a += __shfl_xor_sync(0xffffffffu, a, 1);
      a += __shfl_xor_sync(0xffffffffu, a, 2);
      a += __shfl_xor_sync(0xffffffffu, a, 4);
      if (k < K && s8 == 0) {
        const float zt = sm.zt[k] + (a + p.cor_b2[k]);
        sm.zt[k] = zt;
        logits[(size_t)row * d.vocab + sm.fi[k]] = zt;
      }
    }
    __syncthreads();
  }

  for (int k = tid; k < K; k += kT) {
    topk_idx[(size_t)row * K + k] = sm.fi[k];
    topk_val[(size_t)row * K + k] = sm.zt[k];
  }
  if (features && tid < 8) features[(size_t)row * 8 + tid] = sm.phi[tid];
  if (tid == 0) {
    risk[row] = 1.0f / (1.0f + expf(-f));
    gate[row] = gated ? 1 : 0;
    ws.tk[row] = 0u;
  }
  if (next_token && warp == 0) {
    // greedy token: the best of the corrected window and z_(K+1), the lower
    // index on ties (a total order, so the lanes' partial bests reduce)
    float bv = lane == 0 ? key_value(sm.fk[K]) : -INFINITY;
    int bi = lane == 0 ? sm.fi[K] : INT_MAX;
    for (int k = lane; k < K; k += 32)
      if (sm.zt[k] > bv || (sm.zt[k] == bv && sm.fi[k] < bi)) {
        bv = sm.zt[k];
        bi = sm.fi[k];
      }
#pragma unroll
    for (int o = 16; o; o >>= 1) {
      const float ov = __shfl_xor_sync(0xffffffffu, bv, o);
      const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
      if (ov > bv || (ov == bv && oi < bi)) {
        bv = ov;
        bi = oi;
      }
    }
    if (lane == 0) next_token[row] = bi;
  }
}

// Two CTAs per SM when W1 is not staged (at most 128 registers).
__global__ void __launch_bounds__(kT, 2)
    dgap_kernel(DgapDims d, dgap_params p, float* __restrict__ logits, int32_t* topk_idx,
                float* topk_val, float* risk, uint8_t* gate, int32_t* next_token,
                float* features, DWs ws, int w1_staged) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  Smem& sm = *reinterpret_cast<Smem*>(smem_raw);
  // programmatic dependent launch: the logits are the previous kernel's output
  asm volatile("griddepcontrol.launch_dependents;\ngriddepcontrol.wait;" ::: "memory");
  const int tid = threadIdx.x;
  const int chunk = blockIdx.x, row = blockIdx.y, K1 = d.K + 1;
  const float* z = logits + (size_t)row * d.vocab;
  const int base = chunk * kChunk;

  float v[kPer];
  uint32_t k[kPer];
  int ix[kPer];
  float lm = -INFINITY;
#pragma unroll
  for (int i = 0; i < kPer; ++i) {
    const int e = base + i * kT + tid;
    if (e < d.vocab) {
      v[i] = z[e];
      k[i] = order_key(v[i]);
      ix[i] = e;
      lm = fmaxf(lm, v[i]);
    } else {
      v[i] = -INFINITY;
      k[i] = 0u;
      ix[i] = INT_MAX;
    }
  }
  const float m = block_max(lm, sm.red);
  float s1 = 0.0f, s2 = 0.0f;
#pragma unroll
  for (int i = 0; i < kPer; ++i) {
    if (ix[i] != INT_MAX) {
      const float dz = v[i] - m;
      const float e = expf(dz);
      s1 += e;
      s2 = fmaf(dz, e, s2);
    }
  }
  s1 = block_sum(s1, sm.red);
  s2 = block_sum(s2, sm.red);

  select_top(k, ix, K1, sm.sel, sm.sv, sm.fk, sm.fi, [&]() {
#pragma unroll
    for (int i = 0; i < kPer; ++i) {
      sm.u.srt.sk[i * kT + tid] = k[i];
      sm.u.srt.si[i * kT + tid] = ix[i];
    }
    __syncthreads();
    block_select(kChunk, K1, [&](int i, uint32_t& kk, int& ii) {
      kk = sm.u.srt.sk[i];
      ii = sm.u.srt.si[i];
    }, sm.sel, sm.fk, sm.fi, &sm.wk[0][0], &sm.wi[0][0]);
  });
  uint2* out = ws.cand + ((size_t)row * d.n_chunks + chunk) * K1;
  for (int r = tid; r < K1; r += kT) out[r] = make_uint2(sm.fk[r], (uint32_t)sm.fi[r]);
  if (tid == 0) ws.stats[(size_t)row * d.n_chunks + chunk] = make_float4(m, s1, s2, 0.0f);

  __syncthreads();
  if (tid == 0) {
    unsigned t;
    asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], 1;" : "=r"(t) : "l"(&ws.tk[row]) : "memory");
    sm.last = (t == (unsigned)d.n_chunks - 1);
  }
  __syncthreads();
  if (!sm.last) return;
  finalize_row(d, p, logits, row, topk_idx, topk_val, risk, gate, next_token, features, ws, sm,
               w1_staged);
}

}  // namespace

int dgap_chunks(int vocab) { return (vocab + kChunk - 1) / kChunk; }
int dgap_max_chunks() { return kMaxChunks; }

size_t dgap_workspace_bytes_impl(int batch, int vocab, int K) {
  const int nc = dgap_chunks(vocab);
  return a256((size_t)batch * nc * sizeof(float4)) +
         a256((size_t)batch * nc * (K + 1) * sizeof(uint2)) + a256((size_t)batch * 4);
}

cudaError_t launch_dgap(const DgapDims& d, const dgap_params& p, float* logits, int32_t* topk_idx,
                        float* topk_val, float* risk, uint8_t* gate, int32_t* next_token,
                        float* features, void* workspace, cudaStream_t stream) {
  const DWs ws = carve(workspace, d.batch, d.n_chunks, d.K);
  static int sms = 0;
  if (!sms) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      return cudaGetLastError();
  }
  const int w1_staged = stage_w1(d, p, sms) ? 1 : 0;
  const size_t smem = w1_staged ? sizeof(Smem) : kSmemNoW1;
  static_assert(sizeof(Smem) <= 227 * 1024, "DGAP shared memory must fit one SM");
  cudaError_t e = cudaFuncSetAttribute(dgap_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)sizeof(Smem));
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(d.n_chunks, d.batch);
  cfg.blockDim = dim3(kT);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  e = cudaLaunchKernelEx(&cfg, dgap_kernel, d, p, logits, topk_idx, topk_val, risk, gate,
                         next_token, features, ws, w1_staged);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace kvq
