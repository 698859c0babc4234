// kvq_decode_attn: one decode step of grouped-query attention
// softmax(q K^T * scale) V (Sec. 1 of the paper) over the packed KbVb cache.
//
// Grid (S, n_kv_heads, batch) of 512-thread CTAs, one per SM.  The S CTAs
// of one (sequence, kv-head) share its work: the packed 32-token blocks and
// the 32-token chunks of the fp16 residual window are cut into contiguous
// ranges, one per warp (a warp takes only blocks or only window chunks).
// Each warp streams its own pages into a private ring of shared-memory slots
// with bulk asynchronous copies (cp.async.bulk + one mbarrier per slot) and
// keeps a running softmax state.  The warps of a CTA merge in shared memory
// into one partial (max, sum, unnormalised row) per query head; with S > 1
// the last CTA of a (sequence, kv-head) to finish (atomic ticket, no
// waiting) merges the S partials:
//   out = sum_s 2^{m_s - M} o_s / sum_s 2^{m_s - M} l_s.
// Scores are kept in the log2 domain (scaled by softmax_scale * log2 e).
//
// Packed blocks run on the tensor cores (mma.sync m16n8k16, f16 in, f32
// accumulate) with operands built in registers straight from the packed
// codes:
//
//   keys    S[t][h] = sum_c code[t][c] * (q_h[c] s_c) + sum_c q_h[c] z_c
//           A = codes (M = tokens, K = channels), B = q*s split into an fp16
//           high part and its exact fp16 residual, so the products are
//           exact; the zero-point term is one more MMA with A = z, B = q.
//           1-bit keys with 5..8-head groups instead scale A: A = code * s
//           (one fp16 multiply per register), B = q, one MMA per tile.
//   values  o[c][h] += sum_t code[t][c] * (p_h[t] s_t,g) + sum_t p_h[t] z_t,g
//           A = codes (M = channels, K = tokens), B = p*s with p split into
//           high / low fp16 parts; P moves from the score (accumulator)
//           layout to the B layout with movmatrix.
// The B operand's 8 columns hold, for query groups of up to 4 heads, the
// high parts of the 4 heads in columns 0..3 and the low parts in 4..7 (one
// MMA per operand pair, "narrow"); for groups of 5..8 heads one head per
// column, and the high and low parts are two MMAs into the same accumulator
// ("wide"), so the codes of a block are converted once for all heads.
//
// Codes become fp16 values without a table: for 1-bit codes (stored in
// fragment order) a rotated bit lands on an exponent bit (value 2^e), for
// wider codes the code is OR-ed into the mantissa of 1024 and 1024 is
// subtracted.  The resulting per-row power-of-two factors are undone on the
// fp32 results.  The fp16 residual window takes the same MMAs with operands
// loaded by ldmatrix from rows staged in shared memory.

#include <float.h>

#include <mutex>

#include "common.cuh"

namespace kvq {
namespace {

#include "attn_core.cuh"

constexpr int kFinCap = 2 * kWarps + 2;           // final merges one CTA can owe (<= kWarps + 1)
constexpr int kLenCap = 1024;                     // sequence lengths a CTA keeps in shared memory

// Split partials: slots [0, ctas + P) for the CTA partials, then one warp
// partial per pair (P = batch * n_kv_heads pairs); tickets: one per pair,
// then the decode step's count of finished CTAs.
struct Ws {
  float* m;       // [slots][gq] row maxima (log2 domain)
  float* l;       // [slots][gq] row sums
  float* o;       // [slots][gq][128] unnormalised rows
  unsigned* tk;   // [P + 1]
};

__host__ __device__ inline size_t align256(size_t x) { return (x + 255) / 256 * 256; }

__host__ __device__ inline size_t ws_slots(int batch, int hkv, int ctas) {
  return (size_t)ctas + 2 * (size_t)batch * hkv;
}
__host__ __device__ inline Ws carve(void* base, int batch, int hq, int hkv, int ctas) {
  Ws w;
  char* p = static_cast<char*>(base);
  const size_t nml = ws_slots(batch, hkv, ctas) * (size_t)(hq / hkv);
  w.m = reinterpret_cast<float*>(p);
  p += align256(nml * 4);
  w.l = reinterpret_cast<float*>(p);
  p += align256(nml * 4);
  w.o = reinterpret_cast<float*>(p);
  p += align256(nml * kHeadDim * 4);
  w.tk = reinterpret_cast<unsigned*>(p);
  return w;
}

// Small shared arrays of the merges (static shared memory).
struct MergeSmall {
  float ww[kWarps][kHeads];             // warp merge weights 2^(m_w - M)
  float gm[kWarps][kHeads];             // a group's maximum M
};
// The CTA's merge groups: warps [w0, w1) end in the same pair; cnt = the
// pair's partials in all.
struct MergeGroups {
  int w0[kWarps], w1[kWarps], cnt[kWarps];
  int n;
};

// ---------------------------------------------------------------------------
// The flat work plan.  Pair p = b * Hkv + h (sequence b, kv-head h) is a list
// of items: its packed 32-token blocks (cost 1 each), then the 32-token
// chunks of its fp16 window (cost cw each); the first item costs sc more (a
// warp that starts a pair waits once for its first pages).  All pairs' items
// lie end to end in cost units, cut into n_v equal contiguous unit ranges,
// one per virtual warp; an item belongs to the virtual warp whose range holds
// its first unit.  The virtual warps are cut into n_cta contiguous groups of
// at most kWarps, one per CTA.  So every warp streams one contiguous run of
// blocks, possibly across pair boundaries, and all warps carry the same
// cost: the launch is one wave of CTAs with no per-pair split count.
// n_v <= units / (cw + sc) keeps every range long enough to hold the first
// unit of an item, so no virtual warp is empty.
//
// Partials.  A warp keeps one softmax state per pair it touches.  The state
// of its last pair goes to its CTA, which merges the warps that end in the
// same pair into one CTA partial (slot cta + p, unique: CTA ranges and pair
// ranges are both ordered).  A state of a pair the warp leaves for the next
// one is a warp partial (slot n_slots_cta + p; at most one per pair: only the
// owner of the pair's last item can continue past it).  Each partial bumps
// the pair's ticket; the one that completes it merges the pair's partials
// (pair_partials gives their number).  A pair with one partial in all is
// written out directly.
// ---------------------------------------------------------------------------

// Cost weights: a window chunk costs cw units, the first item of a pair sc
// more (measured: a chunk takes ~4 blocks' time, a pair start ~1), and the
// block that leaves the window in a decode step fu more (its warp quantizes
// the block alone; Mistral-7B shape, K2V2, ragged batch of 16 where some
// sequence flushes on most steps: 0, 4, 8 and 12 units gave 4.30, 4.24,
// 4.19 and 4.18 ms mean and 4.70, 4.54, 4.40 and 4.37 ms p95 per 32-layer
// step).  A launch with too little work
// for every warp to hold an item under those weights takes lighter ones
// (FlatGrid::k), down to one unit per item.
struct Costs {
  int cw, sc, fu;
};

struct PairShape {
  int Lq, nb, nr;  // packed tokens, packed blocks, window chunks
};
__host__ __device__ inline PairShape pair_shape(int L, int residual) {
  PairShape s;
  s.Lq = packed_len(L, residual);
  s.nb = s.Lq / kGroup;
  s.nr = (L - s.Lq + kGroup - 1) / kGroup;
  return s;
}
// Extra units f of a pair whose last packed block leaves the window in this
// launch (a decode step that appends a token: L = L0 + 1).
__host__ __device__ inline int flush_units(int L0, int L, int residual, Costs k) {
  return L > L0 && packed_len(L, residual) > packed_len(L0, residual) ? k.fu : 0;
}
__host__ __device__ inline int pair_cost(const PairShape& s, Costs k, int f) {
  return s.nb + s.nr > 0 ? k.sc + s.nb + f + k.cw * s.nr : 0;
}
// First unit (pair-local) of item i; the last packed block (nb - 1) costs
// 1 + f units.
__host__ __device__ inline int item_unit(int i, int nb, Costs k, int f) {
  return i == 0 ? 0 : k.sc + (i < nb ? i : nb + f + k.cw * (i - nb));
}
// Largest cost of one item under the weights (a warp's range holds at least
// this many units, so every warp holds an item start).
__host__ __device__ inline int max_item_cost(Costs k) {
  return k.cw + k.sc > 1 + k.fu + k.sc ? k.cw + k.sc : 1 + k.fu + k.sc;
}
// Number of items of a pair whose first unit (pair-local) is below x.
__host__ __device__ inline int items_below(long long x, int nb, int nr, Costs k, int f) {
  if (x <= 0 || nb + nr == 0) return 0;
  int c = 1;
  if (nb > 1) c += (int)min((long long)(nb - 1), max(0LL, x - k.sc - 1));
  const int lo_w = nb == 0 ? 1 : 0;
  if (nr > lo_w) {
    const long long t = x - k.sc - nb - f;
    const int sh = k.cw == 4 ? 2 : k.cw == 2 ? 1 : 0;  // cw is 1, 2 or 4
    const long long n = t <= 0 ? 0 : (t + k.cw - 1) >> sh;
    c += (int)max(0LL, min(n, (long long)nr) - lo_w);
  }
  return c;
}

// Work totals of a launch: packed blocks, window chunks, non-empty pairs,
// pairs with a block leaving the window.
struct WorkSums {
  long long nb, nr, np, nf;
};

// floor(x / d) from r = floor((2^64 - 1) / d): the high half of x * r is at
// most two below the quotient (r >= 2^64 / d - 1, x < 2^64), so two checks
// make it exact.  Integer division on the GPU is a long software sequence;
// the plan divides by the same N and n_v many times.
__host__ __device__ inline unsigned long long rcp64(unsigned long long d) {
  return d ? ~0ULL / d : 0ULL;
}
__host__ __device__ inline long long div_rcp(unsigned long long x, unsigned long long d,
                                             unsigned long long r) {
#ifdef __CUDA_ARCH__
  unsigned long long q = __umul64hi(x, r);
#else
  unsigned long long q = (unsigned long long)(((unsigned __int128)x * r) >> 64);
#endif
  if ((q + 1) * d <= x) ++q;
  if ((q + 1) * d <= x) ++q;
  return (long long)q;
}

struct FlatGrid {
  long long N;               // cost units of all pairs
  int n_v;                   // virtual warps (0 when N == 0)
  int n_cta;                 // CTAs that carry work, <= gridDim.x
  Costs k;                   // cost weights
  unsigned long long rN, rV; // reciprocals of N and n_v (div_rcp)
};
__host__ __device__ inline FlatGrid flat_grid(const WorkSums& w, int ctas) {
  FlatGrid g;
  const long long cap = (long long)kWarps * ctas;
  // the heaviest weights under which every one of the cap warps can still
  // hold an item start (each range >= the largest item cost)
  const Costs pick[3] = {{4, 1, 12}, {2, 1, 6}, {1, 0, 0}};
  int i = 0;
  for (; i < 2; ++i) {
    const long long N = w.nb + pick[i].cw * w.nr + pick[i].sc * w.np + pick[i].fu * w.nf;
    if (N / max_item_cost(pick[i]) >= cap) break;
  }
  g.k = pick[i];
  g.N = w.nb + g.k.cw * w.nr + g.k.sc * w.np + g.k.fu * w.nf;
  const long long nv = g.N / max_item_cost(g.k);
  g.n_v = g.N == 0 ? 0 : (int)(nv < 1 ? 1 : (nv < cap ? nv : cap));
  g.n_cta = g.n_v < ctas ? g.n_v : ctas;
  g.rN = rcp64((unsigned long long)g.N);
  g.rV = rcp64((unsigned long long)g.n_v);
  return g;
}
__host__ __device__ inline int unit_owner(long long u, const FlatGrid& g) {
  return (int)div_rcp((unsigned long long)(u + 1) * g.n_v - 1, g.N, g.rN);
}
__host__ __device__ inline long long v_first_unit(int v, const FlatGrid& g) {
  return div_rcp((unsigned long long)g.N * v, g.n_v, g.rV);
}
// (n_v < 2^12 and n_cta < 2^8: 32-bit arithmetic)
__host__ __device__ inline int cta_of(int v, const FlatGrid& g) {
  return (int)(((unsigned)(v + 1) * (unsigned)g.n_cta - 1u) / (unsigned)g.n_v);
}
__host__ __device__ inline int cta_first_v(int c, const FlatGrid& g) {
  return (int)((unsigned)g.n_v * (unsigned)c / (unsigned)g.n_cta);
}
// Partials of a non-empty pair (first unit U, cost C): the CTA partials of
// CTAs [c_a, c_a + n_cta) and, if `cont`, one warp partial.
__host__ __device__ inline int pair_partials(long long U, int C, int nb, int nr, int f,
                                             const FlatGrid& g, int& c_a, int& n_cta,
                                             bool& cont) {
  const int wf = unit_owner(U, g);
  const int wl = unit_owner(U + item_unit(nb + nr - 1, nb, g.k, f), g);
  cont = U + C < g.N && unit_owner(U + C, g) == wl;
  const int hv = wl - (cont ? 1 : 0);
  c_a = cta_of(wf, g);
  n_cta = hv >= wf ? cta_of(hv, g) - c_a + 1 : 0;
  return n_cta + (cont ? 1 : 0);
}

// Length a kernel attends: the decode step counts its own token.
__device__ __forceinline__ int attended_len(int L0, const Dims& d, bool append) {
  return append && L0 < d.max_len ? L0 + 1 : L0;
}
__device__ __forceinline__ long long warp_sum_ll(long long v) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
// Work totals of all pairs (lengths as the kernel attends them).
__device__ WorkSums plan_sums(const int* seq_len, const Dims& d, bool append) {
  const int lane = threadIdx.x & 31;
  long long nb = 0, nr = 0, np = 0, nf = 0;
  const Costs one = {1, 0, 1};
  for (int b0 = 0; b0 < d.batch; b0 += 32) {
    const int b = b0 + lane;
    const int L0 = b < d.batch ? read_len(seq_len + b) : 0;
    const int L = b < d.batch ? attended_len(L0, d, append) : 0;
    const PairShape s = pair_shape(L, d.residual);
    nb += warp_sum_ll((long long)d.hkv * s.nb);
    nr += warp_sum_ll((long long)d.hkv * s.nr);
    np += warp_sum_ll(s.nb + s.nr > 0 ? d.hkv : 0);
    nf += warp_sum_ll((long long)d.hkv * flush_units(L0, L, d.residual, one));
  }
  WorkSums w;
  w.nb = nb;
  w.nr = nr;
  w.np = np;
  w.nf = nf;
  return w;
}

// A warp's walk over the pairs its unit range [a, e) meets, in order.
struct Walk {
  int b, h;        // current sequence and kv-head
  long long Ub;    // first unit of sequence b
  int L0, L, pc;   // stored and attended length of b, cost of one of its pairs
  int f;           // flush units of b's pairs
};
__device__ __forceinline__ void walk_load(Walk& w, const int* seq_len, const Dims& d,
                                          bool append, Costs k) {
  if (w.b < d.batch) {
    w.L0 = read_len(seq_len + w.b);
    w.L = attended_len(w.L0, d, append);
    w.f = flush_units(w.L0, w.L, d.residual, k);
    w.pc = pair_cost(pair_shape(w.L, d.residual), k, w.f);
  }
}
// Position at the first pair whose units reach past a (an empty pair at or
// after a included): a scan of the sequences' costs, 32 at a time.
__device__ Walk walk_start(long long a, const int* seq_len, const Dims& d, bool append, Costs k) {
  const int lane = threadIdx.x & 31;
  Walk w;
  long long base = 0;
  for (int b0 = 0; b0 < d.batch; b0 += 32) {
    const int b = b0 + lane;
    const int L0 = b < d.batch ? read_len(seq_len + b) : 0;
    const int L = attended_len(L0, d, append);
    const int f = flush_units(L0, L, d.residual, k);
    const int pc = b < d.batch ? pair_cost(pair_shape(L, d.residual), k, f) : 0;
    const long long cst = (long long)d.hkv * pc;
    long long incl = cst;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const long long y = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += y;
    }
    incl += base;
    const long long excl = incl - cst;
    const unsigned hit = __ballot_sync(0xffffffffu, b < d.batch && (incl > a || (cst == 0 && excl >= a)));
    if (hit) {
      const int l = __ffs(hit) - 1;
      w.b = b0 + l;
      w.Ub = __shfl_sync(0xffffffffu, excl, l);
      w.L0 = __shfl_sync(0xffffffffu, L0, l);
      w.L = __shfl_sync(0xffffffffu, L, l);
      w.pc = __shfl_sync(0xffffffffu, pc, l);
      w.f = __shfl_sync(0xffffffffu, f, l);
      w.h = w.pc > 0 && a > w.Ub ? (int)((a - w.Ub) / w.pc) : 0;
      return w;
    }
    base = __shfl_sync(0xffffffffu, incl, 31);
  }
  w.b = d.batch;
  w.h = 0;
  w.Ub = base;
  w.L0 = w.L = w.pc = w.f = 0;
  return w;
}
__device__ __forceinline__ void walk_next(Walk& w, const int* seq_len, const Dims& d, bool append,
                                          Costs k) {
  if (++w.h < d.hkv) return;
  w.h = 0;
  w.Ub += (long long)d.hkv * w.pc;
  ++w.b;
  walk_load(w, seq_len, d, append, k);
}




// Fold packed blocks [lo, hi) of one pair into st, streaming their pages
// through the warp's ring.  *pos_io counts the ring slots the warp has used
// in this kernel (slot pos % R, phase parity (pos / R) & 1) and moves past
// this call's slots; `pre` slots holding blocks [lo_h, pre_end) were
// streamed early from position 0 and are consumed without use unless this
// range begins with them.  keep_tail: the block after hi leaves the window
// in this kernel and folds after this call (tc_fold_flush); blocks fold in
// units of NB from lo, as kvq_decode_attn folds lo .. hi after kvq_pack, so
// if the range ends in a unit of one, that unit is not folded here and its
// page stays in the ring (*tail_out; otherwise nullptr) to fold with the
// flushed block: both paths then take the same softmax updates (1-bit values
// round their fp16 weights against the running maximum).
template <int BK, int BV, bool kWide>
__device__ __forceinline__ TcState tc_packed_warp(TcState st, const PageMap pm, int lo_h, int pre,
                                                  int pre_end, int lo, int hi, char* ring,
                                                  uint64_t* full, int* pos_io, const char* zero,
                                                  const __half* qh, int gq, float scale_log2,
                                                  unsigned* flag, bool keep_tail,
                                                  const char** tail_out) {
  TableWin tw;
  table_win_init(tw);
  constexpr int page = page_bytes_c(BK, BV);
  constexpr int NB = ring_blocks(page);
  constexpr int R = ring_slots(page);
  const int lane = threadIdx.x & 31;
  const bool reuse = pre > 0 && lo == lo_h && min(lo + pre * NB, hi) == pre_end;
  const int skip = reuse ? 0 : pre;
  const int n_units = hi > lo ? (hi - lo + NB - 1) / NB : 0;
  const int total = skip + n_units;
  const int p0 = *pos_io;
  const bool hold = keep_tail && NB == 2 && n_units > 0 && ((hi - lo) & 1);
  const char* tail = nullptr;
  int issued = pre;  // slots issued so far
  auto real_issue = [&](int s) {
    const int u = s - skip;
    // the slot may have been read (or written by generic stores: window rows,
    // a flushed page) before: order that before the copy that overwrites it
    issue_slot<BK, BV>(pm, tw, ring, full, R, p0 + s, lo + u * NB, min(NB, hi - lo - u * NB), flag,
                       true);
    issued = s + 1;
  };
  for (int s = pre; s < min(total, R); ++s) real_issue(s);

  const Lane ln = make_lane<BK, BV>(lane);
  uint32_t qb[16];
  load_qb<true, kWide>(qb, qh, gq, ln);
  int consumed = 0;
  for (int s = 0; s < total; ++s) {
    const int slot = (p0 + s) % R;
    // every lane waits; the warp leaves together if any lane gave up
    if (!__all_sync(0xffffffffu, mbar_wait(full + slot, ((p0 + s) / R) & 1))) {
      if (lane == 0) atomicOr(flag, KVQ_FLAG_WAIT_TIMEOUT);
      break;
    }
    consumed = s + 1;
    if (s >= skip) {
      const int u = s - skip;
      const char* base = ring + (size_t)slot * NB * page;
      if (hold && s == total - 1) {
        tail = base;
      } else if (lo + u * NB + NB <= hi) {
        const char* pg[NB];
#pragma unroll
        for (int i = 0; i < NB; ++i) pg[i] = base + i * page;
        tc_unit<BK, BV, NB, kWide>(pg, zero, qb, ln, scale_log2, st);
      } else {
        const char* pg[1] = {base};
        tc_unit<BK, BV, 1, kWide>(pg, zero, qb, ln, scale_log2, st);
      }
    }
    __syncwarp();
    if (s + R < total) real_issue(s + R);
  }
  // Copies issued but not consumed (a wait gave up, or the range shrank) land
  // before the ring is reused; bounded waits.
  if (lane == 0)
    for (int s = max(consumed, issued - R); s < issued; ++s)
      mbar_wait(full + (p0 + s) % R, ((p0 + s) / R) & 1);
  __syncwarp();
  *pos_io = p0 + issued;
  *tail_out = tail;
  return st;
}

// The block `blk` of a pair leaves the window in this kernel (decode step)
// and has no page yet: the warp quantizes it from the fp16 ring rows exactly
// as kvq_pack does (quantize_quarter, common.cuh) into its idle ring (or the
// second page of the held tail unit), writes the page and folds it, with the
// tail unit if there is one.  Rare (one block in 32 steps), so out of line.
template <int BK, int BV, bool kWide>
__device__ __noinline__ TcState tc_fold_flush(TcState st, const PageMap pm, int blk,
                                              const char* tail, char* ring, const char* zero,
                                              const __half* qh, int gq, float scale_log2,
                                              unsigned* flag, const __half* ring_k,
                                              const __half* ring_v, int ring_len) {
  constexpr int page = page_bytes_c(BK, BV);
  const int lane = threadIdx.x & 31;
  TableWin tw;
  table_win_init(tw);
  char* img = tail ? const_cast<char*>(tail) + page : ring;
  for (int qi = 0; qi < 4; ++qi) flush_quarter<BK, BV>(ring_k, ring_v, blk * kGroup, ring_len, qi, img);
  __syncwarp();
  char* dst = const_cast<char*>(block_addr(pm, tw, blk));
  if (dst) {
    uint4* d4 = reinterpret_cast<uint4*>(dst);
    for (int i = lane; i < page / 16; i += 32) d4[i] = reinterpret_cast<const uint4*>(img)[i];
  } else if (lane == 0) {
    atomicOr(flag, (unsigned)KVQ_FLAG_BAD_PAGE);
  }
  const Lane ln = make_lane<BK, BV>(lane);
  uint32_t qb[16];
  load_qb<true, kWide>(qb, qh, gq, ln);
  if (ring_blocks(page) == 2 && tail) {
    const char* pg[2] = {tail, img};
    tc_unit<BK, BV, 2, kWide>(pg, zero, qb, ln, scale_log2, st);
  } else {
    const char* pg[1] = {img};
    tc_unit<BK, BV, 1, kWide>(pg, zero, qb, ln, scale_log2, st);
  }
  __syncwarp();
  return st;
}


// Bring ring rows [p0, p0 + n) (one or two contiguous runs) into L2.
__device__ __forceinline__ void prefetch_rows_l2(const __half* ring_base, int p0, int n, int ring) {
  const int s0 = p0 % ring;
  const int n1 = min(n, ring - s0);
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(ring_base + (long long)s0 * kHeadDim),
               "r"((uint32_t)(n1 * kHeadDim * 2))
               : "memory");
  if (n > n1)
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(ring_base),
                 "r"((uint32_t)((n - n1) * kHeadDim * 2))
                 : "memory");
}

// Window chunks [i0, i1) of one pair (chunk u = tokens Lq + 32 u ...), staged
// in the warp's (idle) ring; *phase_io is the parity count of the warp's
// staging barrier, kept across calls.  A bounded wait that gives up sets
// KVQ_FLAG_WAIT_TIMEOUT and ends the chunks.
// Out of line, like tc_packed_warp.
template <int BK, int BV, bool kWide>
__device__ __noinline__ TcState tc_window_chunks(TcState st, const Dims d, const __half* ring_k,
                                                 const __half* ring_v, int Lq, int L, int i0,
                                                 int i1, char* area, const __half* qh, int gq,
                                                 float scale_log2, int p_new,
                                                 const __half* k_row, const __half* v_row,
                                                 uint64_t* bar, uint32_t* phase_io,
                                                 unsigned* flag) {
  uint32_t phase = *phase_io;
  const int lane = threadIdx.x & 31;
  const Lane ln = make_lane<BK, BV>(lane);
  uint32_t qb[16];
  load_qb<false, kWide>(qb, qh, gq, ln);
  __half* rows = reinterpret_cast<__half*>(area);
  for (int u = i0; u < i1; ++u) {
    const int p0 = Lq + u * kGroup;
    const int n_tok = min(kGroup, L - p0);
    uint32_t pt[1][2][2], pl[1][2][2];
    if (!stage_rows_bulk(rows, ring_k, p0, n_tok, d.ring, p_new, k_row, bar, phase++ & 1u)) {
      if (lane == 0) atomicOr(flag, KVQ_FLAG_WAIT_TIMEOUT);
      break;
    }
    tc_resid_scores<kWide, BV == 1>(rows, n_tok, qb, ln, scale_log2, st, pt, pl);
    __syncwarp();
    if (!stage_rows_bulk(rows, ring_v, p0, n_tok, d.ring, p_new, v_row, bar, phase++ & 1u)) {
      if (lane == 0) atomicOr(flag, KVQ_FLAG_WAIT_TIMEOUT);
      break;
    }
    tc_resid_values<kWide, BV == 1>(rows, pt, pl, st);
    __syncwarp();
  }
  *phase_io = phase;
  return st;
}


// Inverse of tc_write_state<false>: a WarpState (natural channel order) back
// into registers in the window layout (channel = 16 m-tile + row, no
// zero-point term), so the window chunks of a pair continue the state its
// packed blocks began.  Row sums go to the lanes of gid 0.
template <bool kWide>
__device__ __forceinline__ void tc_read_state(TcState& st, const WarpState& ws, int lane) {
  const int gid = lane >> 2, tig = lane & 3;
  const bool keep = kWide || tig < 2;  // narrow: lanes tig and tig^2 share heads
#pragma unroll
  for (int hh = 0; hh < 2; ++hh) {
    const int head = 2 * (kWide ? tig : (tig & 1)) + hh;
    st.m[hh] = ws.m[head];
    st.l[hh] = gid == 0 ? ws.l[head] : 0.0f;
  }
#pragma unroll
  for (int mtp = 0; mtp < 8; ++mtp)
#pragma unroll
    for (int rh = 0; rh < 2; ++rh)
#pragma unroll
      for (int hh = 0; hh < 2; ++hh) {
        const int head = 2 * (kWide ? tig : (tig & 1)) + hh;
        st.acc[mtp][2 * rh + hh] = keep ? ws.o[head][16 * mtp + gid + 8 * rh] : 0.0f;
      }
#pragma unroll
  for (int r = 0; r < 4; ++r) st.zv[r] = 0.0f;
}

// Global partial slots: CTA partials [0, n_cta_slots + P), then one warp
// partial per pair.  Each holds m[gq], l[gq], o[gq][128] (Ws arrays).
__device__ __forceinline__ long long warp_slot(int ctas, int P, int p) {
  return (long long)ctas + P + p;
}

// A pair whose partials this CTA completed (final merge at the end), or a
// warp's final state.
struct SegRec {
  long long U;      // first cost unit of the pair
  int p, pc, nb, nr, f;
};

// Row o / l of every head of a WarpState into out (a pair's only partial).
__device__ __forceinline__ void warp_state_out(const WarpState& s, void* out, int out_f16,
                                               long long head0, int gq, int lane) {
  for (int i = lane; i < gq * kHeadDim; i += 32) {
    const int g = i / kHeadDim, ch = i % kHeadDim;
    const float l = s.l[g];
    store_out(out, out_f16, (head0 + g) * kHeadDim + ch, l > 0.0f ? s.o[g][ch] / l : 0.0f);
  }
}

// The final merge of pair p: its partials are the CTA slots [c_a + p,
// c_a + p + n_cta) and, if cont, its warp slot.  All threads of the CTA; the
// partials are copied into shared memory (`scratch`, the idle rings, of
// scratch_bytes) with one round of independent loads when they fit.
__device__ void final_merge(const SegRec& r, const FlatGrid& g, const Dims& d, const Ws& ws,
                            void* out, int out_f16, float* scratch, size_t scratch_bytes) {
  const int P = d.batch * d.hkv, gq = d.gq;
  int c_a, n_cta;
  bool cont;
  const int cnt = pair_partials(r.U, r.pc, r.nb, r.nr, r.f, g, c_a, n_cta, cont);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int rows = gq * kHeadDim;                  // floats of one partial's rows
  float* wv = scratch;                             // [gq][cnt] maxima, then weights
  float* lv = wv + gq * cnt;                       // [gq][cnt] sums
  float* lsum = lv + gq * cnt;                     // [gq]
  float* osm = scratch + ((2 * gq * cnt + gq + 3) / 4) * 4;  // [cnt][gq][128], 16-byte aligned
  const bool staged = ((size_t)(osm - scratch) + (size_t)cnt * rows) * 4 <= scratch_bytes;
  const long long s0 = (long long)c_a + r.p;       // first CTA slot
  const long long sw = warp_slot(gridDim.x, P, r.p);
  auto slot = [&](int k) -> long long { return k < n_cta ? s0 + k : sw; };
  for (int i = threadIdx.x; i < gq * cnt; i += kThreads) {
    const int gg = i / cnt, k = i % cnt;
    wv[i] = __ldcg(ws.m + slot(k) * gq + gg);
    lv[i] = __ldcg(ws.l + slot(k) * gq + gg);
  }
  if (staged) {
    const float4* src = reinterpret_cast<const float4*>(ws.o + s0 * rows);
    float4* dst = reinterpret_cast<float4*>(osm);
    const int n4 = n_cta * rows / 4;
    for (int i = threadIdx.x; i < n4; i += kThreads) dst[i] = __ldcg(src + i);
    if (cont) {
      const float4* sw4 = reinterpret_cast<const float4*>(ws.o + sw * rows);
      for (int i = threadIdx.x; i < rows / 4; i += kThreads) dst[n4 + i] = __ldcg(sw4 + i);
    }
  }
  __syncthreads();
  for (int gg = warp; gg < gq; gg += kWarps) {
    float M = -INFINITY;
    for (int k = lane; k < cnt; k += 32) M = fmaxf(M, wv[gg * cnt + k]);
    M = warp_max(M);
    float Ls = 0.0f;
    for (int k = lane; k < cnt; k += 32) {
      const float m = wv[gg * cnt + k];
      const float w = (m == -INFINITY) ? 0.0f : exp2f(m - M);
      Ls += w * lv[gg * cnt + k];
      wv[gg * cnt + k] = w;
    }
    Ls = warp_sum(Ls);
    if (lane == 0) lsum[gg] = Ls;
  }
  __syncthreads();
  const long long head0 = (long long)(r.p / d.hkv) * d.hq + (long long)(r.p % d.hkv) * gq;
  for (int it = threadIdx.x; it < rows; it += kThreads) {
    const int gg = it / kHeadDim;
    float o = 0.0f;
    if (staged) {
      for (int k = 0; k < cnt; ++k) o = fmaf(wv[gg * cnt + k], osm[k * rows + it], o);
    } else {
      for (int k = 0; k < cnt; ++k) o = fmaf(wv[gg * cnt + k], __ldcg(ws.o + slot(k) * rows + it), o);
    }
    const float Ls = lsum[gg];
    store_out(out, out_f16, head0 * kHeadDim + it, Ls > 0.0f ? o / Ls : 0.0f);
  }
  if (threadIdx.x == 0) ws.tk[r.p] = 0u;
  __syncthreads();
}


// A warp's walk over its pairs and the segment it is folding, in shared
// memory.
struct WarpCtx {
  Walk w;                        // the pair the walk is at
  SegRec seg;                    // the segment being folded
  long long a, e;                // the warp's unit range
  int i0, i1;                    // the segment's window chunks
  int last, last_v;              // the segment ends the range; last virtual warp
  int pre, pre_end, lo_h, p_h;   // early copies: count, end block, first block, pair
  int pos;                       // ring slots used
  uint32_t wphase;               // window staging barrier parity count
  int j1;                        // the segment's end block
};

// ---------------------------------------------------------------------------
// The kernel
// ---------------------------------------------------------------------------

template <int BK, int BV, bool kWide>
__global__ void __launch_bounds__(kThreads, kCtasPerSm)
    decode_attn_kernel(Dims d, kvq_cache c, const __half* __restrict__ q, void* __restrict__ out,
                       int out_f16, float scale_log2, unsigned smem_size, Ws ws,
                       const __half* __restrict__ k_new, const __half* __restrict__ v_new) {
  extern __shared__ __align__(128) unsigned char smem[];
  __shared__ MergeSmall ms;
  __shared__ __align__(8) uint64_t wbar[kWarps];  // a warp's window-row staging barrier
  __shared__ SegRec rec[kWarps];                  // each warp's final state (p < 0: none)
  __shared__ SegRec fin[kFinCap];                 // pairs whose partials this CTA completed
  __shared__ int fin_n;
  __shared__ int pub_last;
  __shared__ WarpCtx wctx[kWarps];                // each warp's walk and segment
  __shared__ FlatGrid grid_s;                     // the plan's grid
  __shared__ int len_s[kLenCap];                  // the lengths the plan reads (batch <= kLenCap)
  __shared__ MergeGroups mg;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  pdl_launch_dependents();
  const bool append = k_new != nullptr;
  const int P = d.batch * d.hkv, gq = d.gq;
  constexpr int page = page_bytes_c(BK, BV);
  constexpr int R = ring_slots(page);
  const int wbytes = warp_ring_bytes(page);
  char* ring = reinterpret_cast<char*>(smem) + (size_t)warp * wbytes;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + (size_t)kWarps * wbytes) + warp * R;
  // 512 bytes at the end of shared memory: metadata rows of the zero-point
  // MMAs that carry no block, all zero except bytes 256..319, which only the
  // value zero-point MMA's row 4 reads: fp16 ones, so that row sums the
  // softmax weights (the row sum l).
  unsigned* zero = reinterpret_cast<unsigned*>(smem + smem_size - 16 - kZeroBytes);
  for (int i = threadIdx.x; i < kZeroBytes / 4; i += kThreads)
    zero[i] = i >= kOnesWord0 && i < kOnesWord0 + 16 ? 0x3C003C00u : 0u;
  unsigned* flag = reinterpret_cast<unsigned*>(c.seq_len) + d.batch;
  if (threadIdx.x == 0) fin_n = 0;
  if (lane == 0) {
    for (int i = 0; i < R; ++i) mbar_init(full + i, 1);
    mbar_init(&wbar[warp], 1);
    fence_mbar_init();
    rec[warp].p = -1;
  }
  __syncwarp();

  WarpCtx& X = wctx[warp];
  if (lane == 0) {
    X.pre = 0;
    X.pre_end = 0;
    X.lo_h = -1;
    X.p_h = -1;
    X.pos = 0;
    X.wphase = 0u;
    X.last = 0;
  }
  __syncwarp();
  // The plan reads the lengths many times: one coalesced read into shared
  // memory after the dependency wait instead of global round trips.  (No
  // copies are started before the wait: the next CTA of an SM starts only
  // when the previous kernel's CTA there has left, so little would overlap,
  // and the reads after the wait would queue behind them.)
  const int* lens = d.batch <= kLenCap ? len_s : c.seq_len;
  __syncthreads();  // zero rows written
  pdl_wait();

  // ---- the plan from the lengths after the wait ----
  // (kept in shared memory: it is needed again only after the streaming)
  if (d.batch <= kLenCap)
    for (int b = threadIdx.x; b < d.batch; b += kThreads) len_s[b] = read_len(c.seq_len + b);
  __syncthreads();
  {
    const FlatGrid g0 = flat_grid(plan_sums(lens, d, append), gridDim.x);
    if (threadIdx.x == 0) grid_s = g0;
  }
  __syncthreads();
  const FlatGrid& g = grid_s;
  if (g.N == 0 && blockIdx.x == 0 && warp == 0)
    for (int i = lane; i < P * gq * kHeadDim; i += 32) store_out(out, out_f16, i, 0.0f);
  // Early copies still in flight that no packed range consumed land before
  // the ring is used otherwise (bounded waits).
  auto drain_pre = [&]() {
    const int pre = X.pre;
    if (pre > 0) {
      if (lane == 0) {
        for (int s = 0; s < pre; ++s) mbar_wait(full + s % R, (s / R) & 1);
        X.pos = pre;
        X.pre = 0;
      }
      __syncwarp();
    }
  };
  // A state the warp leaves for the next pair: its pair's only partial goes
  // out directly, any other to the warp slot and the pair's ticket.
  auto emit_warp_partial = [&](const TcState& st, bool packed_kind, const SegRec& r,
                               long long head0) {
    int c_a, n_cta;
    bool cont;
    const int cnt = pair_partials(r.U, r.pc, r.nb, r.nr, r.f, g, c_a, n_cta, cont);
    WarpState& s = *reinterpret_cast<WarpState*>(ring);
    if (packed_kind) tc_write_state<true, BV, kWide>(st, s, lane);
    else tc_write_state<false, BV, kWide>(st, s, lane);
    __syncwarp();
    if (cnt == 1) {
      warp_state_out(s, out, out_f16, head0, gq, lane);
    } else {
      const long long sl = warp_slot(gridDim.x, P, r.p);
      for (int i = lane; i < gq * kHeadDim; i += 32)
        ws.o[sl * gq * kHeadDim + i] = s.o[i / kHeadDim][i % kHeadDim];
      if (lane < gq) {
        ws.m[sl * gq + lane] = s.m[lane];
        ws.l[sl * gq + lane] = s.l[lane];
      }
      __threadfence();
      __syncwarp();
      if (lane == 0 && atom_add_acq_rel(&ws.tk[r.p], 1u) == (unsigned)cnt - 1u) {
        const int i = atomicAdd(&fin_n, 1);
        if (i < kFinCap) fin[i] = r;
      }
    }
    __syncwarp();
  };

  // The walk and the current segment live in shared memory (X): nothing of
  // them holds registers across the streaming loop, which gets them all.
  const int v = (int)blockIdx.x < g.n_cta ? cta_first_v(blockIdx.x, g) + warp : -1;
  if (v >= 0 && v < cta_first_v(blockIdx.x + 1, g)) {
    {
      const long long a = v_first_unit(v, g);
      const Walk w0 = walk_start(a, lens, d, append, g.k);
      if (lane == 0) {
        X.w = w0;
        X.a = a;
        X.e = v_first_unit(v + 1, g);
        X.last_v = v == g.n_v - 1;
      }
      __syncwarp();
    }
    for (;;) {
      Walk w = X.w;
      if (w.b >= d.batch) break;
      const long long a = X.a, e = X.e;
      const bool last_v = X.last_v;
      const long long U = w.Ub + (long long)w.h * w.pc;
      const int p = w.b * d.hkv + w.h;
      const long long head0 = (long long)w.b * d.hq + (long long)w.h * gq;
      // empty pairs: zero output from the warp whose range holds their unit
      // (the last warp takes those at the very end)
      if (U >= e && !(last_v && U >= g.N)) break;
      if (w.pc == 0) {
        if (U >= a)
          for (int i = lane; i < gq * kHeadDim; i += 32) store_out(out, out_f16, head0 * kHeadDim + i, 0.0f);
        walk_next(w, lens, d, append, g.k);
        __syncwarp();
        if (lane == 0) X.w = w;
        __syncwarp();
        continue;
      }
      const PairShape s = pair_shape(w.L, d.residual);
      const int k0 = items_below(a - U, s.nb, s.nr, g.k, w.f);
      const int k1 = items_below(e - U, s.nb, s.nr, g.k, w.f);
      if (lane == 0) X.last = U + w.pc >= e;
      __syncwarp();
      if (k1 > k0) {
        const int j0 = min(k0, s.nb), j1 = min(k1, s.nb);
        const int i0 = max(k0 - s.nb, 0), i1 = max(k1 - s.nb, 0);
        const long long bh = (long long)w.b * d.hkv + w.h;
        const __half* ring_k = reinterpret_cast<const __half*>(c.k_resid) + bh * d.ring * kHeadDim;
        const __half* ring_v = reinterpret_cast<const __half*>(c.v_resid) + bh * d.ring * kHeadDim;
        const bool grew = w.L > w.L0;  // this kernel appends the token at position L0
        if (grew && k0 == 0) {  // the new token into its ring slot
          const long long sl = (long long)(w.L0 % d.ring) * kHeadDim;
          __half* rk = const_cast<__half*>(ring_k) + sl;
          __half* rv = const_cast<__half*>(ring_v) + sl;
          if (lane < 16) reinterpret_cast<uint4*>(rk)[lane] = reinterpret_cast<const uint4*>(k_new + bh * kHeadDim)[lane];
          else reinterpret_cast<uint4*>(rv)[lane - 16] = reinterpret_cast<const uint4*>(v_new + bh * kHeadDim)[lane - 16];
        }
        if (i1 > i0 && lane == 0) {
          // window rows into L2 while the packed blocks stream (a hint; the
          // newest row is not written yet)
          const int p0 = s.Lq + i0 * kGroup;
          const int n = min(w.L, s.Lq + i1 * kGroup) - (grew ? 1 : 0) - p0;
          if (n > 0) {
            prefetch_rows_l2(ring_k, p0, n, d.ring);
            prefetch_rows_l2(ring_v, p0, n, d.ring);
          }
        }
        if (lane == 0) {
          X.seg.U = U;
          X.seg.p = p;
          X.seg.pc = w.pc;
          X.seg.nb = s.nb;
          X.seg.nr = s.nr;
          X.seg.f = w.f;
          X.i0 = i0;
          X.i1 = i1;
          X.j1 = j1;
        }
        __syncwarp();
        TcState st;
        init_state(st);
        if (j1 > j0) {
          // the early slots (ring positions 0 .. pre - 1) are this range's
          // first ones if it begins where the early plan's did; a block that
          // leaves the window in this kernel folds after the streamed ones
          const bool flush = grew && s.Lq > packed_len(w.L0, d.residual) && j1 == s.nb;
          const char* tail = nullptr;
          st = tc_packed_warp<BK, BV, kWide>(st, page_map(d, c, w.b, w.h), p == X.p_h ? X.lo_h : -1,
                                             X.pre, X.pre_end, j0, flush ? j1 - 1 : j1, ring, full,
                                             &X.pos, reinterpret_cast<const char*>(zero),
                                             q + head0 * kHeadDim, gq, scale_log2, flag, flush,
                                             &tail);
          __syncwarp();
          if (lane == 0) X.pre = 0;
          __syncwarp();
          {
            // the flush (segment read back from X)
            const Walk wf = X.w;
            const PairShape sf = pair_shape(wf.L, d.residual);
            if (wf.L > wf.L0 && sf.Lq > packed_len(wf.L0, d.residual) && X.j1 == sf.nb) {
              const long long bhf = (long long)wf.b * d.hkv + wf.h;
              st = tc_fold_flush<BK, BV, kWide>(
                  st, page_map(d, c, wf.b, wf.h), sf.nb - 1, tail, ring,
                  reinterpret_cast<const char*>(zero),
                  q + ((long long)wf.b * d.hq + (long long)wf.h * gq) * kHeadDim, gq, scale_log2,
                  flag, reinterpret_cast<const __half*>(c.k_resid) + bhf * d.ring * kHeadDim,
                  reinterpret_cast<const __half*>(c.v_resid) + bhf * d.ring * kHeadDim, d.ring);
            }
          }
          if (X.i1 > X.i0) {
            // the window chunks continue this state in their own layout
            WarpState& t = *reinterpret_cast<WarpState*>(ring);
            tc_write_state<true, BV, kWide>(st, t, lane);
            __syncwarp();
            tc_read_state<kWide>(st, t, lane);
            __syncwarp();
          }
        }
        // everything below reads the segment back from X
        const SegRec r = X.seg;
        const Walk wr = X.w;
        const bool has_w = X.i1 > X.i0;
        if (has_w) {
          drain_pre();
          const long long bh2 = (long long)wr.b * d.hkv + wr.h;
          const PairShape s2 = pair_shape(wr.L, d.residual);
          const bool grew2 = wr.L > wr.L0;
          st = tc_window_chunks<BK, BV, kWide>(
              st, d, reinterpret_cast<const __half*>(c.k_resid) + bh2 * d.ring * kHeadDim,
              reinterpret_cast<const __half*>(c.v_resid) + bh2 * d.ring * kHeadDim, s2.Lq, wr.L,
              X.i0, X.i1, ring, q + ((long long)wr.b * d.hq + (long long)wr.h * gq) * kHeadDim, gq,
              scale_log2, grew2 ? wr.L0 : -1, grew2 ? k_new + bh2 * kHeadDim : nullptr,
              grew2 ? v_new + bh2 * kHeadDim : nullptr, &wbar[warp], &X.wphase, flag);
        }
        drain_pre();
        if (X.last) {
          WarpState& t = *reinterpret_cast<WarpState*>(ring);
          if (!has_w) tc_write_state<true, BV, kWide>(st, t, lane);
          else tc_write_state<false, BV, kWide>(st, t, lane);
          if (lane == 0) rec[warp] = r;
        } else {
          emit_warp_partial(st, !has_w, r,
                            (long long)(r.p / d.hkv) * d.hq + (long long)(r.p % d.hkv) * gq);
        }
      }
      {
        Walk wn = X.w;
        const bool stop = X.last && !X.last_v;
        walk_next(wn, lens, d, append, g.k);
        __syncwarp();
        if (lane == 0) X.w = wn;
        __syncwarp();
        if (stop) break;
      }
    }
  }
  drain_pre();
  __syncthreads();

  // ---- merge the warps of this CTA that end in the same pair ----
  // Groups are runs of warps with the same final pair (warp order is unit
  // order).  All groups merge at once, then their tickets go out together.
  const size_t wstride = (size_t)wbytes;
  auto wstate = [&](int w) -> const WarpState& {
    return *reinterpret_cast<const WarpState*>(smem + (size_t)w * wstride);
  };
  if (warp == 0) {  // groups from two ballots over the warps' final pairs
    const int p = lane < kWarps ? rec[lane].p : -1;
    const int prev = lane > 0 && lane < kWarps ? rec[lane - 1].p : -2;
    const int next = lane + 1 < kWarps ? rec[lane + 1].p : -2;
    const unsigned starts = __ballot_sync(0xffffffffu, p >= 0 && prev != p);
    const unsigned ends = __ballot_sync(0xffffffffu, p >= 0 && next != p);
    const unsigned below = (1u << lane) - 1u;
    if (starts & (1u << lane)) mg.w0[__popc(starts & below)] = lane;
    if (ends & (1u << lane)) mg.w1[__popc(ends & below)] = lane + 1;
    if (lane == 0) mg.n = __popc(starts);
  }
  __syncthreads();
  const int ng = mg.n;
  if (threadIdx.x < ng) {  // a group's partial count, once (64-bit divisions)
    const SegRec r = rec[mg.w0[threadIdx.x]];
    int c_a, n_cta;
    bool cont;
    mg.cnt[threadIdx.x] = pair_partials(r.U, r.pc, r.nb, r.nr, r.f, g, c_a, n_cta, cont);
  }
  if (threadIdx.x < ng * gq) {  // (group, head): maximum and warp weights
    const int k = threadIdx.x / gq, gg = threadIdx.x - k * gq;
    const int w0 = mg.w0[k], w1 = mg.w1[k];
    float mw[kWarps];
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) {  // independent loads, then the maximum
      mw[w] = w >= w0 && w < w1 ? wstate(w).m[gg] : -INFINITY;
      M = fmaxf(M, mw[w]);
    }
#pragma unroll
    for (int w = 0; w < kWarps; ++w)
      if (w >= w0 && w < w1) ms.ww[w][gg] = mw[w] == -INFINITY ? 0.0f : fast_exp2(mw[w] - M);
    ms.gm[k][gg] = M;
  }
  __syncthreads();
  for (int it = threadIdx.x; it < ng * gq * kHeadDim; it += kThreads) {
    const int ch = it & (kHeadDim - 1), kg = it >> 7;  // kHeadDim == 128
    const int k = kg / gq, gg = kg - k * gq;
    const int w0 = mg.w0[k], w1 = mg.w1[k];
    float o = 0.0f, l = 0.0f;
    for (int w = w0; w < w1; ++w) {
      const float wt = ms.ww[w][gg];
      o = fmaf(wt, wstate(w).o[gg][ch], o);
      l = fmaf(wt, wstate(w).l[gg], l);
    }
    const int pp = rec[w0].p;
    if (mg.cnt[k] == 1) {
      const long long head0 = (long long)(pp / d.hkv) * d.hq + (long long)(pp % d.hkv) * gq;
      store_out(out, out_f16, (head0 + gg) * kHeadDim + ch, l > 0.0f ? o / l : 0.0f);
    } else {
      const long long sl = (long long)blockIdx.x + pp;
      ws.o[(sl * gq + gg) * kHeadDim + ch] = o;
      if (ch == 0) {
        ws.m[sl * gq + gg] = ms.gm[k][gg];
        ws.l[sl * gq + gg] = l;
      }
    }
  }
  __syncthreads();
  if (threadIdx.x < ng && mg.cnt[threadIdx.x] > 1) {
    const SegRec r = rec[mg.w0[threadIdx.x]];
    __threadfence();  // cumulativity: the CTA's partial rows before the ticket
    if (atom_add_acq_rel(&ws.tk[r.p], 1u) == (unsigned)mg.cnt[threadIdx.x] - 1u) {
      const int i = atomicAdd(&fin_n, 1);
      if (i < kFinCap) fin[i] = r;
    }
  }
  __syncthreads();

  // ---- final merges of the pairs whose last partial came from this CTA ----
  const int nf = min(fin_n, kFinCap);
  for (int i = 0; i < nf; ++i)
    final_merge(fin[i], g, d, ws, out, out_f16, reinterpret_cast<float*>(smem),
                (size_t)kWarps * wbytes);

  // ---- the decode step publishes the new lengths once every CTA is done ----
  if (append) {
    __syncthreads();
    if (threadIdx.x == 0) {
      __threadfence();
      pub_last = atom_add_acq_rel(&ws.tk[P], 1u) == gridDim.x - 1u;
    }
    __syncthreads();
    if (pub_last) {
      for (int b = threadIdx.x; b < d.batch; b += kThreads) {
        const int L0 = read_len(c.seq_len + b);
        if (L0 < d.max_len) c.seq_len[b] = L0 + 1;
        else atomicOr(flag, (unsigned)KVQ_FLAG_OVERFLOW);
      }
      if (threadIdx.x == 0) ws.tk[P] = 0u;
    }
  }
}

size_t smem_bytes(const Dims& d) {
  const int page = (int)d.page_bytes;
  const size_t rings = (size_t)kWarps * warp_ring_bytes(page) +
                       (size_t)kWarps * ring_slots(page) * sizeof(uint64_t);
  // + the zero rows of the zero-point MMAs
  return (rings + kZeroBytes + 16 + 127) / 128 * 128;
}

template <int BK, int BV, bool kWide>
cudaError_t prepare(const Dims& d) {
  return cudaFuncSetAttribute(decode_attn_kernel<BK, BV, kWide>,
                              cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_bytes(d));
}

// Kernel instance for (bits_k, bits_v, query-group width): groups of up to 4
// heads take the narrow MMA layout, 5..8 heads the wide one.
template <int BK, int BV, typename Op>
cudaError_t dispatch_width(const Dims& d, const Op& op) {
  return d.gq <= 4 ? op.template run<BK, BV, false>() : op.template run<BK, BV, true>();
}
template <int BK, typename Op>
cudaError_t dispatch_bv(const Dims& d, const Op& op) {
  switch (d.bits_v) {
    case 1: return dispatch_width<BK, 1>(d, op);
    case 2: return dispatch_width<BK, 2>(d, op);
    case 4: return dispatch_width<BK, 4>(d, op);
    default: return dispatch_width<BK, 8>(d, op);
  }
}
template <typename Op>
cudaError_t dispatch(const Dims& d, const Op& op) {
  switch (d.bits_k) {
    case 1: return dispatch_bv<1>(d, op);
    case 2: return dispatch_bv<2>(d, op);
    case 4: return dispatch_bv<4>(d, op);
    default: return dispatch_bv<8>(d, op);
  }
}

struct LaunchOp {
  const Dims& d;
  const kvq_cache& c;
  const __half* q;
  void* out;
  int out_f16;
  float sl2;
  int S;
  const Ws& ws;
  cudaStream_t st;
  const __half* k_new = nullptr;
  const __half* v_new = nullptr;
  template <int BK, int BV, bool kWide>
  cudaError_t run() const {
    cudaError_t e = prepare<BK, BV, kWide>(d);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(S);  // the flat plan's CTAs
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem_bytes(d);
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, decode_attn_kernel<BK, BV, kWide>, d, c, q, out, out_f16, sl2,
                           (unsigned)smem_bytes(d), ws, k_new, v_new);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
  }
};

// Bounded-wait self-test: one warp arms an mbarrier for 16 bytes that no copy
// delivers and waits on it with the given cycle limit, the same loop the
// attention kernel's copy waits use.  The wait gives up, the kernel sets
// KVQ_FLAG_WAIT_TIMEOUT in *flag and returns (no copy is in flight).
__global__ void __launch_bounds__(32) wait_selftest_kernel(unsigned* flag, long long limit) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    fence_mbar_init();
    mbar_expect_tx(&bar, 16u);  // the arrival; 16 bytes stay pending
  }
  __syncwarp();
  const bool ok = __all_sync(0xffffffffu, mbar_wait_for(&bar, 0u, limit));
  if (!ok && threadIdx.x == 0) atomicOr(flag, (unsigned)KVQ_FLAG_WAIT_TIMEOUT);
}

}  // namespace

cudaError_t launch_wait_selftest(unsigned* flag, long long limit_cycles, cudaStream_t st) {
  wait_selftest_kernel<<<1, 32, 0, st>>>(flag, limit_cycles);
  return cudaGetLastError();
}

// The flat plan on `ctas` CTAs: partial slots for the launch's CTAs and the
// pairs (the same carve the kernel uses), one ticket per pair and the decode
// step's count of finished CTAs.
size_t attn_workspace_bytes(const Dims& d, int ctas) {
  const size_t nml = ws_slots(d.batch, d.hkv, ctas) * (size_t)d.gq;
  return align256(nml * 4) * 2 + align256(nml * kHeadDim * 4) +
         align256(((size_t)d.batch * d.hkv + 1) * 4);
}

cudaError_t launch_decode_attn(const Dims& d, const kvq_cache& c, const __half* q, void* out,
                               int out_f16, float scale_log2, int ctas, void* workspace,
                               cudaStream_t st) {
  const Ws ws = carve(workspace, d.batch, d.hq, d.hkv, ctas);
  return dispatch(d, LaunchOp{d, c, q, out, out_f16, scale_log2, ctas, ws, st});
}

cudaError_t launch_decode_step(const Dims& d, const kvq_cache& c, const __half* k_new,
                               const __half* v_new, const __half* q, void* out, int out_f16,
                               float scale_log2, int ctas, void* workspace, cudaStream_t st) {
  const Ws ws = carve(workspace, d.batch, d.hq, d.hkv, ctas);
  LaunchOp op{d, c, q, out, out_f16, scale_log2, ctas, ws, st};
  op.k_new = k_new;
  op.v_new = v_new;
  return dispatch(d, op);
}

// CTAs of a flat-plan launch: one per resident CTA slot of the GPU.
int attn_flat_ctas(int sm_count) {
  const int n = kCtasPerSm * sm_count;
  return n > kMaxSplits - 1 ? kMaxSplits - 1 : (n < 1 ? 1 : n);
}

// Split plan: CTAs per (sequence, kv-head) so that every resident CTA slot
// of the GPU holds one, with at least a few blocks per CTA.
int attn_default_splits(const Dims& d, int sm_count) {
  const int bh = d.batch * d.hkv;
  int n = kCtasPerSm * sm_count / bh;
  const int cap = (d.max_blocks + 3) / 4;
  if (n > cap) n = cap;
  if (n > kMaxSplits - 1) n = kMaxSplits - 1;
  return n < 1 ? 1 : n;
}

// The plan for host-known lengths: the split plan (its count) when one wave
// of its CTAs fills the GPU, as for batch-1 decoding, where a launch is bound
// by latency;
// otherwise 0, the flat plan, which streams every warp's share in one wave
// instead of paying a CTA's start and merges once per wave (Qwen2.5-14B
// shape, batch 8 x 64k, K1V1: 98.7 against 104.2 us per layer with 7 splits
// in 2.95 waves).
int attn_splits_for_lengths(const Dims& d, int sm_count, const int32_t* lengths) {
  (void)lengths;
  const long long bh = (long long)d.batch * d.hkv;
  const int S = attn_default_splits(d, sm_count);
  return (long long)S * bh * 10 >= 9LL * kCtasPerSm * sm_count ? S : 0;  // one wave, >= 90% full
}

// ---------------------------------------------------------------------------
// Decode attention without caller-supplied scratch (kvq_decode_attn_noalloc).
//
// Some callers cannot allocate device memory where they run a decode step: a
// host framework whose pool owns every byte of the GPU (a raw allocation would
// fail or fragment it), or a serving loop that must not allocate per step.
// For them the split partials and tickets live in this one file-scope device
// array of fixed size, which every GPU that loads the library holds until the
// process exits.  All calls share it, so calls that overlap on the GPU race.
// ---------------------------------------------------------------------------

namespace {
constexpr size_t kStaticScratchBytes = size_t(4) << 20;  // 4 MiB
constexpr int kMaxDevices = 64;
__device__ __align__(256) unsigned char g_attn_scratch[kStaticScratchBytes];

// Device address of g_attn_scratch on the current device, looked up once per
// device with that device current.  In host code the symbol is only a
// host-side stand-in: passing it to a kernel would fault or silently use the
// wrong memory, so only the looked-up address is ever used.
cudaError_t static_scratch(void** out) {
  static std::mutex mu;
  static void* addr[kMaxDevices] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(mu);
  if (!addr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_attn_scratch);
    if (e != cudaSuccess) return e;
    addr[dev] = p;
  }
  *out = addr[dev];
  return cudaSuccess;
}
}  // namespace

size_t attn_static_scratch_bytes() { return kStaticScratchBytes; }

cudaError_t launch_decode_attn_static(const Dims& d, const kvq_cache& c, const __half* q,
                                      float* out, float scale_log2, int n_splits,
                                      cudaStream_t st) {
  void* ws = nullptr;
  cudaError_t e = static_scratch(&ws);
  if (e != cudaSuccess) return e;
  // The array keeps the previous call's contents: the tickets must start at
  // zero, the partials are always written before they are read.  n_splits >
  // 0: the split plan (attn_split.cu); < 0: the flat plan on -n_splits CTAs.
  if (n_splits > 0) {
    size_t tk_bytes = 0;
    unsigned* tk = attn_split_tickets(d, n_splits, ws, &tk_bytes);
    e = cudaMemsetAsync(tk, 0, tk_bytes, st);
    if (e != cudaSuccess) return e;
    return launch_decode_attn_split(d, c, q, out, 0, scale_log2, n_splits, ws, st);
  }
  const Ws w = carve(ws, d.batch, d.hq, d.hkv, -n_splits);
  e = cudaMemsetAsync(w.tk, 0, ((size_t)d.batch * d.hkv + 1) * sizeof(unsigned), st);
  if (e != cudaSuccess) return e;
  return launch_decode_attn(d, c, q, out, 0, scale_log2, -n_splits, ws, st);
}

}  // namespace kvq
