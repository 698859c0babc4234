// kvq_decode_attn / kvq_decode_step, the split plan (n_splits > 0): one
// decode step of grouped-query attention softmax(q K^T * scale) V (Sec. 1 of
// the paper) over the packed KbVb cache.  (The flat plan, n_splits = 0, is
// attn.cu: it shares the per-block arithmetic and runs multi-wave workloads
// in one wave; this plan is the one for launches that fit one wave, such as
// batch-1 decoding.)
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


struct Ws {
  float* m;       // [B][Hq][S]
  float* l;       // [B][Hq][S]
  float* o;       // [B][Hq][S][128]
  unsigned* tk;   // [B][Hkv] (sized [B][Hq])
};

__host__ __device__ inline size_t align256(size_t x) { return (x + 255) / 256 * 256; }

__host__ __device__ inline Ws carve(void* base, int batch, int hq, int hkv, int S) {
  Ws w;
  char* p = static_cast<char*>(base);
  const size_t nml = (size_t)batch * hq * S;
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
  float cta_m[kHeads];
  int last;
};

// A 16-byte asynchronous copy (q into shared memory).
__device__ __forceinline__ void cp_async16(void* dst, const void* src, uint32_t src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_addr(dst)), "l"(src),
               "r"(src_bytes)
               : "memory");
}

// Shared-memory page image of a block that leaves the window (decode step).
__host__ __device__ constexpr int image_bytes(int page) { return (page + 127) / 128 * 128; }

// ---------------------------------------------------------------------------
// Work of one (sequence, kv-head): nb packed blocks and n_res window chunks
// over NV warps.  The last n_resw warps take the window chunks (strided), the
// other np warps contiguous block ranges whose sizes differ by at most one.
// ---------------------------------------------------------------------------

struct Plan {
  int Lq, nb, n_res, n_resw, np;
};

__host__ __device__ inline Plan make_plan(int L, int residual, int NV) {
  Plan p;
  p.Lq = packed_len(L, residual);
  p.nb = p.Lq / kGroup;
  p.n_res = (L - p.Lq + kGroup - 1) / kGroup;
  const int cap = p.nb == 0 ? NV : (NV / 4 > 1 ? NV / 4 : 1);
  p.n_resw = p.n_res < cap ? p.n_res : cap;
  p.np = NV - p.n_resw;
  return p;
}

// Blocks [lo, hi) of packed warp v (v < np), in 32-bit arithmetic while
// (v + 1) * nb fits (v < 4096 warps).
__host__ __device__ inline void block_range(const Plan& p, int v, int& lo, int& hi) {
  if (p.nb < (1 << 20)) {
    lo = (int)((unsigned)v * (unsigned)p.nb / (unsigned)p.np);
    hi = (int)((unsigned)(v + 1) * (unsigned)p.nb / (unsigned)p.np);
  } else {
    lo = (int)((long long)v * p.nb / p.np);
    hi = (int)((long long)(v + 1) * p.nb / p.np);
  }
}


__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
}

// Fold blocks [lo, hi) into st; `pre` slots holding blocks [lo_h, pre_end)
// were streamed early.
// Fold blocks [lo, hi) into st; `pre` slots holding blocks [lo_h, pre_end)
// were streamed early.
template <int BK, int BV, bool kWide>
__device__ void tc_packed_warp(const PageMap& pm, TableWin& tw, int lo_h, int pre, int pre_end,
                               int lo, int hi_all, char* ring, uint64_t* full, int R,
                               const char* zero, const __half* qh, int gq, float scale_log2,
                               unsigned* flag, TcState& st, int flush_blk, uint64_t* fl_bar,
                               char* image) {
  constexpr int page = page_bytes_c(BK, BV);
  constexpr int NB = ring_blocks(page);
  const int lane = threadIdx.x & 31;
  // a block that leaves the window in this kernel has no page yet: it is
  // quantized from the ring after the streamed ones
  const bool flush = flush_blk >= lo && flush_blk == hi_all - 1;
  const int hi = flush ? hi_all - 1 : hi_all;
  // the early slots are this range's first units if they start at lo and
  // cover what its first `pre` units cover
  const bool reuse = pre > 0 && lo == lo_h && min(lo + pre * NB, hi) == pre_end;
  const int skip = reuse ? 0 : pre;
  const int n_units = (hi - lo + NB - 1) / NB;
  const int total = skip + n_units;
  int issued = pre;  // slots issued so far
  auto real_issue = [&](int s, bool fence) {
    const int u = s - skip;
    issue_slot<BK, BV>(pm, tw, ring, full, R, s, lo + u * NB, min(NB, hi - lo - u * NB), flag,
                       fence);
    issued = s + 1;
  };
  for (int s = pre; s < min(total, R); ++s) real_issue(s, false);

  const Lane ln = make_lane<BK, BV>(lane);
  uint32_t qb[16];
  load_qb<true, kWide>(qb, qh, gq, ln);
  int consumed = 0;
  for (int s = 0; s < total; ++s) {
    const int slot = s % R;
    // every lane waits; the warp leaves together if any lane gave up
    if (!__all_sync(0xffffffffu, mbar_wait(full + slot, (s / R) & 1))) {
      if (lane == 0) atomicOr(flag, KVQ_FLAG_WAIT_TIMEOUT);
      break;
    }
    consumed = s + 1;
    if (s >= skip) {
      const int u = s - skip;
      const char* base = ring + (size_t)slot * NB * page;
      if (lo + u * NB + NB <= hi) {
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
    if (s + R < total) real_issue(s + R, true);
  }
  // Copies issued but not consumed (a wait gave up, or the range shrank) land
  // before the ring is reused; bounded waits.
  if (lane == 0)
    for (int s = max(consumed, issued - R); s < issued; ++s) mbar_wait(full + s % R, (s / R) & 1);
  __syncwarp();
  if (flush) {
    // the page image is complete once its four quarters have arrived
    char* dst = const_cast<char*>(block_addr(pm, tw, flush_blk));
    if (__all_sync(0xffffffffu, mbar_wait(fl_bar, 0u))) {
      if (dst) {
        uint4* d4 = reinterpret_cast<uint4*>(dst);
        for (int i = lane; i < page / 16; i += 32) d4[i] = reinterpret_cast<const uint4*>(image)[i];
      } else if (lane == 0) {
        atomicOr(flag, (unsigned)KVQ_FLAG_BAD_PAGE);
      }
      const char* pg[1] = {image};
      tc_unit<BK, BV, 1, kWide>(pg, zero, qb, ln, scale_log2, st);
    } else if (lane == 0) {
      atomicOr(flag, KVQ_FLAG_WAIT_TIMEOUT);
    }
  }
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

// Window warp: chunks c0, c0 + stride, ... of the fp16 window.
template <int BK, int BV, bool kWide>
__device__ void tc_window_warp(const Dims& d, const __half* ring_k, const __half* ring_v,
                               const Plan& p, int L, int c0, int stride, char* area,
                               const __half* qh, int gq, float scale_log2, TcState& st,
                               int p_new, const __half* k_row, const __half* v_row,
                               uint64_t* bar, unsigned* flag) {
  const int lane = threadIdx.x & 31;
  const Lane ln = make_lane<BK, BV>(lane);
  uint32_t qb[16];
  load_qb<false, kWide>(qb, qh, gq, ln);
  __half* rows = reinterpret_cast<__half*>(area);
  uint32_t phase = 0u;
  for (int u = c0; u < p.n_res; u += stride) {
    const int p0 = p.Lq + u * kGroup;
    const int n_tok = min(kGroup, L - p0);
    uint32_t pt[1][2][2], pl[1][2][2];
    if (!stage_rows_bulk(rows, ring_k, p0, n_tok, d.ring, p_new, k_row, bar, phase++ & 1u)) {
      if ((threadIdx.x & 31) == 0) atomicOr(flag, KVQ_FLAG_WAIT_TIMEOUT);
      return;
    }
    tc_resid_scores<kWide, BV == 1>(rows, n_tok, qb, ln, scale_log2, st, pt, pl);
    __syncwarp();
    if (!stage_rows_bulk(rows, ring_v, p0, n_tok, d.ring, p_new, v_row, bar, phase++ & 1u)) {
      if ((threadIdx.x & 31) == 0) atomicOr(flag, KVQ_FLAG_WAIT_TIMEOUT);
      return;
    }
    tc_resid_values<kWide, BV == 1>(rows, pt, pl, st);
    __syncwarp();
  }
}


// ---------------------------------------------------------------------------
// The kernel
// ---------------------------------------------------------------------------

template <int BK, int BV, bool kWide>
__global__ void __launch_bounds__(kThreads, kCtasPerSm)
    decode_attn_kernel(Dims d, kvq_cache c, const __half* __restrict__ q, void* __restrict__ out,
                       int out_f16, float scale_log2, int S, unsigned smem_size, Ws ws,
                       const __half* __restrict__ k_new, const __half* __restrict__ v_new) {
  extern __shared__ __align__(128) unsigned char smem[];
  __shared__ MergeSmall ms;
  __shared__ int len_s[2];  // length attended, length before the append
  __shared__ __align__(16) __half q_s[kHeads * kHeadDim];  // the CTA's query heads
  __shared__ __align__(8) uint64_t wbar[kWarps];      // a window warp's staging barrier
  __shared__ __align__(8) uint64_t fl_bar;            // page image of a flush complete

  const int h = blockIdx.y, b = blockIdx.z;
  const int gq = d.gq;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int NV = gridDim.x * kWarps;     // warps per (sequence, kv-head)
  const int v = blockIdx.x * kWarps + warp;
  pdl_launch_dependents();
  const long long bh = (long long)b * d.hkv + h;
  const PageMap pm = page_map(d, c, b, h);
  TableWin tw;
  table_win_init(tw);
  const __half* ring_k = reinterpret_cast<const __half*>(c.k_resid) + bh * d.ring * kHeadDim;
  const __half* ring_v = reinterpret_cast<const __half*>(c.v_resid) + bh * d.ring * kHeadDim;
  const long long head0 = (long long)b * d.hq + (long long)h * gq;
  const __half* qh = q + head0 * kHeadDim;
  unsigned* flag = reinterpret_cast<unsigned*>(c.seq_len) + d.batch;
  // Decode step (k_new given): this kernel appends one token per sequence
  // before attending.  seq_len[b] is read once per CTA; the last CTA of the
  // sequence to have read it (ticket) publishes L0 + 1.
  const bool append = k_new != nullptr;
  unsigned seq_ticket = 0u;

  {
    constexpr int page = page_bytes_c(BK, BV);
    const int R = ring_slots(page);
    const int wbytes = warp_ring_bytes(page);
    char* ring = reinterpret_cast<char*>(smem) + (size_t)warp * wbytes;
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + (size_t)kWarps * wbytes) + warp * R;
    // 512 bytes at the end of shared memory: metadata rows of the
    // zero-point MMAs that carry no block, all zero except bytes 256..319,
    // which only the value zero-point MMA's row 4 reads: fp16 ones, so that
    // row sums the softmax weights (the row sum l).
    unsigned* zero = reinterpret_cast<unsigned*>(smem + smem_size - 16 - kZeroBytes);
    for (int i = threadIdx.x; i < kZeroBytes / 4; i += kThreads)
      zero[i] = i >= kOnesWord0 && i < kOnesWord0 + 16 ? 0x3C003C00u : 0u;
    int hint = 0;
    if (lane == 0) {
      for (int i = 0; i < R; ++i) mbar_init(full + i, 1);
      mbar_init(&wbar[warp], 1);
      if (warp == 0) mbar_init(&fl_bar, 4 * 32);
      fence_mbar_init();
      hint = read_len(c.seq_len + b);
    }
    hint = __shfl_sync(0xffffffffu, hint, 0);
    if (append && hint < d.max_len) ++hint;  // the length this kernel will attend
    __syncwarp();
    const Plan ph = make_plan(hint, d.residual, NV);
    int lo_h = 0, hi_h = 0, pre = 0, pre_end = 0;
    if (v < ph.np) {
      block_range(ph, v, lo_h, hi_h);
      // the newest block may be the one the previous kernel is writing
      pre = tc_pre_issue<BK, BV>(pm, tw, lo_h, hi_h, ph.nb - 1, ring, full, R, pre_end, flag);
      // a decode step that pushes a group out of the window: its owner brings
      // the group's ring rows (old, unchanging) into L2 for the flush
      if (append && lane == 0 && hi_h == ph.nb && ph.nb > 0 &&
          ph.Lq > packed_len(hint - 1, d.residual)) {
        prefetch_rows_l2(ring_k, ph.Lq - kGroup, kGroup, d.ring);
        prefetch_rows_l2(ring_v, ph.Lq - kGroup, kGroup, d.ring);
      }
    } else if (lane == 0) {
      // window rows of the length read before the wait into L2 (rows below
      // the newest token do not change; this is a hint, nothing waits on it)
      const int last = hint - (append ? 1 : 0) - 1;  // newest row not yet written
      for (int u = v - ph.np; u < ph.n_res; u += ph.n_resw) {
        const int p0 = ph.Lq + u * kGroup;
        const int n = min(kGroup, last - p0);
        if (n > 0) {
          prefetch_rows_l2(ring_k, p0, n, d.ring);
          prefetch_rows_l2(ring_v, p0, n, d.ring);
        }
      }
    }
    __syncthreads();  // zero rows written
    pdl_wait();
    // q (written by the previous kernel) into shared memory while the length
    // is read: one round trip for both
    if (threadIdx.x < gq * kHeadDim / 8)
      cp_async16(q_s + threadIdx.x * 8, qh + threadIdx.x * 8, 16u);
    asm volatile("cp.async.commit_group;" ::: "memory");
    if (threadIdx.x == 0) {
      const int L0 = read_len(c.seq_len + b);
      int L = L0;
      if (append) {
        if (L0 < d.max_len) L = L0 + 1;
        else atomicOr(flag, (unsigned)KVQ_FLAG_OVERFLOW);
      }
      len_s[0] = L;
      len_s[1] = L0;
    }
    asm volatile("cp.async.wait_group 0;" ::: "memory");
    __syncthreads();
    const int L = len_s[0], L0 = len_s[1];
    const bool grew = L > L0;  // this kernel appends the token at position L0
    if (append && threadIdx.x == 0)
      seq_ticket = atomicAdd(reinterpret_cast<unsigned*>(c.seq_len) + d.batch + 2 + b, 1u);
    const __half* k_row = grew ? k_new + bh * kHeadDim : nullptr;
    const __half* v_row = grew ? v_new + bh * kHeadDim : nullptr;
    if (grew && blockIdx.x == 0 && warp == 0) {  // the new token into its ring slot
      const long long slot = (long long)(L0 % d.ring) * kHeadDim;
      __half* rk = const_cast<__half*>(ring_k) + slot;
      __half* rv = const_cast<__half*>(ring_v) + slot;
      if (lane < 16) reinterpret_cast<uint4*>(rk)[lane] = reinterpret_cast<const uint4*>(k_row)[lane];
      else reinterpret_cast<uint4*>(rv)[lane - 16] = reinterpret_cast<const uint4*>(v_row)[lane - 16];
    }
    const bool same = L == hint;  // the plan made before the wait holds
    const Plan p = same ? ph : make_plan(L, d.residual, NV);
    const int flush_blk = grew && p.Lq > packed_len(L0, d.residual) ? p.nb - 1 : -1;
    const bool packed = v < p.np;
    // A flush is folded in by the packed warp np - 1 (it owns the last
    // block).  The window warps of its CTA quantize the block's four quarters
    // into the image while it streams; with no window warp in that CTA it
    // does them itself, before streaming.
    char* image = reinterpret_cast<char*>(smem + smem_size - 16 - kZeroBytes - image_bytes(page));
    const int cta_f = (p.np - 1) / kWarps;
    const int n_help = (cta_f + 1) * kWarps - p.np;  // window warps in CTA cta_f
    if (flush_blk >= 0 && (int)blockIdx.x == cta_f && (n_help > 0 ? !packed : v == p.np - 1)) {
      const int nw = n_help > 0 ? n_help : 1;
      for (int qi = n_help > 0 ? v - p.np : 0; qi < 4; qi += nw) {
        flush_quarter<BK, BV>(ring_k, ring_v, flush_blk * kGroup, d.ring, qi, image);
        mbar_arrive(&fl_bar);
      }
    }
    TcState st;
    init_state(st);
    if (packed || pre > 0) {
      // a warp that streamed early retires its slots even if it now has no blocks
      int lo = lo_h, hi = hi_h;
      if (!same) {
        lo = hi = 0;
        if (packed) block_range(p, v, lo, hi);
      }
      tc_packed_warp<BK, BV, kWide>(pm, tw, lo_h, pre, pre_end, lo, hi, ring, full, R,
                             reinterpret_cast<const char*>(zero), q_s, gq, scale_log2, flag, st,
                             flush_blk, &fl_bar, image);
    }
    if (!packed)
      tc_window_warp<BK, BV, kWide>(d, ring_k, ring_v, p, L, v - p.np, p.n_resw, ring, q_s, gq,
                             scale_log2, st, grew ? L0 : -1, k_row, v_row, &wbar[warp], flag);
    // the warp's ring is idle now: its state goes to the start of it
    WarpState& mine = *reinterpret_cast<WarpState*>(ring);
    if (packed) tc_write_state<true, BV, kWide>(st, mine, lane);
    else tc_write_state<false, BV, kWide>(st, mine, lane);
  }
  __syncthreads();

  // ---- merge the warps of this CTA: one partial per query head ----
  const size_t wstride = (size_t)warp_ring_bytes(page_bytes_c(BK, BV));
  auto wstate = [&](int w) -> const WarpState& {
    return *reinterpret_cast<const WarpState*>(smem + (size_t)w * wstride);
  };
  if (threadIdx.x < kWarps * gq) {
    const int w = threadIdx.x / gq, g = threadIdx.x % gq;
    float M = -INFINITY;
#pragma unroll
    for (int i = 0; i < kWarps; ++i) M = fmaxf(M, wstate(i).m[g]);
    const float m = wstate(w).m[g];
    ms.ww[w][g] = (m == -INFINITY) ? 0.0f : exp2f(m - M);
    if (w == 0) ms.cta_m[g] = M;
  }
  __syncthreads();
  const int n_items = gq * kHeadDim;
  for (int it = threadIdx.x; it < n_items; it += kThreads) {
    const int g = it / kHeadDim, ch = it % kHeadDim;
    float o = 0.0f, l = 0.0f;
#pragma unroll
    for (int i = 0; i < kWarps; ++i) {
      const float w = ms.ww[i][g];
      o = fmaf(w, wstate(i).o[g][ch], o);
      l = fmaf(w, wstate(i).l[g], l);
    }
    if (S == 1) {
      store_out(out, out_f16, (head0 + g) * kHeadDim + ch, l > 0.0f ? o / l : 0.0f);
    } else {
      const long long row = (head0 + g) * S + blockIdx.x;
      ws.o[row * kHeadDim + ch] = o;
      if (ch == 0) {
        ws.m[row] = ms.cta_m[g];
        ws.l[row] = l;
      }
    }
  }
  if (append && threadIdx.x == 0 &&
      seq_ticket == gridDim.y * gridDim.x - 1u) {  // every CTA of b has read L0
    const int L1 = len_s[0];
    __threadfence();
    c.seq_len[b] = L1;
    reinterpret_cast<unsigned*>(c.seq_len)[d.batch + 2 + b] = 0u;
  }
  if (S == 1) return;

  // ---- the last CTA of this (sequence, kv-head) merges the S partials ----
  __syncthreads();
  if (threadIdx.x == 0) ms.last = atom_add_acq_rel(&ws.tk[bh], 1u) == (unsigned)S - 1;
  __syncthreads();
  if (!ms.last) return;
  // The partial rows of this (sequence, kv-head) are one contiguous range: a
  // bulk copy brings them into shared memory (when they fit) while the maxima
  // and sums are loaded and turned into weights.
  const size_t o_bytes = (size_t)gq * S * kHeadDim * sizeof(float);
  float* wv = reinterpret_cast<float*>(smem);           // [gq][S] maxima, then weights
  float* lv = wv + gq * S;                               // [gq][S] sums
  float* lsum = lv + gq * S;                             // [gq]
  // the bulk copy's destination starts on a 128-byte boundary
  const size_t head_bytes = ((size_t)(2 * gq * S + 16) * sizeof(float) + 127) / 128 * 128;
  float* osm = reinterpret_cast<float*>(smem + head_bytes);  // [gq][S][128]
  const bool staged = head_bytes + o_bytes + 16 <= smem_size;
  uint64_t* mbar = reinterpret_cast<uint64_t*>(smem + smem_size - 16);
  if (staged && threadIdx.x == 0) {
    mbar_init(mbar, 1);
    fence_mbar_init();
    asm volatile("fence.proxy.async.global;" ::: "memory");
    mbar_expect_tx(mbar, (uint32_t)o_bytes);
    bulk_g2s(osm, ws.o + head0 * S * kHeadDim, (uint32_t)o_bytes, mbar);
  }
  for (int i = threadIdx.x; i < gq * S; i += kThreads) {
    wv[i] = __ldcg(ws.m + head0 * S + i);
    lv[i] = __ldcg(ws.l + head0 * S + i);
  }
  __syncthreads();
  for (int g = warp; g < gq; g += kWarps) {
    float M = -INFINITY;
    for (int k = lane; k < S; k += 32) M = fmaxf(M, wv[g * S + k]);
    M = warp_max(M);
    float Ls = 0.0f;
    for (int k = lane; k < S; k += 32) {
      const float m = wv[g * S + k];
      const float w = (m == -INFINITY) ? 0.0f : exp2f(m - M);
      Ls += w * lv[g * S + k];
      wv[g * S + k] = w;
    }
    Ls = warp_sum(Ls);
    if (lane == 0) lsum[g] = Ls;
  }
  bool ok = true;
  if (staged) ok = mbar_wait(mbar, 0);
  __syncthreads();
  for (int it = threadIdx.x; it < n_items; it += kThreads) {
    const int g = it / kHeadDim, ch = it % kHeadDim;
    float o = 0.0f;
    if (staged && ok) {
      const float* src = osm + (size_t)g * S * kHeadDim + ch;
#pragma unroll 8
      for (int k = 0; k < S; ++k) o = fmaf(wv[g * S + k], src[(size_t)k * kHeadDim], o);
    } else {
      const float* src = ws.o + (head0 + g) * S * kHeadDim + ch;
#pragma unroll 8
      for (int k = 0; k < S; ++k) o = fmaf(wv[g * S + k], __ldcg(src + (size_t)k * kHeadDim), o);
    }
    const float Ls = lsum[g];
    store_out(out, out_f16, (head0 + g) * kHeadDim + ch, Ls > 0.0f ? o / Ls : 0.0f);
  }
  if (threadIdx.x == 0) ws.tk[bh] = 0u;
}

size_t smem_bytes(const Dims& d) {
  const int page = (int)d.page_bytes;
  const size_t rings = (size_t)kWarps * warp_ring_bytes(page) +
                       (size_t)kWarps * ring_slots(page) * sizeof(uint64_t);
  // + a flushed block's page image, the zero rows of the packed warps and
  // the final merge's mbarrier
  return (rings + image_bytes(page) + kZeroBytes + 16 + 127) / 128 * 128;
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
    cfg.gridDim = dim3(S, d.hkv, d.batch);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem_bytes(d);
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, decode_attn_kernel<BK, BV, kWide>, d, c, q, out, out_f16, sl2, S,
                           (unsigned)smem_bytes(d), ws, k_new, v_new);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
  }
};


}  // namespace

// n_splits = CTAs per (sequence, kv-head); partial rows for exactly the
// n_splits CTAs of the launch (the same carve the kernel uses).  Tickets: one
// per (sequence, kv-head), sized one per query head.
size_t attn_split_workspace_bytes(const Dims& d, int n_splits) {
  const int S = n_splits;
  const size_t nml = (size_t)d.batch * d.hq * S;
  return align256(nml * 4) * 2 + align256(nml * kHeadDim * 4) +
         align256((size_t)d.batch * d.hq * 4);
}

// The tickets of a split-plan workspace (they must start at zero).
unsigned* attn_split_tickets(const Dims& d, int n_splits, void* workspace, size_t* bytes) {
  *bytes = (size_t)d.batch * d.hq * sizeof(unsigned);
  return carve(workspace, d.batch, d.hq, d.hkv, n_splits).tk;
}

cudaError_t launch_decode_attn_split(const Dims& d, const kvq_cache& c, const __half* q,
                                     void* out, int out_f16, float scale_log2, int n_splits,
                                     void* workspace, cudaStream_t st) {
  const Ws ws = carve(workspace, d.batch, d.hq, d.hkv, n_splits);
  return dispatch(d, LaunchOp{d, c, q, out, out_f16, scale_log2, n_splits, ws, st});
}

cudaError_t launch_decode_step_split(const Dims& d, const kvq_cache& c, const __half* k_new,
                                     const __half* v_new, const __half* q, void* out,
                                     int out_f16, float scale_log2, int n_splits,
                                     void* workspace, cudaStream_t st) {
  const Ws ws = carve(workspace, d.batch, d.hq, d.hkv, n_splits);
  LaunchOp op{d, c, q, out, out_f16, scale_log2, n_splits, ws, st};
  op.k_new = k_new;
  op.v_new = v_new;
  return dispatch(d, op);
}

}  // namespace kvq
