// DDAE fusion + top-K selection (Sec. 3.3, Eq. 7) and the gather of kept rows.
//
// pace_ddae_select: one CTA of 1024 threads per image.  Thread t owns scores t, t + 1024, ..
// (every warp access to the maps is one coalesced row of 32 scores); min/max, mean and the
// population variance are block reductions in a fixed order (bit-stable run to run); the K-th
// largest S_final is found by histogram rounds over the fp32 bit patterns (S_final >= 0, so
// integer order equals float order), and the kept set is compacted in ascending index order
// with warp ballots, the lower index winning among equal scores.
//
// pace_gather: one warp per kept row, 16-byte vector loads and stores.
#include <algorithm>
#include <atomic>
#include <cfloat>
#include <cmath>

#include "pace_common.cuh"
#include "pace_select.cuh"

namespace pace {
namespace {

constexpr int kSelThreads = 1024;
constexpr int kSelWarps = kSelThreads / 32;
static_assert(kSelWarps == 32, "block reductions take one warp partial per lane");
constexpr int kSelMaxB = 256;
constexpr int kSelBins = 4096;           // bins of one selection round (4 per thread)
constexpr int kSelRegMax = 12;           // scores per thread held in registers (12288 per map)
constexpr int kSelCompK = 16;            // score rows (of 1024) per compaction chunk
constexpr int kSelCand = kSelThreads;    // largest value bucket ranked directly (one score per thread)

struct SelectTable {
  int v0[kSelMaxB];  // first global row of image b
  int nv[kSelMaxB];  // visual tokens of image b
  int k0[kSelMaxB];  // first output slot of image b
  int nk[kSelMaxB];  // tokens kept for image b
};

struct SelShared {
  float red[8][kSelWarps];      // warp partials of the block reduction (min, max and two moments per map)
  unsigned bins[kSelBins];      // histogram of the current selection round
  unsigned wtot[kSelWarps];     // per-warp totals (bin prefix)
  unsigned sel[2];              // selected bin, entries in the bins above it
  unsigned cand[kSelCand];      // keys of the selected value bucket
  int cidx[kSelCand];           // and their indices in the map
  unsigned ncand;
  // compaction: per (score row k, warp) ballots of the keys above / equal to the threshold, the
  // exclusive prefix of their counts along the row (above in the low, equal in the high 16
  // bits), and the row totals
  unsigned mgt[kSelCompK][kSelWarps];
  unsigned meq[kSelCompK][kSelWarps];
  unsigned pre[kSelCompK][kSelWarps];
  unsigned rtot[kSelCompK];
};

__device__ __forceinline__ float warp_min(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fminf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ unsigned warp_incl_scan(unsigned v) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const unsigned n = __shfl_up_sync(0xffffffffu, v, o);
    if (lane >= o) v += n;
  }
  return v;
}

// Selection key of a fused score: its bit pattern (integer order = float order for values > 0);
// zero, negative and NaN scores take key 0, below every positive score.
__device__ __forceinline__ unsigned sel_key(float f) { return f > 0.f ? __float_as_uint(f) : 0u; }

// Bucket of a key for the first selection round: 64 buckets per octave of the score (the exponent
// and the top 6 mantissa bits), from 2^-63 (bucket 0 takes everything below, key 0 included) to
// the top bucket, which takes everything from about 1.98 up (S_final lies in [0, 1]).  Monotone in the
// key, so a bucket is one key range: sel_bucket_lo(b) .. sel_bucket_lo(b + 1) - 1.  Fused scores
// crowd near 0 when a map has a few large outliers; relative widths keep every bucket short
// there as well as near 1.
constexpr unsigned kSelKeyBase = 0x20000000u;   // 2^-63
constexpr int kSelKeyShift = 17;
__device__ __forceinline__ unsigned sel_bucket(unsigned key) {
  return key < kSelKeyBase ? 0u : min((key - kSelKeyBase) >> kSelKeyShift, static_cast<unsigned>(kSelBins - 1));
}
__device__ __forceinline__ unsigned sel_bucket_lo(unsigned b) {
  return b == 0u ? 0u : b >= static_cast<unsigned>(kSelBins) ? 0x7F800001u : kSelKeyBase + (b << kSelKeyShift);
}

// The bin holding the r-th largest entry of sh.bins, counting from bin 4095 down (1 <= r <= total):
// sh.sel[0] = that bin, sh.sel[1] = entries in the bins above it.  Every thread of the block calls
// it; thread t owns bins 4095 - 4t .. 4092 - 4t.  Ends with the result visible to all threads.
__device__ __forceinline__ void sel_bin_from_top(SelShared& sh, unsigned r) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int top = kSelBins - 1 - 4 * static_cast<int>(threadIdx.x);
  unsigned c[4], s4 = 0u;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    c[q] = sh.bins[top - q];
    s4 += c[q];
  }
  unsigned incl = warp_incl_scan(s4);
  if (lane == 31) sh.wtot[warp] = incl;
  __syncthreads();
  // entries in the warps before this one
  incl += __reduce_add_sync(0xffffffffu, lane < warp ? sh.wtot[lane] : 0u);
  const unsigned excl = incl - s4;
  if (excl < r && incl >= r) {   // exactly one thread
    unsigned above = excl;
    int q = 0;
#pragma unroll
    for (int qq = 0; qq < 3; ++qq)
      if (q == qq && above + c[qq] < r) {
        above += c[qq];
        q = qq + 1;
      }
    sh.sel[0] = static_cast<unsigned>(top - q);
    sh.sel[1] = above;
  }
  __syncthreads();
}

// Fusion + top-K of one map per CTA (1024 threads).  Thread t owns the scores i = k * 1024 + t,
// k = 0 .. R - 1 (R = ceil(nv / 1024)); with RM > 0 they stay in registers (R <= RM), with
// RM = 0 (maps above 12288 tokens) every pass reads the raw scores again and recomputes them
// with the same operations in the same order, so both give the same bits.
//   1. one block reduction of both raw maps: min, max, and the sums of x - c and (x - c)^2 with c
//      the map's first score (the shifted-data form of the variance); any non-finite raw score
//      records PACE_ERR_INVALID_ARG;
//   2. min-max normalisation is affine (a constant map becomes 0), so the normalised maps'
//      population variances follow from those sums;
//   3. the Eq. 7 weights (or a fixed ablation pair);
//   4. S_final = alpha_w norm(S_llm) + beta_w norm(S_vis) (written out);
//   5. the K-th largest S_final: 4096 buckets (64 per octave); if the selected bucket holds at
//      most 1024 scores, their keys are gathered and ranked directly, else rounds of 4096 bins
//      over the key bits inside the selected range run until one key T is left (exact either way);
//      for maps of up to 16384 scores with such a bucket, the pass that gathers the bucket also
//      records which scores lie above it, and each bucket score places itself by its own rank,
//      so 6. starts from those records;
//   6. kept = every score above T plus the lowest-index scores equal to T, written in index order:
//      score i sits at place (k, warp, lane) of that order, so the per (k, warp) ballot counts,
//      scanned along each row and summed over the rows before, give every kept score its slot.
// Reductions run in a fixed order, so results are the same from run to run.
template <int RM>
__global__ void __launch_bounds__(kSelThreads) ddae_select_kernel(const float* __restrict__ s_llm,
                                                                  const float* __restrict__ s_vis,
                                                                  const __grid_constant__ SelectTable tab,
                                                                  float tau, int fusion, float* __restrict__ s_final,
                                                                  float* __restrict__ weights,
                                                                  int32_t* __restrict__ kept, int b_base, int* status) {
  __shared__ SelShared sh;
  const int b = blockIdx.x;
  const int nv = tab.nv[b], v0 = tab.v0[b];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int R = (nv + kSelThreads - 1) / kSelThreads;   // the same for the whole block
  auto idx = [&](int k) { return k * kSelThreads + tid; };
  auto has = [&](int k) { return idx(k) < nv; };
  constexpr int RL = RM > 0 ? RM : 1;
  float ra[RL], rv[RL];
  const float* pa = s_llm + v0;
  const float* pv = s_vis + v0;

  // 1. min / max and shifted moments (and the finiteness check); the first round's bins are
  // cleared on the way
  const float ca = __ldg(pa), cv = __ldg(pv);
  for (int q = tid; q < kSelBins; q += kSelThreads) sh.bins[q] = 0u;
  if (tid == 0) sh.ncand = 0u;
  float amin = FLT_MAX, amax = -FLT_MAX, vmin = FLT_MAX, vmax = -FLT_MAX;
  float s1a = 0.f, s2a = 0.f, s1v = 0.f, s2v = 0.f;
  bool bad = false;
  auto take = [&](float a, float v) {
    bad |= !(fabsf(a) <= FLT_MAX) || !(fabsf(v) <= FLT_MAX);
    amin = fminf(amin, a); amax = fmaxf(amax, a);
    vmin = fminf(vmin, v); vmax = fmaxf(vmax, v);
    const float da = a - ca, dv = v - cv;
    s1a += da; s2a = fmaf(da, da, s2a);
    s1v += dv; s2v = fmaf(dv, dv, s2v);
  };
  if constexpr (RM > 0) {
#pragma unroll
    for (int k = 0; k < RM; ++k)
      if (has(k)) {
        ra[k] = __ldg(pa + idx(k));
        rv[k] = __ldg(pv + idx(k));
      }
#pragma unroll
    for (int k = 0; k < RM; ++k)
      if (has(k)) take(ra[k], rv[k]);
  } else {
    for (int k = 0; k < R; ++k)
      if (has(k)) take(__ldg(pa + idx(k)), __ldg(pv + idx(k)));
  }
  amin = warp_min(amin); amax = warp_max(amax);
  vmin = warp_min(vmin); vmax = warp_max(vmax);
  s1a = warp_sum(s1a); s2a = warp_sum(s2a);
  s1v = warp_sum(s1v); s2v = warp_sum(s2v);
  if (lane == 0) {
    sh.red[0][warp] = amin; sh.red[1][warp] = amax; sh.red[2][warp] = vmin; sh.red[3][warp] = vmax;
    sh.red[4][warp] = s1a; sh.red[5][warp] = s2a; sh.red[6][warp] = s1v; sh.red[7][warp] = s2v;
  }
  if (__syncthreads_or(bad) && tid == 0) record_error(status, PACE_ERR_INVALID_ARG, K_DDAE_SELECT);
  // lane l takes warp l's partials; the butterflies leave the block's values in every lane
  const float mna = warp_min(sh.red[0][lane]), mxa = warp_max(sh.red[1][lane]);
  const float mnv = warp_min(sh.red[2][lane]), mxv = warp_max(sh.red[3][lane]);
  const float t1a = warp_sum(sh.red[4][lane]), t2a = warp_sum(sh.red[5][lane]);
  const float t1v = warp_sum(sh.red[6][lane]), t2v = warp_sum(sh.red[7][lane]);
  const float ar = mxa - mna, vr = mxv - mnv;
  // (x - min) / range as a product with the range's reciprocal: within an ulp of the quotient,
  // and exact when the range is a power of two (a map spanning [0, 1] keeps its values)
  const float ia = ar > 0.f ? 1.0f / ar : 0.f, iv = vr > 0.f ? 1.0f / vr : 0.f;

  // 2-3. the normalised maps' population variances: (x - min) / range has the variance of x
  // divided by range^2, and var x = E[(x - c)^2] - (E[x - c])^2
  const float inv_n = 1.0f / static_cast<float>(nv);
  const float m1a = t1a * inv_n, m1v = t1v * inv_n;
  const float var_a = fmaxf(fmaf(-m1a, m1a, t2a * inv_n), 0.f) * ia * ia;
  const float var_v = fmaxf(fmaf(-m1v, m1v, t2v * inv_n), 0.f) * iv * iv;
  const float sig_a = sqrtf(var_a), sig_v = sqrtf(var_v);
  float wa, wv;
  if (fusion == PACE_DDAE_ONLY_LLM) {
    wa = 1.f;
    wv = 0.f;
  } else if (fusion == PACE_DDAE_ONLY_VIT) {
    wa = 0.f;
    wv = 1.f;
  } else if (fusion == PACE_DDAE_FIXED) {
    wa = wv = 0.5f;
  } else {   // Eq. 7
    // (every thread evaluates these; the fast intrinsics are within a few ulp)
    const float za = __fdividef(sig_a, tau), zv = __fdividef(sig_v, tau), zm = fmaxf(za, zv);
    const float ea = __expf(za - zm), ev = __expf(zv - zm);
    const float inv = __fdividef(1.0f, ea + ev);
    wa = ea * inv;
    wv = ev * inv;
  }
  if (tid == 0 && weights != nullptr) {
    weights[2 * (b_base + b)] = wa;
    weights[2 * (b_base + b) + 1] = wv;
  }

  // 4. S_final (in registers, ra reused, when RM > 0: written out by the first counting pass
  // below, or before an early return; otherwise written here)
  // alpha_w (a - min_a) / range_a + beta_w (v - min_v) / range_v with each map's weight and
  // reciprocal range folded into one coefficient
  const float cfa = wa * ia, cfv = wv * iv;
  auto fused = [&](float a, float v) { return fmaf(cfa, a - mna, cfv * (v - mnv)); };
  if constexpr (RM > 0) {
#pragma unroll
    for (int k = 0; k < RM; ++k)
      if (has(k)) ra[k] = fused(ra[k], rv[k]);
  } else if (s_final != nullptr) {
    for (int k = 0; k < R; ++k)
      if (has(k)) s_final[v0 + idx(k)] = fused(__ldg(pa + idx(k)), __ldg(pv + idx(k)));
  }
  auto store_final = [&](int k) {
    if constexpr (RM > 0)
      if (s_final != nullptr && has(k)) s_final[v0 + idx(k)] = ra[k];
  };
  // key of this thread's score k (0 where it has none: below every positive score)
  auto key_of = [&](int k) -> unsigned {
    if (!has(k)) return 0u;
    if constexpr (RM > 0) return sel_key(ra[k]);
    else return sel_key(fused(__ldg(pa + idx(k)), __ldg(pv + idx(k))));
  };
  // calls f(k) for k = kb .. ke - 1 (the same k for every thread at each call)
  auto for_rows = [&](int kb, int ke, auto&& f) {
    if constexpr (RM > 0) {
#pragma unroll
      for (int k = 0; k < RM; ++k)
        if (k >= kb && k < ke) f(k);
    } else {
      for (int k = kb; k < ke; ++k) f(k);
    }
  };

  const int K = tab.nk[b], k0 = tab.k0[b];
  if (K <= 0 || K >= nv) {
    for_rows(0, R, store_final);
    if (K > 0)
      for (int i = tid; i < nv; i += kSelThreads) kept[k0 + i] = v0 + i;
    return;
  }

  // Writes the kept indices of score rows kb .. ke - 1 from the ballots in sh.mgt / sh.meq (row
  // k - kb, warp w: the lanes whose score k * 1024 + 32 w + lane is above / equal to T): an
  // exclusive scan along each row (warp k - kb of the block), then thread (k - kb, w) adds the rows
  // before and places the set bits of its two ballots.  gbase / ebase count the keys above / equal
  // to T in the rows before kb; the counts after ke are returned.  Every row total fits 16 bits.
  auto compact_rows = [&](int kb, int ke, unsigned remaining, unsigned gbase, unsigned ebase) {
    const int nr = ke - kb;
    if (warp < nr) {
      const unsigned v = __popc(sh.mgt[warp][lane]) | (__popc(sh.meq[warp][lane]) << 16);
      const unsigned incl = warp_incl_scan(v);
      sh.pre[warp][lane] = incl - v;
      if (lane == 31) sh.rtot[warp] = incl;
    }
    __syncthreads();
    if (tid < nr * kSelWarps) {
      const int kr = tid >> 5, wp = tid & 31;
      unsigned pw = sh.pre[kr][wp];
      for (int q = 0; q < kr; ++q) pw += sh.rtot[q];
      const unsigned g0 = gbase + (pw & 0xFFFFu), e0 = ebase + (pw >> 16);
      const unsigned gm = sh.mgt[kr][wp], em = sh.meq[kr][wp];
      const int first = (kb + kr) * kSelThreads + wp * 32;
      for (unsigned m = gm | em; m != 0u; m &= m - 1u) {
        const int bit = __ffs(m) - 1;
        const unsigned lt = (1u << bit) - 1u;
        const unsigned gb = g0 + __popc(gm & lt), eb = e0 + __popc(em & lt);
        if ((gm >> bit) & 1u) __stcg(kept + k0 + gb + min(eb, remaining), v0 + first + bit);
        else if (eb < remaining) __stcg(kept + k0 + gb + eb, v0 + first + bit);
      }
    }
    unsigned tot = 0u;
    for (int q = 0; q < nr; ++q) tot += sh.rtot[q];
    return make_uint2(gbase + (tot & 0xFFFFu), ebase + (tot >> 16));
  };

  // 5. the K-th largest key.  Round 0 counts sel_bucket buckets; each later round splits the key
  // range [lo, lo + span) of the selected bin into 4096 bins of 2^shift keys until shift = 0.
  unsigned lo = 0u, span = 0u, r = static_cast<unsigned>(K);
  int shift = -1;   // round 0: sel_bucket
  // Histogram of this round.  A warp whose 32 scores share one bin (a flat stretch of the map, or
  // ties) adds once; otherwise each lane adds for itself and the rare same-bin lanes are
  // serialised by the shared-memory atomics.
  auto count_one = [&](int k) {
    if (shift < 0) store_final(k);
    unsigned bin = kSelBins;   // no bin
    if (has(k)) {
      const unsigned key = key_of(k);
      if (shift < 0) {
        bin = sel_bucket(key);
      } else {
        const unsigned off = key - lo;   // wraps for keys below lo
        if (off < span) bin = off >> shift;
      }
    }
    const unsigned b0 = __shfl_sync(0xffffffffu, bin, 0);
    if (__all_sync(0xffffffffu, bin == b0)) {
      if (lane == 0 && b0 < kSelBins) atomicAdd(&sh.bins[b0], 32u);
    } else if (bin < kSelBins) {
      atomicAdd(&sh.bins[bin], 1u);
    }
  };
  while (true) {
    if (shift >= 0) {   // round 0 counts into the bins cleared at the start
      for (int q = tid; q < kSelBins; q += kSelThreads) sh.bins[q] = 0u;
      __syncthreads();
    }
    for_rows(0, R, count_one);
    __syncthreads();
    sel_bin_from_top(sh, r);
    const unsigned bsel = sh.sel[0], above = sh.sel[1];
    r -= above;
    if (shift < 0) {
      lo = sel_bucket_lo(bsel);
      span = sel_bucket_lo(bsel + 1) - lo;   // the top bucket takes everything up to +inf
      const unsigned c = sh.bins[bsel];   // scores in the selected bucket (block-uniform)
      if (c <= static_cast<unsigned>(kSelCand) && R <= kSelCompK) {
        // kept masks per (row, warp): the scores above the bucket now, the bucket's own below
        for_rows(0, R, [&](int k) {
          const unsigned key = key_of(k);
          const unsigned off = key - lo;
          const bool in = has(k) && off < span;
          const unsigned um = __ballot_sync(0xffffffffu, has(k) && key >= lo && off >= span);
          if (lane == 0) {
            sh.mgt[k][warp] = um;
            sh.meq[k][warp] = 0u;
          }
          const unsigned m = __ballot_sync(0xffffffffu, in);
          if (m != 0u) {   // one slot claim per warp
            unsigned base = 0u;
            if (lane == 0) base = atomicAdd(&sh.ncand, static_cast<unsigned>(__popc(m)));
            base = __shfl_sync(0xffffffffu, base, 0) + __popc(m & ((1u << lane) - 1u));
            if (in) {
              sh.cand[base] = key;
              sh.cidx[base] = idx(k);
            }
          }
        });
        __syncthreads();
        // a bucket score x with fewer than r bucket scores >= x lies above T; with fewer than r
        // above it but at least r at or above it, x = T (and r - #above of them are kept)
        int ci;
        unsigned gt, ge;
        if (rank_in_list(sh.cand, c, ci, gt, ge)) {
          const int i = sh.cidx[ci];
          const unsigned bit = 1u << (i & 31);
          if (ge < r) {
            atomicOr(&sh.mgt[i >> 10][(i >> 5) & 31], bit);
          } else if (gt < r) {
            atomicOr(&sh.meq[i >> 10][(i >> 5) & 31], bit);
            sh.sel[1] = r - gt;   // the same value from every score equal to T
          }
        }
        __syncthreads();
        compact_rows(0, R, sh.sel[1], 0u, 0u);
        return;
      }
      if (c <= static_cast<unsigned>(kSelCand)) {
        // gather their keys (in any order) and rank them: the r-th largest is the key with fewer
        // than r keys above it and at least r at or above it
        for_rows(0, R, [&](int k) {
          const unsigned key = key_of(k);
          const bool in = has(k) && key - lo < span;
          const unsigned m = __ballot_sync(0xffffffffu, in);
          unsigned base = 0u;
          if (lane == 0 && m != 0u) base = atomicAdd(&sh.ncand, static_cast<unsigned>(__popc(m)));
          base = __shfl_sync(0xffffffffu, base, 0);
          if (in) sh.cand[base + __popc(m & ((1u << lane) - 1u))] = key;
        });
        __syncthreads();
        int ci;
        unsigned gt, ge;
        if (rank_in_list(sh.cand, c, ci, gt, ge)) {
          if (gt < r && ge >= r) {   // every thread holding the threshold key writes the same pair
            sh.sel[0] = sh.cand[ci];
            sh.sel[1] = r - gt;
          }
        }
        __syncthreads();
        lo = sh.sel[0];
        r = sh.sel[1];
        break;
      }
    } else {
      lo += bsel << shift;
      span = min(span - (bsel << shift), 1u << shift);
      if (shift == 0) break;
    }
    const int bits = 32 - __clz(span - 1u);   // keys lo .. lo + span - 1 need `bits` bits
    shift = bits > 12 ? bits - 12 : 0;
    __syncthreads();   // everyone has read sel before the next round rewrites it
  }
  const unsigned T = lo;        // key of the K-th largest S_final
  const unsigned remaining = r; // how many keys equal to T are kept (lowest indices first)

  // 6. compaction in index order, kSelCompK score rows at a time
  unsigned gbase = 0u, ebase = 0u;   // keys above / equal to T in the rows before
  for (int kb = 0; kb < R; kb += kSelCompK) {
    const int ke = min(R, kb + kSelCompK);
    __syncthreads();   // the previous readers of sh.sel / sh.mgt are done
    for_rows(kb, ke, [&](int k) {
      const unsigned key = key_of(k);
      const unsigned gm = __ballot_sync(0xffffffffu, key > T), em = __ballot_sync(0xffffffffu, key == T && has(k));
      if (lane == 0) {
        sh.mgt[k - kb][warp] = gm;
        sh.meq[k - kb][warp] = em;
      }
    });
    __syncthreads();
    const uint2 tot = compact_rows(kb, ke, remaining, gbase, ebase);
    gbase = tot.x;
    ebase = tot.y;
  }
}

// One warp per 2 KB piece of a row (128 16-byte vectors, 4 per lane, all in flight), so that a
// few thousand short rows still spread over every SM.
constexpr int kGatherU = 4;
constexpr int kGatherPiece = 32 * kGatherU;   // vectors per warp-piece

__global__ void __launch_bounds__(256) gather_rows_v16(const uint4* __restrict__ src, int64_t n_src,
                                                       int64_t row_vec, const int32_t* __restrict__ idx,
                                                       int64_t n_idx, uint4* __restrict__ dst, int* status) {
  const int lane = threadIdx.x & 31;
  const int64_t warp0 = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5;
  const int64_t pieces = (row_vec + kGatherPiece - 1) / kGatherPiece;
  for (int64_t w = warp0; w < n_idx * pieces; w += nwarps) {
    const int64_t r = w / pieces;
    const int64_t c0 = (w - r * pieces) * kGatherPiece;
    const int64_t s = idx[r];
    uint4* dp = dst + r * row_vec;
    if (s < 0 || s >= n_src) {
      for (int64_t c = c0 + lane; c < min(row_vec, c0 + kGatherPiece); c += 32) dp[c] = make_uint4(0u, 0u, 0u, 0u);
      if (lane == 0 && c0 == 0) record_error(status, PACE_ERR_INVALID_ARG, K_GATHER);
      continue;
    }
    const uint4* sp = src + s * row_vec;
    uint4 v[kGatherU];
#pragma unroll
    for (int u = 0; u < kGatherU; ++u) {
      const int64_t c = c0 + u * 32 + lane;
      if (c < row_vec) v[u] = __ldcs(sp + c);
    }
#pragma unroll
    for (int u = 0; u < kGatherU; ++u) {
      const int64_t c = c0 + u * 32 + lane;
      if (c < row_vec) __stcs(dp + c, v[u]);
    }
  }
}

// Rows of up to 32 U 16-byte vectors: one warp per row, grid-stride over the kept rows; every
// vector of a row is in flight at once (U per lane), and the warp reads its next row's index
// before it stores this one, so a row costs one memory round trip.
template <int U>
__global__ void __launch_bounds__(128) gather_rows_warp(const uint4* __restrict__ src, int64_t n_src, int row_vec,
                                                        const int32_t* __restrict__ idx, int64_t n_idx,
                                                        uint4* __restrict__ dst, int* status) {
  const int lane = threadIdx.x & 31;
  const int64_t nwarps = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5;
  int64_t r = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  int64_t s_next = r < n_idx ? __ldg(idx + r) : 0;
  for (; r < n_idx; r += nwarps) {
    const int64_t s = s_next;
    if (r + nwarps < n_idx) s_next = __ldg(idx + r + nwarps);
    uint4* dp = dst + r * row_vec;
    if (s < 0 || s >= n_src) {
      for (int c = lane; c < row_vec; c += 32) dp[c] = make_uint4(0u, 0u, 0u, 0u);
      if (lane == 0) record_error(status, PACE_ERR_INVALID_ARG, K_GATHER);
      continue;
    }
    const uint4* sp = src + s * row_vec;
    uint4 v[U];
#pragma unroll
    for (int u = 0; u < U; ++u)
      if (u * 32 + lane < row_vec) v[u] = __ldcs(sp + u * 32 + lane);
#pragma unroll
    for (int u = 0; u < U; ++u)
      if (u * 32 + lane < row_vec) __stcs(dp + u * 32 + lane, v[u]);
  }
}

// Byte-granular fallback for rows that are not 16-byte multiples or not 16-byte aligned.
__global__ void __launch_bounds__(256) gather_rows_bytes(const uint8_t* __restrict__ src, int64_t n_src,
                                                         int64_t row_bytes, const int32_t* __restrict__ idx,
                                                         int64_t n_idx, uint8_t* __restrict__ dst, int* status) {
  const int lane = threadIdx.x & 31;
  const int64_t warp0 = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5;
  for (int64_t r = warp0; r < n_idx; r += nwarps) {
    const int64_t s = idx[r];
    uint8_t* dp = dst + r * row_bytes;
    if (s < 0 || s >= n_src) {
      for (int64_t c = lane; c < row_bytes; c += 32) dp[c] = 0;
      if (lane == 0) record_error(status, PACE_ERR_INVALID_ARG, K_GATHER);
      continue;
    }
    const uint8_t* sp = src + s * row_bytes;
    for (int64_t c = lane; c < row_bytes; c += 32) dp[c] = sp[c];
  }
}

// Row list of the pruned LLM sequences (Sec. 3.3; App. C): sequence b (rows seq0 .. seq0 +
// n_pre - 1 of the packed pre-prune batch) keeps every position outside its visual span
// [vis, vis + n_vis) and the visual positions of its kept tokens, in sequence order.
constexpr int kPruneMaxB = 256;
struct PruneTable {
  int seq0[kPruneMaxB];   // first pre-prune row of sequence b
  int n_pre[kPruneMaxB];  // pre-prune length
  int vis[kPruneMaxB];    // start of the visual span within the sequence
  int v0[kPruneMaxB];     // first global visual index of image b (as in the kept list)
  int nv[kPruneMaxB];     // visual tokens of image b
  int k0[kPruneMaxB];     // first kept entry of image b
  int nk[kPruneMaxB];     // kept tokens of image b
  int post0[kPruneMaxB];  // first output row of sequence b
  int nb;
};

__global__ void __launch_bounds__(256) prune_index_kernel(const __grid_constant__ PruneTable t,
                                                          const int32_t* __restrict__ kept,
                                                          int32_t* __restrict__ out, int* status) {
  const int b = blockIdx.y;
  const int n_post = t.n_pre[b] - t.nv[b] + t.nk[b];
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n_post; i += gridDim.x * blockDim.x) {
    int row;
    if (i < t.vis[b]) {
      row = i;                                                    // before the visual span
    } else if (i < t.vis[b] + t.nk[b]) {
      const int k = kept[t.k0[b] + i - t.vis[b]] - t.v0[b];       // kept visual token (local)
      if (k < 0 || k >= t.nv[b]) {
        record_error(status, PACE_ERR_INVALID_ARG, K_PRUNE_INDEX);
        row = -1;
        out[t.post0[b] + i] = row;
        continue;
      }
      row = t.vis[b] + k;
    } else {
      row = i - t.nk[b] + t.nv[b];                                // after the visual span
    }
    out[t.post0[b] + i] = t.seq0[b] + row;
  }
}

// One launch over several tensors gathered with the same row list (hidden states, KV-cache
// rows, position ids ...): work item = (tensor, slab, output row), one warp each.
struct GatherMultiTable {
  pace_gather_tensor g[PACE_GATHER_MAX_TENSORS];
  int64_t item_prefix[PACE_GATHER_MAX_TENSORS + 1];   // slabs x rows per tensor
  int width[PACE_GATHER_MAX_TENSORS];                  // copy width in bytes: 16, 4 or 1
  int n;
};

template <typename V>
__device__ __forceinline__ void copy_row(const uint8_t* sp, uint8_t* dp, int64_t bytes, int lane) {
  const V* s = reinterpret_cast<const V*>(sp);
  V* d = reinterpret_cast<V*>(dp);
  const int64_t n = bytes / static_cast<int64_t>(sizeof(V));
  for (int64_t c = lane; c < n; c += 32) d[c] = s[c];
}
template <typename V>
__device__ __forceinline__ void zero_row(uint8_t* dp, int64_t bytes, int lane) {
  V* d = reinterpret_cast<V*>(dp);
  const int64_t n = bytes / static_cast<int64_t>(sizeof(V));
  for (int64_t c = lane; c < n; c += 32) d[c] = V{};
}

__global__ void __launch_bounds__(256) gather_multi_kernel(const __grid_constant__ GatherMultiTable t,
                                                           const int32_t* __restrict__ idx, int64_t n_idx,
                                                           int* status) {
  const int lane = threadIdx.x & 31;
  const int64_t warp0 = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5;
  const int64_t total = t.item_prefix[t.n];
  for (int64_t w = warp0; w < total; w += nwarps) {
    int k = 0;
    while (k + 1 < t.n && t.item_prefix[k + 1] <= w) ++k;
    const pace_gather_tensor& g = t.g[k];
    const int64_t local = w - t.item_prefix[k];
    const int64_t slab = local / n_idx, r = local - slab * n_idx;
    const int64_t s = idx[r];
    uint8_t* dp = static_cast<uint8_t*>(g.dst) + slab * g.dst_slab_stride + r * g.dst_row_stride;
    if (s < 0 || s >= g.n_src_rows) {
      if (t.width[k] == 16) zero_row<uint4>(dp, g.row_bytes, lane);
      else if (t.width[k] == 4) zero_row<uint32_t>(dp, g.row_bytes, lane);
      else zero_row<uint8_t>(dp, g.row_bytes, lane);
      if (lane == 0) record_error(status, PACE_ERR_INVALID_ARG, K_GATHER_MULTI);
      continue;
    }
    const uint8_t* sp = static_cast<const uint8_t*>(g.src) + slab * g.src_slab_stride + s * g.src_row_stride;
    if (t.width[k] == 16) copy_row<uint4>(sp, dp, g.row_bytes, lane);
    else if (t.width[k] == 4) copy_row<uint32_t>(sp, dp, g.row_bytes, lane);
    else copy_row<uint8_t>(sp, dp, g.row_bytes, lane);
  }
}

}  // namespace
}  // namespace pace

using namespace pace;

extern "C" pace_status_t pace_ddae_select(const float* s_llm_raw, const float* s_vis_raw, const int32_t* cu_v,
                                          const int32_t* cu_keep, int B, const pace_ddae_params* params,
                                          float* s_final, float* weights, int32_t* kept, pace_stream_t stream) {
  if (B < 0 || (B > 0 && (cu_v == nullptr || cu_keep == nullptr))) return PACE_ERR_INVALID_ARG;
  if (B == 0) return PACE_OK;
  if (s_llm_raw == nullptr || s_vis_raw == nullptr) return PACE_ERR_INVALID_ARG;
  if (cu_v[0] != 0 || cu_keep[0] != 0) return PACE_ERR_INVALID_ARG;
  int max_nv = 0;
  for (int b = 0; b < B; ++b) {
    const int nv = cu_v[b + 1] - cu_v[b], nk = cu_keep[b + 1] - cu_keep[b];
    if (nv < 1 || nk < 0 || nk > nv) return PACE_ERR_INVALID_ARG;
    if (nv > max_nv) max_nv = nv;
  }
  if (cu_keep[B] > 0 && kept == nullptr) return PACE_ERR_INVALID_ARG;
  const float tau = params ? params->tau : 0.5f;
  const int fusion = params ? params->fusion : PACE_DDAE_ADAPTIVE;
  if (!(tau > 0.f) || !std::isfinite(tau)) return PACE_ERR_INVALID_ARG;
  if (fusion < PACE_DDAE_ADAPTIVE || fusion > PACE_DDAE_FIXED) return PACE_ERR_INVALID_ARG;
  PACE_CHECK(check_device());
  int* status = device_status_word();
  for (int c0 = 0; c0 < B; c0 += kSelMaxB) {
    const int nb = (B - c0) < kSelMaxB ? (B - c0) : kSelMaxB;
    SelectTable t;
    int per_thread = 1;
    for (int i = 0; i < nb; ++i) {
      const int b = c0 + i;
      t.v0[i] = cu_v[b];
      t.nv[i] = cu_v[b + 1] - cu_v[b];
      t.k0[i] = cu_keep[b];
      t.nk[i] = cu_keep[b + 1] - cu_keep[b];
      per_thread = std::max(per_thread, (t.nv[i] + kSelThreads - 1) / kSelThreads);
    }
    // scores per thread in registers: 4 or 12, else (maps above 12288 tokens) read again per pass
    if (per_thread <= 4)
      ddae_select_kernel<4><<<nb, kSelThreads, 0, stream>>>(s_llm_raw, s_vis_raw, t, tau, fusion, s_final, weights,
                                                             kept, c0, status);
    else if (per_thread <= kSelRegMax)
      ddae_select_kernel<kSelRegMax><<<nb, kSelThreads, 0, stream>>>(s_llm_raw, s_vis_raw, t, tau, fusion, s_final,
                                                                      weights, kept, c0, status);
    else
      ddae_select_kernel<0><<<nb, kSelThreads, 0, stream>>>(s_llm_raw, s_vis_raw, t, tau, fusion, s_final, weights,
                                                             kept, c0, status);
    PACE_CHECK(check_launch());
  }
  return PACE_OK;
}

extern "C" pace_status_t pace_gather(const void* src, int64_t n_src_rows, int64_t row_bytes, const int32_t* idx,
                                     int64_t n_idx, void* dst, pace_stream_t stream) {
  if (n_idx < 0 || row_bytes <= 0 || n_src_rows < 0) return PACE_ERR_INVALID_ARG;
  if (n_idx == 0) return PACE_OK;
  if (src == nullptr || idx == nullptr || dst == nullptr) return PACE_ERR_INVALID_ARG;
  PACE_CHECK(check_device());
  int* status = device_status_word();
  int sms = 152;
  int dev = 0;
  if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int64_t warps_per_block = 8;
  int64_t blocks = (n_idx + warps_per_block - 1) / warps_per_block;
  const int64_t cap = static_cast<int64_t>(sms) * 16;
  if (blocks > cap) blocks = cap;
  const bool vec = (row_bytes % 16 == 0) && (reinterpret_cast<uintptr_t>(src) % 16 == 0) &&
                   (reinterpret_cast<uintptr_t>(dst) % 16 == 0);
  const int64_t row_vec = row_bytes / 16;
  if (vec && row_vec <= 32 * 16) {
    // a warp per row: enough resident warps for every SM (about 24 per SM at U = 16), no more
    // than there are rows
    // than there are rows; blocks of 4 warps, so that a few thousand rows still reach every SM
    const int64_t b = std::min<int64_t>((n_idx + 3) / 4, static_cast<int64_t>(sms) * 8);
    const unsigned g = static_cast<unsigned>(b);
    const int rv = static_cast<int>(row_vec);
    const uint4* s4 = static_cast<const uint4*>(src);
    uint4* d4 = static_cast<uint4*>(dst);
    if (row_vec <= 32 * 4) gather_rows_warp<4><<<g, 128, 0, stream>>>(s4, n_src_rows, rv, idx, n_idx, d4, status);
    else if (row_vec <= 32 * 8) gather_rows_warp<8><<<g, 128, 0, stream>>>(s4, n_src_rows, rv, idx, n_idx, d4, status);
    else gather_rows_warp<16><<<g, 128, 0, stream>>>(s4, n_src_rows, rv, idx, n_idx, d4, status);
  } else if (vec) {
    const int64_t pieces = (row_bytes / 16 + kGatherPiece - 1) / kGatherPiece;
    blocks = std::min<int64_t>((n_idx * pieces + warps_per_block - 1) / warps_per_block, static_cast<int64_t>(sms) * 8);
    gather_rows_v16<<<static_cast<unsigned>(blocks), 256, 0, stream>>>(
        static_cast<const uint4*>(src), n_src_rows, row_bytes / 16, idx, n_idx, static_cast<uint4*>(dst), status);
  } else {
    gather_rows_bytes<<<static_cast<unsigned>(blocks), 256, 0, stream>>>(
        static_cast<const uint8_t*>(src), n_src_rows, row_bytes, idx, n_idx, static_cast<uint8_t*>(dst), status);
  }
  return check_launch();
}

extern "C" pace_status_t pace_prune_index(int B, const int32_t* cu_seq, const int32_t* vis_start,
                                          const int32_t* cu_vis, const int32_t* cu_keep, const int32_t* kept,
                                          int32_t* out_idx, pace_stream_t stream) {
  if (B < 0) return PACE_ERR_INVALID_ARG;
  if (B == 0) return PACE_OK;
  if (cu_seq == nullptr || vis_start == nullptr || cu_vis == nullptr || cu_keep == nullptr) return PACE_ERR_INVALID_ARG;
  if (cu_seq[0] != 0 || cu_vis[0] != 0 || cu_keep[0] != 0) return PACE_ERR_INVALID_ARG;
  int64_t n_out = 0;
  for (int b = 0; b < B; ++b) {
    const int n_pre = cu_seq[b + 1] - cu_seq[b], nv = cu_vis[b + 1] - cu_vis[b], nk = cu_keep[b + 1] - cu_keep[b];
    if (n_pre < 0 || nv < 0 || nk < 0 || nk > nv || vis_start[b] < 0 || vis_start[b] + nv > n_pre)
      return PACE_ERR_INVALID_ARG;
    n_out += n_pre - nv + nk;
  }
  if (n_out == 0) return PACE_OK;
  if (out_idx == nullptr || (cu_keep[B] > 0 && kept == nullptr)) return PACE_ERR_INVALID_ARG;
  PACE_CHECK(check_device());
  int* status = device_status_word();
  int post = 0;
  for (int c0 = 0; c0 < B; c0 += kPruneMaxB) {
    const int nb = (B - c0) < kPruneMaxB ? (B - c0) : kPruneMaxB;
    PruneTable t{};
    t.nb = nb;
    int max_post = 1;
    for (int i = 0; i < nb; ++i) {
      const int b = c0 + i;
      t.seq0[i] = cu_seq[b];
      t.n_pre[i] = cu_seq[b + 1] - cu_seq[b];
      t.vis[i] = vis_start[b];
      t.v0[i] = cu_vis[b];
      t.nv[i] = cu_vis[b + 1] - cu_vis[b];
      t.k0[i] = cu_keep[b];
      t.nk[i] = cu_keep[b + 1] - cu_keep[b];
      t.post0[i] = post;
      const int np = t.n_pre[i] - t.nv[i] + t.nk[i];
      post += np;
      if (np > max_post) max_post = np;
    }
    const dim3 grid(static_cast<unsigned>(std::min((max_post + 255) / 256, 64)), static_cast<unsigned>(nb));
    prune_index_kernel<<<grid, 256, 0, stream>>>(t, kept, out_idx, status);
    PACE_CHECK(check_launch());
  }
  return PACE_OK;
}

extern "C" pace_status_t pace_gather_multi(const pace_gather_tensor* tensors, int n_tensors, const int32_t* idx,
                                           int64_t n_idx, pace_stream_t stream) {
  if (n_tensors < 0 || n_tensors > PACE_GATHER_MAX_TENSORS || n_idx < 0) return PACE_ERR_INVALID_ARG;
  if (n_tensors == 0 || n_idx == 0) return PACE_OK;
  if (tensors == nullptr || idx == nullptr) return PACE_ERR_INVALID_ARG;
  GatherMultiTable t{};
  t.n = n_tensors;
  t.item_prefix[0] = 0;
  for (int k = 0; k < n_tensors; ++k) {
    const pace_gather_tensor& g = tensors[k];
    if (g.src == nullptr || g.dst == nullptr || g.row_bytes <= 0 || g.n_slabs < 0 || g.n_src_rows < 0 ||
        g.src_row_stride < g.row_bytes || g.dst_row_stride < g.row_bytes)
      return PACE_ERR_INVALID_ARG;
    t.g[k] = g;
    const uintptr_t a = reinterpret_cast<uintptr_t>(g.src) | reinterpret_cast<uintptr_t>(g.dst) |
                        static_cast<uintptr_t>(g.row_bytes) | static_cast<uintptr_t>(g.src_row_stride) |
                        static_cast<uintptr_t>(g.dst_row_stride) | static_cast<uintptr_t>(g.src_slab_stride) |
                        static_cast<uintptr_t>(g.dst_slab_stride);
    t.width[k] = (a % 16 == 0) ? 16 : (a % 4 == 0) ? 4 : 1;
    t.item_prefix[k + 1] = t.item_prefix[k] + g.n_slabs * n_idx;
  }
  if (t.item_prefix[n_tensors] == 0) return PACE_OK;
  PACE_CHECK(check_device());
  int* status = device_status_word();
  int sms = 152, dev = 0;
  if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  int64_t blocks = (t.item_prefix[n_tensors] + 7) / 8;
  const int64_t cap = static_cast<int64_t>(sms) * 16;
  if (blocks > cap) blocks = cap;
  gather_multi_kernel<<<static_cast<unsigned>(blocks), 256, 0, stream>>>(t, idx, n_idx, status);
  return check_launch();
}
