// DDAE fusion + top-K selection (Sec. 3.3, Eq. 7) and the gather of kept rows.
//
// pace_ddae_select: one CTA of 1024 threads per image.  Both raw maps are staged in
// shared memory; min/max, mean and the population variance are block reductions in a
// fixed order (bit-stable run to run); the K-th largest S_final is found by an MSB-first
// 8-bit radix select on the fp32 bit patterns (S_final >= 0, so integer order equals
// float order), and the kept set is compacted in ascending index order with warp
// ballots, the lower index winning among equal scores.
//
// pace_gather: one warp per kept row, 16-byte vector loads and stores.
#include <algorithm>
#include <atomic>
#include <cfloat>
#include <cmath>

#include "pace_common.cuh"

namespace pace {
namespace {

constexpr int kSelThreads = 1024;
constexpr int kSelWarps = kSelThreads / 32;
constexpr int kSelMaxB = 256;
constexpr int kSelBins = 4096;           // bins of one selection round (4 per thread)
constexpr int kSelRegMax = 12;           // scores per thread held in registers (12288 per map)

struct SelectTable {
  int v0[kSelMaxB];  // first global row of image b
  int nv[kSelMaxB];  // visual tokens of image b
  int k0[kSelMaxB];  // first output slot of image b
  int nk[kSelMaxB];  // tokens kept for image b
};

struct SelShared {
  float red[3][4][kSelWarps];   // warp partials of the three block reductions
  unsigned bins[kSelBins];      // histogram of the current selection round
  unsigned wtot[kSelWarps];     // per-warp totals (bin prefix, compaction scans)
  unsigned wtot2[kSelWarps];
  unsigned sel[2];              // selected bin, entries in the bins above it
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

// Value bucket of a key for the first selection round: floor(4096 f), capped at the top bucket
// (monotone in the key; S_final lies in [0, 1]).
__device__ __forceinline__ unsigned sel_bucket(unsigned key) {
  return min(__float2uint_rz(__uint_as_float(key) * 4096.0f), static_cast<unsigned>(kSelBins - 1));
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
  unsigned before = 0u;   // entries in the warps before this one (fixed order)
  for (int w = 0; w < warp; ++w) before += sh.wtot[w];
  incl += before;
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

// Fusion + top-K of one map per CTA (1024 threads).  Thread t owns the contiguous scores
// [t R, t R + R) of its map (R = ceil(nv / 1024)); with RM > 0 they stay in registers (R <= RM),
// with RM = 0 (maps above 16384 tokens) every pass reads the raw scores again and recomputes
// them with the same operations in the same order, so both give the same bits.
//   1. min / max of both raw maps; any non-finite raw score records PACE_ERR_INVALID_ARG;
//   2. min-max normalisation (a constant map becomes 0) and the two means;
//   3. population variances, then the Eq. 7 weights (or a fixed ablation pair);
//   4. S_final = alpha_w S_llm + beta_w S_vis (written out);
//   5. the K-th largest S_final: 4096 value buckets, then rounds of 4096 bins over the key bits
//      inside the selected range until one key T is left (exact);
//   6. kept = every score above T plus the lowest-index scores equal to T, written in index order
//      from one block-wide scan of per-thread counts.
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
  const int R = (nv + kSelThreads - 1) / kSelThreads;
  const int i0 = tid * R;                                 // first score of this thread
  const int n_mine = max(0, min(R, nv - i0));             // scores this thread owns
  constexpr int RL = RM > 0 ? RM : 1;
  float ra[RL], rv[RL];
  const float* pa = s_llm + v0;
  const float* pv = s_vis + v0;

  // 1. min / max (and the finiteness check)
  float amin = FLT_MAX, amax = -FLT_MAX, vmin = FLT_MAX, vmax = -FLT_MAX;
  bool bad = false;
  if constexpr (RM > 0) {
#pragma unroll
    for (int k = 0; k < RM; ++k)
      if (k < n_mine) {
        ra[k] = __ldg(pa + i0 + k);
        rv[k] = __ldg(pv + i0 + k);
      }
#pragma unroll
    for (int k = 0; k < RM; ++k)
      if (k < n_mine) {
        bad |= !(fabsf(ra[k]) <= FLT_MAX) || !(fabsf(rv[k]) <= FLT_MAX);
        amin = fminf(amin, ra[k]); amax = fmaxf(amax, ra[k]);
        vmin = fminf(vmin, rv[k]); vmax = fmaxf(vmax, rv[k]);
      }
  } else {
    for (int k = 0; k < n_mine; ++k) {
      const float a = __ldg(pa + i0 + k), v = __ldg(pv + i0 + k);
      bad |= !(fabsf(a) <= FLT_MAX) || !(fabsf(v) <= FLT_MAX);
      amin = fminf(amin, a); amax = fmaxf(amax, a);
      vmin = fminf(vmin, v); vmax = fmaxf(vmax, v);
    }
  }
  amin = warp_min(amin); amax = warp_max(amax);
  vmin = warp_min(vmin); vmax = warp_max(vmax);
  if (lane == 0) {
    sh.red[0][0][warp] = amin; sh.red[0][1][warp] = amax;
    sh.red[0][2][warp] = vmin; sh.red[0][3][warp] = vmax;
  }
  if (__syncthreads_or(bad) && tid == 0) record_error(status, PACE_ERR_INVALID_ARG, K_DDAE_SELECT);
  float mna = FLT_MAX, mxa = -FLT_MAX, mnv = FLT_MAX, mxv = -FLT_MAX;
  for (int w = 0; w < kSelWarps; ++w) {
    mna = fminf(mna, sh.red[0][0][w]); mxa = fmaxf(mxa, sh.red[0][1][w]);
    mnv = fminf(mnv, sh.red[0][2][w]); mxv = fmaxf(mxv, sh.red[0][3][w]);
  }
  const float ar = mxa - mna, vr = mxv - mnv;
  // (x - min) / range as a product with the range's reciprocal: within an ulp of the quotient,
  // and exact when the range is a power of two (a map spanning [0, 1] keeps its values)
  const float ia = ar > 0.f ? 1.0f / ar : 0.f, iv = vr > 0.f ? 1.0f / vr : 0.f;
  auto norm_a = [&](float a) { return (a - mna) * ia; };
  auto norm_v = [&](float v) { return (v - mnv) * iv; };

  // 2. normalisation and the means
  float sa = 0.f, sv = 0.f;
  if constexpr (RM > 0) {
#pragma unroll
    for (int k = 0; k < RM; ++k)
      if (k < n_mine) {
        ra[k] = norm_a(ra[k]);
        rv[k] = norm_v(rv[k]);
        sa += ra[k];
        sv += rv[k];
      }
  } else {
    for (int k = 0; k < n_mine; ++k) {
      sa += norm_a(__ldg(pa + i0 + k));
      sv += norm_v(__ldg(pv + i0 + k));
    }
  }
  sa = warp_sum(sa);
  sv = warp_sum(sv);
  if (lane == 0) { sh.red[1][0][warp] = sa; sh.red[1][1][warp] = sv; }
  __syncthreads();
  float ta = 0.f, tv = 0.f;
  for (int w = 0; w < kSelWarps; ++w) { ta += sh.red[1][0][w]; tv += sh.red[1][1][w]; }
  const float ma = ta / nv, mv = tv / nv;

  // 3. population variances and the fusion weights
  float qa = 0.f, qv = 0.f;
  if constexpr (RM > 0) {
#pragma unroll
    for (int k = 0; k < RM; ++k)
      if (k < n_mine) {
        const float da = ra[k] - ma, dv = rv[k] - mv;
        qa = fmaf(da, da, qa);
        qv = fmaf(dv, dv, qv);
      }
  } else {
    for (int k = 0; k < n_mine; ++k) {
      const float da = norm_a(__ldg(pa + i0 + k)) - ma, dv = norm_v(__ldg(pv + i0 + k)) - mv;
      qa = fmaf(da, da, qa);
      qv = fmaf(dv, dv, qv);
    }
  }
  qa = warp_sum(qa);
  qv = warp_sum(qv);
  if (lane == 0) { sh.red[2][0][warp] = qa; sh.red[2][1][warp] = qv; }
  __syncthreads();
  float ua = 0.f, uv = 0.f;
  for (int w = 0; w < kSelWarps; ++w) { ua += sh.red[2][0][w]; uv += sh.red[2][1][w]; }
  const float sig_a = sqrtf(ua / nv), sig_v = sqrtf(uv / nv);
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
    const float za = sig_a / tau, zv = sig_v / tau, zm = fmaxf(za, zv);
    const float ea = expf(za - zm), ev = expf(zv - zm);
    wa = ea / (ea + ev);
    wv = ev / (ea + ev);
  }
  if (tid == 0 && weights != nullptr) {
    weights[2 * (b_base + b)] = wa;
    weights[2 * (b_base + b) + 1] = wv;
  }

  // 4. S_final, kept in registers as selection keys (ra reused)
  auto fused = [&](float a, float v) { return fmaf(wa, a, wv * v); };
  if constexpr (RM > 0) {
#pragma unroll
    for (int k = 0; k < RM; ++k)
      if (k < n_mine) {
        const float f = fused(ra[k], rv[k]);
        if (s_final != nullptr) s_final[v0 + i0 + k] = f;
        ra[k] = __uint_as_float(sel_key(f));
      }
  } else if (s_final != nullptr) {
    for (int k = 0; k < n_mine; ++k) s_final[v0 + i0 + k] = fused(norm_a(__ldg(pa + i0 + k)), norm_v(__ldg(pv + i0 + k)));
  }
  auto key_of = [&](int k) -> unsigned {
    if constexpr (RM > 0) return __float_as_uint(ra[k]);
    else return sel_key(fused(norm_a(__ldg(pa + i0 + k)), norm_v(__ldg(pv + i0 + k))));
  };
  // calls f(k, key) for every score of this thread, in index order
  auto for_each_key = [&](auto&& f) {
    if constexpr (RM > 0) {
#pragma unroll
      for (int k = 0; k < RM; ++k)
        if (k < n_mine) f(k, key_of(k));
    } else {
      for (int k = 0; k < n_mine; ++k) f(k, key_of(k));
    }
  };

  const int K = tab.nk[b], k0 = tab.k0[b];
  if (K <= 0) return;
  if (K >= nv) {
    for (int i = tid; i < nv; i += kSelThreads) kept[k0 + i] = v0 + i;
    return;
  }

  // 5. the K-th largest key.  Round 0 counts value buckets; each later round splits the key
  // range [lo, lo + span) of the selected bin into 4096 bins of 2^shift keys until shift = 0.
  unsigned lo = 0u, span = 0u, r = static_cast<unsigned>(K);
  int shift = -1;   // round 0: value buckets
  // Histogram of this round: lanes of a warp holding the same bin add once (fused scores crowd a
  // few low buckets, and equal keys one bin, which would otherwise serialise on one counter).
  // Every lane takes part in every step (a lane without a score brings the no-bin value).
  auto count_one = [&](int k) {
    unsigned bin = kSelBins;   // no bin
    if (k < n_mine) {
      const unsigned key = key_of(k);
      if (shift < 0) {
        bin = sel_bucket(key);
      } else {
        const unsigned off = key - lo;   // wraps for keys below lo
        if (off < span) bin = off >> shift;
      }
    }
    const unsigned peers = __match_any_sync(0xffffffffu, bin);
    if (bin < kSelBins && lane == __ffs(peers) - 1) atomicAdd(&sh.bins[bin], static_cast<unsigned>(__popc(peers)));
  };
  auto count_bins = [&]() {
    if constexpr (RM > 0) {
#pragma unroll
      for (int k = 0; k < RM; ++k) count_one(k);
    } else {
      for (int k = 0; k < R; ++k) count_one(k);   // R is the same for the whole block
    }
  };
  while (true) {
    for (int q = tid; q < kSelBins; q += kSelThreads) sh.bins[q] = 0u;
    __syncthreads();
    count_bins();
    __syncthreads();
    sel_bin_from_top(sh, r);
    const unsigned bsel = sh.sel[0], above = sh.sel[1];
    r -= above;
    if (shift < 0) {
      lo = __float_as_uint(static_cast<float>(bsel) * (1.0f / kSelBins));
      const unsigned hi = bsel == kSelBins - 1 ? 0x7F800001u   // the top bucket takes everything up to +inf
                                               : __float_as_uint(static_cast<float>(bsel + 1) * (1.0f / kSelBins));
      span = hi - lo;
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

  // 6. ascending compaction from per-thread counts
  unsigned gt = 0u, eq = 0u;
  for_each_key([&](int, unsigned key) {
    gt += key > T;
    eq += key == T;
  });
  const unsigned gi = warp_incl_scan(gt), ei = warp_incl_scan(eq);
  __syncthreads();   // the last round's readers of sh.sel / sh.wtot are done
  if (lane == 31) { sh.wtot[warp] = gi; sh.wtot2[warp] = ei; }
  __syncthreads();
  unsigned g_before = gi - gt, e_before = ei - eq;
  for (int w = 0; w < warp; ++w) { g_before += sh.wtot[w]; e_before += sh.wtot2[w]; }
  for_each_key([&](int k, unsigned key) {
    if (key > T) {
      kept[k0 + g_before + min(e_before, remaining)] = v0 + i0 + k;
      ++g_before;
    } else if (key == T) {
      if (e_before < remaining) kept[k0 + g_before + e_before] = v0 + i0 + k;
      ++e_before;
    }
  });
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
  if (vec) {
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
