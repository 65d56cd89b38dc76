// Condense: Adaptive Pixel Compressor (Sec. 3.2, Eq. 1-6) and the bicubic resize (App. B.3).
//
// Density, three kernels on the caller's stream:
//   apc_pass1  one CTA per strip of up to 32 patches of one patch row.  The strip's
//              14 image rows are staged in shared memory with coalesced 2- or 4-byte
//              loads; each warp reduces |x|^2 of its patches (exact integers) to the
//              inverse token norm 1/|T_i|; the strip's weighted column sums
//              sum_i x_ik / (255 |T_i|) (and sum_i 1/|T_i| for the constant coordinate)
//              are added to a per-image 589-vector as 2^-32 fixed-point integers, so the
//              reduction is exact and independent of the CTA order.
//   apc_pass2  same strips: c = sums / N, phi = |c|^2, c_hat = c / |c| (recomputed per
//              CTA from the 589 integers), then d_i = |t_i - c_hat| computed directly from
//              the staged pixels (no 2 - 2cos cancellation), counted into the tail's value
//              buckets (global atomics).
//   apc_tail_scan  one CTA per 4096 distances of an image: the k_tail-th largest's bucket from
//              the counts, the distances above it summed (2^-32 fixed point) and the bucket's
//              members listed; the image's last CTA ranks the members (directly, or by offset
//              rounds over their fp32 bits) and computes the tail mean, rho_d, rho, r and the
//              target size.  The token and pixel-statistic densities share it (their pass 2
//              counts the buckets the same way).
// Resize: apc_resample, four CTAs per SM walking the 16 x 32 output tiles of the batch; for
// downscales up to 2.75x per side the input window is staged in shared memory and filtered
// there with precomputed weights, steeper downscales take a generic path with per-tap weights.
#include <algorithm>
#include <atomic>
#include <cfloat>
#include <cmath>
#include <mutex>

#include "pace_common.cuh"
#include "pace_ptx.cuh"
#include "pace_select.cuh"

namespace pace {
namespace {

constexpr int kPatch = 14;
constexpr int kPatchBytes = kPatch * kPatch * 3;     // 588
constexpr int kTokDim = kPatchBytes + 1;             // 589: pixels + constant coordinate
constexpr int kStrip = 32;                           // patches per strip
constexpr int kStripRowBytes = kStrip * kPatch * 3;  // 1344 bytes of one image row per strip
constexpr int kApcThreads = 256;
constexpr int kPairIters = (kPatchBytes / 2 + 31) / 32;   // 10: coordinate pairs per lane
constexpr int kApcMaxB = 64;
// Column sums are 2^-32 fixed point in 64-bit integers.  The conversions below use only 32-bit
// conversions and fp32 (no fp64, which is a slow pipe on this GPU); fix32 rounds exactly like
// rounding v * 2^32 to the nearest integer (ties to even).
__device__ __forceinline__ unsigned long long fix32(float v) {   // 0 <= v < 2^31
  const float h = floorf(v);
  return (static_cast<unsigned long long>(static_cast<uint32_t>(h)) << 32) +
         __float2uint_rn((v - h) * 4294967296.0f);   // v - h is exact; the product is an exact scaling
}
__device__ __forceinline__ unsigned long long fix32_signed(float v) {   // |v| < 2^31, two's complement
  return v >= 0.f ? fix32(v) : 0ull - fix32(-v);
}
// sum * 2^-32 * inv_n for a non-negative (or, with SIGNED, two's-complement) fixed-point sum.
template <bool SIGNED>
__device__ __forceinline__ float unfix32(unsigned long long sum, float inv_n) {
  const bool neg = SIGNED && static_cast<long long>(sum) < 0;
  const unsigned long long m = neg ? 0ull - sum : sum;
  const float hi = static_cast<float>(static_cast<uint32_t>(m >> 32));   // < 2^24 for every use here
  const float v = fmaf(static_cast<float>(static_cast<uint32_t>(m)), 0x1p-32f, hi) * inv_n;
  return neg ? -v : v;
}

struct ApcTable {
  int64_t off[kApcMaxB];    // byte offset of image b
  int H[kApcMaxB];
  int W[kApcMaxB];
  int gw[kApcMaxB];         // patches per row
  int chunks[kApcMaxB];     // strips per patch row
  int patch0[kApcMaxB];     // first global patch (or token) of image b
  int n[kApcMaxB];          // patches (or tokens) of image b
  int ktail[kApcMaxB];
  int unit_prefix[kApcMaxB + 1];
  int nb;
  int b_base;               // global index of image 0 of this table
};

__device__ __forceinline__ int find_image(const ApcTable& t, int unit) {
  int b = 0;
  while (b + 1 < t.nb && t.unit_prefix[b + 1] <= unit) ++b;
  return b;
}

// Asynchronous 4-byte global -> shared copies (no register round trip, all in flight at once).
__device__ __forceinline__ void cp_async4(void* dst, const void* src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(static_cast<uint32_t>(__cvta_generic_to_shared(dst))),
               "l"(src)
               : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_all;" ::: "memory"); }
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait_group() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

// Stages the 14 rows x (np * 42) bytes of one strip into s (row pitch kStripRowBytes).  WIDE:
// asynchronous copies that the caller commits and waits for; otherwise plain loads and stores.
// Either way the caller synchronises the block before reading s.
template <bool WIDE>
__device__ __forceinline__ void load_strip(const uint8_t* __restrict__ img, int W, int py, int px0, int np,
                                           uint8_t* s) {
  const int seg = np * kPatch * 3;  // bytes per row (even; a multiple of 4 when WIDE)
  const int64_t pitch = static_cast<int64_t>(W) * 3;
  const uint8_t* base = img + static_cast<int64_t>(py) * kPatch * pitch + static_cast<int64_t>(px0) * kPatch * 3;
  // a warp per image row (rows warp, warp + 8), lanes along the row: no per-element division
  const int lane = threadIdx.x & 31;
  for (int y = threadIdx.x >> 5; y < kPatch; y += kApcThreads / 32) {
    const uint8_t* src = base + y * pitch;
    uint8_t* dst = s + y * kStripRowBytes;
    if (WIDE) {
      const int words = seg >> 2;
      for (int w = lane; w < words; w += 32)
        cp_async4(dst + 4 * w, reinterpret_cast<const uint32_t*>(src) + w);
    } else {
      const int halves = seg >> 1;
      for (int w = lane; w < halves; w += 32)
        *reinterpret_cast<uint16_t*>(dst + 2 * w) = __ldg(reinterpret_cast<const uint16_t*>(src) + w);
    }
  }
}

__device__ __forceinline__ float warp_sum_f(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// The two bytes of a 16-bit pair as floats: byte permutes build 2^23 + b in each word, one packed
// subtract removes the 2^23.
__device__ __forceinline__ float2 bytes2_to_float2(uint32_t v) {
  const float2 w = make_float2(__uint_as_float(__byte_perm(v, 0x4B000000u, 0x7540)),
                               __uint_as_float(__byte_perm(v, 0x4B000000u, 0x7541)));
  return ptx::fadd2(w, make_float2(-8388608.0f, -8388608.0f));
}

// Shared-memory offset of token coordinates 2j, 2j + 1 of patch 0 in a staged strip (row y of the
// patch, byte kk within its 42-byte row).
__device__ __forceinline__ int pair_offset(int j) {
  const int k = 2 * j, y = k / 42;
  return y * kStripRowBytes + (k - y * 42);
}

// Sum of squares of the 42 bytes at s (2-byte aligned): 4-byte words with dp4a, the unaligned
// ends as 16-bit loads.
__device__ __forceinline__ uint32_t row_sumsq42(const uint8_t* s) {
  uint32_t acc = 0u;
  const int lead = (reinterpret_cast<uintptr_t>(s) & 3u) ? 1 : 0;   // one 16-bit head to reach 4-byte alignment
  if (lead) {
    const uint32_t h = *reinterpret_cast<const uint16_t*>(s);
    acc = __dp4a(h, h, acc);
  }
  const uint32_t* w = reinterpret_cast<const uint32_t*>(s + 2 * lead);
#pragma unroll
  for (int i = 0; i < 10; ++i) acc = __dp4a(w[i], w[i], acc);
  if (!lead) {
    const uint32_t h = *reinterpret_cast<const uint16_t*>(s + 40);
    acc = __dp4a(h, h, acc);
  }
  return acc;
}

struct Strip {
  int b, u, py, px0, np;
};

__device__ __forceinline__ Strip strip_of(const ApcTable& t, int unit) {
  Strip q;
  q.b = find_image(t, unit);
  q.u = unit - t.unit_prefix[q.b];
  q.py = q.u / t.chunks[q.b];
  q.px0 = (q.u - q.py * t.chunks[q.b]) * kStrip;
  q.np = min(kStrip, t.gw[q.b] - q.px0);
  return q;
}

template <bool WIDE>
__device__ __forceinline__ void issue_strip(const uint8_t* __restrict__ img, const ApcTable& t, int unit, uint8_t* s) {
  const Strip q = strip_of(t, unit);
  load_strip<WIDE>(img + t.off[q.b], t.W[q.b], q.py, q.px0, q.np, s);
  cp_async_commit();
}

// Both passes run a grid of resident CTAs over the strips (unit = blockIdx.x, + gridDim.x, ...),
// loading the next strip asynchronously while the current one is worked on.
template <bool WIDE>
__global__ void __launch_bounds__(kApcThreads) apc_pass1(const uint8_t* __restrict__ img,
                                                         const __grid_constant__ ApcTable t, int units,
                                                         float* __restrict__ inv_norm,
                                                         unsigned long long* __restrict__ sums) {
  __shared__ __align__(16) uint8_t s2[2][kPatch * kStripRowBytes];
  __shared__ uint32_t ssq[8][kStrip];
  __shared__ __align__(16) float inv[kStrip];
  int unit = blockIdx.x;
  if (unit >= units) return;
  // weighted column sums: thread slot j (j = tid, tid + 256) owns columns 2j, 2j+1 (a pair never
  // crosses a 42-byte row); slot 294 owns the constant coordinate.  Each strip's sums are rounded
  // to 2^-32 fixed point and added exactly; one atomic per column when the image changes.
  constexpr int kSlots = kPatchBytes / 2 + 1;   // 295
  unsigned long long acc[2][2] = {{0ull, 0ull}, {0ull, 0ull}};
  int cur_b = -1;
  auto flush = [&]() {
    if (cur_b < 0) return;
    unsigned long long* sb = sums + static_cast<int64_t>(t.b_base + cur_b) * kTokDim;
#pragma unroll
    for (int q = 0; q < 2; ++q) {
      const int j = threadIdx.x + q * kApcThreads;
      if (j < kPatchBytes / 2) {
        atomicAdd(sb + 2 * j, acc[q][0]);
        atomicAdd(sb + 2 * j + 1, acc[q][1]);
      } else if (j == kPatchBytes / 2) {
        atomicAdd(sb + kPatchBytes, acc[q][0]);
      }
      acc[q][0] = acc[q][1] = 0ull;
    }
  };
  issue_strip<WIDE>(img, t, unit, s2[0]);
  for (int i = 0; unit < units; ++i, unit += gridDim.x) {
    const int next = unit + static_cast<int>(gridDim.x);
    if (next < units) {
      issue_strip<WIDE>(img, t, next, s2[(i + 1) & 1]);
      cp_async_wait_group<1>();
    } else {
      cp_async_wait_group<0>();
    }
    __syncthreads();
    const uint8_t* s = s2[i & 1];
    const Strip q = strip_of(t, unit);
    if (q.b != cur_b) {
      flush();
      cur_b = q.b;
    }
    // |x|^2 of every patch: thread (p = tid % 32, rows yg and yg + 8)
    {
      const int p = threadIdx.x & 31, yg = threadIdx.x >> 5;
      uint32_t a = 0u;
      if (p < q.np) {
        a = row_sumsq42(s + yg * kStripRowBytes + p * 42);
        if (yg + 8 < kPatch) a += row_sumsq42(s + (yg + 8) * kStripRowBytes + p * 42);
      }
      ssq[yg][p] = a;
    }
    __syncthreads();
    if (threadIdx.x < q.np) {
      const int p = threadIdx.x;
      uint32_t ss = 0u;
#pragma unroll
      for (int g = 0; g < 8; ++g) ss += ssq[g][p];
      const float n2 = static_cast<float>(ss) * (1.0f / 65025.0f) + 1.0f;
      const float iv = 1.0f / sqrtf(n2);
      inv[p] = iv;
      inv_norm[t.patch0[q.b] + q.py * t.gw[q.b] + q.px0 + p] = iv;
    }
    __syncthreads();
    float ivr[kStrip];   // full strips: the 32 inverse norms in registers, the patch loop unrolled
    if (q.np == kStrip) {
#pragma unroll
      for (int p = 0; p < kStrip; p += 4) {
        const float4 v4 = *reinterpret_cast<const float4*>(inv + p);
        ivr[p] = v4.x;
        ivr[p + 1] = v4.y;
        ivr[p + 2] = v4.z;
        ivr[p + 3] = v4.w;
      }
    }
#pragma unroll
    for (int qs = 0; qs < 2; ++qs) {
      const int j = threadIdx.x + qs * kApcThreads;
      if (j < kPatchBytes / 2) {
        const uint16_t* col = reinterpret_cast<const uint16_t*>(s + pair_offset(j));
        float2 a = make_float2(0.f, 0.f);
        if (q.np == kStrip) {
#pragma unroll
          for (int p = 0; p < kStrip; ++p)
            a = ptx::ffma2(make_float2(ivr[p], ivr[p]), bytes2_to_float2(col[p * 21]), a);
        } else {
          for (int p = 0; p < q.np; ++p) {
            const float iv = inv[p];
            a = ptx::ffma2(make_float2(iv, iv), bytes2_to_float2(col[p * 21]), a);
          }
        }
        acc[qs][0] += fix32(a.x * (1.0f / 255.0f));
        acc[qs][1] += fix32(a.y * (1.0f / 255.0f));
      } else if (j == kPatchBytes / 2) {
        float a = 0.f;
        for (int p = 0; p < q.np; ++p) a += inv[p];
        acc[qs][0] += fix32(a);
      }
    }
    __syncthreads();   // this buffer is refilled two strips on
  }
  flush();
  static_assert(kSlots <= 2 * kApcThreads, "column slots");
}

struct TailParams {
  float alpha, gamma, r_min, r_max;
  int align;
};

constexpr int kTailBins = 4096;            // level-1 buckets of the tail select
constexpr int kTailBins2 = 1024;           // level-2 offset bins over a listed bucket

// Bucket of a distance d >= 0: floor(2048 d), capped at the top bucket (monotone in d; NaN goes to
// bucket 0).  Full-rate arithmetic only (no float-to-integer conversion): once clamped to
// [0, 4095], 2048 d + 2^23 rounded toward zero holds floor(2048 d) in its low mantissa bits.
__device__ __forceinline__ int tail_bucket(float v) {
  const float x = fminf(fmaxf(v * 2048.0f, 0.0f), static_cast<float>(kTailBins - 1));
  return __float_as_int(__fadd_rz(x, 8388608.0f)) - 0x4B000000;
}

// Scratch of the density tail over several CTAs per image (apc_tail_scan): the counts of the
// distances per bucket (pass 2 adds them), then the sum and count of the distances above the
// k-th largest's bucket, the members of that bucket, and how many of the image's CTAs are done.
constexpr int kTailChunk = 4096;   // distances per CTA of apc_tail_scan
constexpr int kTailList = 4096;    // members of the selected bucket kept for the last CTA's rank
struct TailWork {
  unsigned long long above_fix;    // distances above the bucket, 2^-32 fixed point
  unsigned above_cnt;
  unsigned list_n;
  unsigned done;
  unsigned pad;
  unsigned hist[kTailBins];
  unsigned list[kTailList];
};

template <bool WIDE>
__global__ void __launch_bounds__(kApcThreads, 4) apc_pass2(const uint8_t* __restrict__ img,
                                                         const __grid_constant__ ApcTable t, int units,
                                                         const float* __restrict__ inv_norm,
                                                         const unsigned long long* __restrict__ sums,
                                                         float* __restrict__ d_out,
                                                         pace_apc_stats* __restrict__ stats,
                                                         TailWork* __restrict__ work) {
  __shared__ __align__(16) uint8_t s2[2][kPatch * kStripRowBytes];
  __shared__ __align__(8) float chat[kTokDim + 3];
  __shared__ float red[kApcThreads / 32];
  int unit = blockIdx.x;
  if (unit >= units) return;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  int off[kPairIters];   // this lane's coordinate pairs j = lane + 32 it
#pragma unroll
  for (int it = 0; it < kPairIters; ++it) off[it] = pair_offset(min(lane + 32 * it, kPatchBytes / 2 - 1));
  int cur_b = -1;
  bool reload = false;
  float2 chr[kPairIters];   // c_hat of this lane's coordinate pairs, in registers
  unsigned* hist = nullptr; // the current image's tail bucket counts
  issue_strip<WIDE>(img, t, unit, s2[0]);
  for (int i = 0; unit < units; ++i, unit += gridDim.x) {
    const int next = unit + static_cast<int>(gridDim.x);
    const Strip q = strip_of(t, unit);
    if (q.b != cur_b) {   // c = sums / N, |c|^2 (fixed summation order), c_hat = c / |c|
      cur_b = q.b;
      reload = true;
      hist = work[t.b_base + q.b].hist;
      const int N = (t.H[q.b] / kPatch) * t.gw[q.b];
      const float inv_n = 1.0f / static_cast<float>(N);
      const unsigned long long* sb = sums + static_cast<int64_t>(t.b_base + q.b) * kTokDim;
      float part = 0.f;
      for (int k = threadIdx.x; k < kTokDim; k += kApcThreads) {
        const float c = unfix32<false>(sb[k], inv_n);
        chat[k] = c;
        part = fmaf(c, c, part);
      }
      part = warp_sum_f(part);
      if (lane == 0) red[warp] = part;
      __syncthreads();
      float phi = 0.f;
#pragma unroll
      for (int w = 0; w < kApcThreads / 32; ++w) phi += red[w];
      const float inv_c = 1.0f / sqrtf(phi);
      __syncthreads();
      for (int k = threadIdx.x; k < kTokDim; k += kApcThreads) chat[k] *= inv_c;
      if (q.u == 0 && threadIdx.x == 0) {
        stats[t.b_base + q.b].phi = phi;
        stats[t.b_base + q.b].rho_g = 1.0f - phi;
        stats[t.b_base + q.b].n_patches = N;
        stats[t.b_base + q.b].k_tail = t.ktail[q.b];
      }
    }
    if (next < units) {
      issue_strip<WIDE>(img, t, next, s2[(i + 1) & 1]);
      cp_async_wait_group<1>();
    } else {
      cp_async_wait_group<0>();
    }
    __syncthreads();
    const uint8_t* s = s2[i & 1];
    // d_i = |t_i - c_hat| computed directly: warp per patch, lanes over column pairs
    const float* pinv = inv_norm + t.patch0[q.b] + q.py * t.gw[q.b] + q.px0;
    const float2* chat2 = reinterpret_cast<const float2*>(chat);
    if (reload) {
#pragma unroll
      for (int it = 0; it < kPairIters; ++it) chr[it] = chat2[min(lane + 32 * it, kPatchBytes / 2 - 1)];
      reload = false;
    }
    for (int p = warp; p < q.np; p += kApcThreads / 32) {
      const float sc = pinv[p] * (1.0f / 255.0f);
      const float2 sc2 = make_float2(sc, sc);
      float2 acc2 = make_float2(0.f, 0.f);
#pragma unroll
      for (int it = 0; it < kPairIters; ++it) {   // lanes over the 294 coordinate pairs
        const int j = lane + 32 * it;
        if (it < kPairIters - 1 || j < kPatchBytes / 2) {
          const uint32_t v = *reinterpret_cast<const uint16_t*>(s + off[it] + p * 42);
          const float2 e = ptx::ffma2(bytes2_to_float2(v), sc2, make_float2(-chr[it].x, -chr[it].y));
          acc2 = ptx::ffma2(e, e, acc2);
        }
      }
      const float iv = pinv[p];
      float acc = warp_sum_f(acc2.x + acc2.y);
      if (lane == 0) {
        const float v = iv - chat[kPatchBytes];
        const float dv = sqrtf(fmaf(v, v, acc));
        d_out[t.patch0[q.b] + q.py * t.gw[q.b] + q.px0 + p] = dv;
        atomicAdd(hist + tail_bucket(dv), 1u);   // the tail's bucket counts
      }
    }
    __syncthreads();   // this buffer is refilled two strips on; chat may be rewritten
  }
}

// ------------------------------------------------------------------------------------------------
// density on preview tokens (Sec. 3.2 "Shallow Feature Preview": T_v from the first ViT block)
// ------------------------------------------------------------------------------------------------
// Same Eq. 1-6 as the pixel path, on caller-supplied bf16 tokens [sum N, D].  A token of zero
// norm counts as t_hat = 0 (its cosine with any token is taken as 0); if every token of an
// image is zero, c_hat = 0.
constexpr int kTokChunk = 32;    // tokens per CTA
constexpr int kTokMaxD = 4096;   // longest token accepted (c_hat is staged in shared memory)

struct TokTable {
  int64_t tok0[kApcMaxB];        // first token of image b
  int n[kApcMaxB];               // tokens of image b
  int unit_prefix[kApcMaxB + 1]; // chunks of kTokChunk tokens (pass 2)
  int unit_prefix1[kApcMaxB + 1]; // chunks of rows1 tokens (pass 1)
  int ktail[kApcMaxB];
  int nb;
  int b_base;
  int D;
  int rows1;                     // tokens per pass-1 chunk (a chunk fits a 40 KB stage)
};

constexpr int kTok1StageBytes = 40960;   // one pass-1 stage: rows1 token rows
constexpr int kTok1MaxSlots = kTokMaxD / 2 / kApcThreads;   // column pairs per thread (8)

__device__ __forceinline__ int find_tok_image(const TokTable& t, int unit) {
  int b = 0;
  while (b + 1 < t.nb && t.unit_prefix[b + 1] <= unit) ++b;
  return b;
}

__device__ __forceinline__ float bf16_lo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t v) { return __uint_as_float(v & 0xffff0000u); }

// Pass 1: 1/|T_i| per token (warp per token) and the column sums of t_hat = T_i / |T_i|, as
// signed 2^-32 fixed point (exact, order-independent).  A grid of resident CTAs walks chunks of
// rows1 tokens; each chunk is staged in shared memory with cp.async while the previous one is
// worked on, so T is read once.  Per-chunk sums are rounded and added in registers; one atomic
// per column when the CTA moves to another image or ends.
__device__ __forceinline__ void tok_issue_chunk(const uint32_t* __restrict__ T, const TokTable& t, int unit,
                                                uint32_t* dst) {
  int b = 0;
  while (b + 1 < t.nb && t.unit_prefix1[b + 1] <= unit) ++b;
  const int r0 = (unit - t.unit_prefix1[b]) * t.rows1;
  const int nt = min(t.rows1, t.n[b] - r0);
  const int words = t.D >> 1;
  const uint32_t* src = T + (t.tok0[b] + r0) * words;
  for (int i = threadIdx.x; i < nt * words; i += kApcThreads) cp_async4(dst + i, src + i);
  cp_async_commit();
}

__global__ void __launch_bounds__(kApcThreads) apc_tok_pass1(const uint32_t* __restrict__ T,
                                                             const __grid_constant__ TokTable t, int units,
                                                             float* __restrict__ inv_norm,
                                                             unsigned long long* __restrict__ sums) {
  extern __shared__ __align__(16) uint32_t tok_smem[];   // two stages of rows1 x words
  __shared__ float inv[2][32];
  int unit = blockIdx.x;
  if (unit >= units) return;
  const int words = t.D >> 1;   // bf16 pairs per token
  const int stage = t.rows1 * words;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  unsigned long long acc[kTok1MaxSlots][2];
#pragma unroll
  for (int q = 0; q < kTok1MaxSlots; ++q) acc[q][0] = acc[q][1] = 0ull;
  int cur_b = -1;
  auto flush = [&]() {
    if (cur_b < 0) return;
    unsigned long long* sb = sums + static_cast<int64_t>(t.b_base + cur_b) * t.D;
#pragma unroll
    for (int q = 0; q < kTok1MaxSlots; ++q) {
      const int w = threadIdx.x + q * kApcThreads;
      if (w < words) {
        atomicAdd(sb + 2 * w, acc[q][0]);
        atomicAdd(sb + 2 * w + 1, acc[q][1]);
      }
      acc[q][0] = acc[q][1] = 0ull;
    }
  };
  tok_issue_chunk(T, t, unit, tok_smem);
  for (int i = 0; unit < units; ++i, unit += gridDim.x) {
    const int next = unit + static_cast<int>(gridDim.x);
    if (next < units) {
      tok_issue_chunk(T, t, next, tok_smem + ((i + 1) & 1) * stage);
      cp_async_wait_group<1>();
    } else {
      cp_async_wait_group<0>();
    }
    __syncthreads();
    int b = 0;
    while (b + 1 < t.nb && t.unit_prefix1[b + 1] <= unit) ++b;
    const int r0 = (unit - t.unit_prefix1[b]) * t.rows1;
    const int nt = min(t.rows1, t.n[b] - r0);
    if (b != cur_b) {
      flush();
      cur_b = b;
    }
    const uint32_t* rows = tok_smem + (i & 1) * stage;
    float* iv_s = inv[i & 1];
    for (int p = warp; p < nt; p += kApcThreads / 32) {
      const uint32_t* row = rows + p * words;
      float ss = 0.f;
      for (int w = lane; w < words; w += 32) {
        const uint32_t v = row[w];
        const float lo = bf16_lo(v), hi = bf16_hi(v);
        ss = fmaf(lo, lo, fmaf(hi, hi, ss));
      }
      ss = warp_sum_f(ss);
      if (lane == 0) {
        const float iv = ss > 0.f ? 1.0f / sqrtf(ss) : 0.f;
        iv_s[p] = iv;
        inv_norm[t.tok0[b] + r0 + p] = iv;
      }
    }
    __syncthreads();
#pragma unroll
    for (int q = 0; q < kTok1MaxSlots; ++q) {
      const int w = threadIdx.x + q * kApcThreads;
      if (w < words) {
        float2 a = make_float2(0.f, 0.f);
        for (int p = 0; p < nt; ++p) {
          const uint32_t v = rows[p * words + w];
          const float iv = iv_s[p];
          a = ptx::ffma2(make_float2(iv, iv), make_float2(bf16_lo(v), bf16_hi(v)), a);
        }
        acc[q][0] += fix32_signed(a.x);
        acc[q][1] += fix32_signed(a.y);
      }
    }
    __syncthreads();   // this stage is refilled two chunks on
  }
  flush();
}

// Pass 2: c = sums / N, phi = |c|^2, c_hat = c / |c|, then d_i = |t_hat_i - c_hat| directly
// (warp per token).
__global__ void __launch_bounds__(kApcThreads) apc_tok_pass2(const uint32_t* __restrict__ T,
                                                             const __grid_constant__ TokTable t,
                                                             const float* __restrict__ inv_norm,
                                                             const unsigned long long* __restrict__ sums,
                                                             float* __restrict__ d_out,
                                                             pace_apc_stats* __restrict__ stats,
                                                             TailWork* __restrict__ work) {
  __shared__ __align__(16) float chat[kTokMaxD];
  __shared__ float red[kApcThreads / 32];
  const int unit = blockIdx.x;
  const int b = find_tok_image(t, unit);
  const int c0 = (unit - t.unit_prefix[b]) * kTokChunk;
  const int nt = min(kTokChunk, t.n[b] - c0);
  const int N = t.n[b], D = t.D, words = D >> 1;
  const float inv_n = 1.0f / static_cast<float>(N);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const unsigned long long* sb = sums + static_cast<int64_t>(t.b_base + b) * D;
  float part = 0.f;
  for (int k = threadIdx.x; k < D; k += kApcThreads) {
    const float cv = unfix32<true>(sb[k], inv_n);
    chat[k] = cv;
    part = fmaf(cv, cv, part);
  }
  part = warp_sum_f(part);
  if (lane == 0) red[warp] = part;
  __syncthreads();
  float phi = 0.f;
#pragma unroll
  for (int w = 0; w < kApcThreads / 32; ++w) phi += red[w];
  const float inv_c = phi > 0.f ? 1.0f / sqrtf(phi) : 0.f;
  for (int k = threadIdx.x; k < D; k += kApcThreads) chat[k] *= inv_c;
  if (c0 == 0 && threadIdx.x == 0) {
    stats[t.b_base + b].phi = phi;
    stats[t.b_base + b].rho_g = 1.0f - phi;
    stats[t.b_base + b].n_patches = N;
    stats[t.b_base + b].k_tail = t.ktail[b];
  }
  __syncthreads();
  const uint32_t* base = T + (t.tok0[b] + c0) * words;
  const float2* chat2 = reinterpret_cast<const float2*>(chat);
  for (int p = warp; p < nt; p += kApcThreads / 32) {
    const uint32_t* row = base + static_cast<int64_t>(p) * words;
    const float iv = inv_norm[t.tok0[b] + c0 + p];
    float acc0 = 0.f, acc1 = 0.f;
    for (int w = lane; w < words; w += 32) {
      const uint32_t v = row[w];
      const float2 ch = chat2[w];
      const float e0 = fmaf(bf16_lo(v), iv, -ch.x), e1 = fmaf(bf16_hi(v), iv, -ch.y);
      acc0 = fmaf(e0, e0, acc0);
      acc1 = fmaf(e1, e1, acc1);
    }
    const float acc = warp_sum_f(acc0 + acc1);
    if (lane == 0) {
      const float dv = sqrtf(acc);
      d_out[t.tok0[b] + c0 + p] = dv;
      atomicAdd(&work[t.b_base + b].hist[tail_bucket(dv)], 1u);   // the tail's bucket counts
    }
  }
}

// Called by all 1024 threads: the bin holding the r-th largest entry, counting from bin NBINS - 1
// down (1 <= r <= total): sel[0] = that bin, sel[1] = entries in the bins above it.  wsum: 32 words.
template <int NBINS>
__device__ __forceinline__ void select_from_top(const unsigned* bins, unsigned r, unsigned* sel, unsigned* wsum) {
  constexpr int PER = NBINS / 1024;   // bins per thread
  static_assert(PER >= 1 && PER * 1024 == NBINS, "bins");
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int top = NBINS - 1 - PER * static_cast<int>(threadIdx.x);   // this thread: bins top .. top - PER + 1
  unsigned c4[PER], s4 = 0u;
#pragma unroll
  for (int q = 0; q < PER; ++q) {
    c4[q] = bins[top - q];
    s4 += c4[q];
  }
  unsigned incl = s4;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const unsigned n = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += n;
  }
  if (lane == 31) wsum[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    unsigned w = wsum[lane];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const unsigned n = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += n;
    }
    wsum[lane] = w;   // entries in warps 0 .. lane
  }
  __syncthreads();
  incl += warp > 0 ? wsum[warp - 1] : 0u;
  const unsigned excl = incl - s4;
  if (excl < r && incl >= r) {   // exactly one thread
    unsigned above = excl;
    int q = 0;
#pragma unroll
    for (int qq = 0; qq < PER - 1; ++qq)
      if (q == qq && above + c4[qq] < r) {
        above += c4[qq];
        q = qq + 1;
      }
    sel[0] = static_cast<unsigned>(top - q);
    sel[1] = above;
  }
  __syncthreads();
}

// Eq. 5-6 and R3-R4 from the tail mean d_top of image b: rho_d, rho, r and the target size.
__device__ __forceinline__ void tail_finish(const ApcTable& t, int b, const TailParams& prm,
                                            pace_apc_stats* __restrict__ stats, float rho_g, float d_top) {
  const float rho_d = fminf(d_top / prm.gamma, 1.0f);
  const float rho = prm.alpha * rho_g + (1.0f - prm.alpha) * rho_d;
  const float r = fminf(fmaxf(rho, prm.r_min), prm.r_max);
  const float sr = sqrtf(fmaxf(r, 0.0f));
  const int al = prm.align;
  const int H = t.H[b], W = t.W[b];
  int ho = al * static_cast<int>(floorf(static_cast<float>(H) * sr / al + 0.5f));
  int wo = al * static_cast<int>(floorf(static_cast<float>(W) * sr / al + 0.5f));
  ho = min(H, max(al, ho));
  wo = min(W, max(al, wo));
  pace_apc_stats& st = stats[t.b_base + b];
  st.d_top = d_top;
  st.rho_d = rho_d;
  st.rho = rho;
  st.r = r;
  st.h_out = ho;
  st.w_out = wo;
}

// The density tail (Eq. 5: the mean of the k_tail largest d_i, then Eq. 6 and R3-R4), several
// CTAs per image; pass 2 has counted the distances into 4096 value buckets of width 1/2048 (the
// top one also takes anything above).  CTA c of image b takes distances c kTailChunk .. : it
// selects the k-th largest's bucket from the counts (level 1), adds the distances above that
// bucket to the image's total in 2^-32 fixed point (exact, so the order of the CTAs does not
// matter) and lists the bucket's members.  The image's last CTA to finish narrows the members to
// the k-th largest distance T (level 2: each member ranked against the others when there are at
// most 1024, else rounds of 1024 bins over the key offsets from the bucket's first fp32 key) and
// writes the statistics; a bucket too crowded for the list is narrowed over the whole array by
// rounds of 4096 bins.
__global__ void __launch_bounds__(1024) apc_tail_scan(const __grid_constant__ ApcTable t, const float* __restrict__ d,
                                                      TailParams prm, pace_apc_stats* __restrict__ stats,
                                                      TailWork* __restrict__ work) {
  __shared__ unsigned bins[kTailBins];
  __shared__ unsigned hist2[kTailBins2];
  __shared__ unsigned sel[2];
  __shared__ unsigned cred[32];
  __shared__ unsigned long long fred[32];
  __shared__ int last;
  const int b = blockIdx.y;
  const int N = t.n[b];
  const int nchunk = (N + kTailChunk - 1) / kTailChunk;
  if (static_cast<int>(blockIdx.x) >= nchunk) return;
  TailWork* w = work + (t.b_base + b);
  const float* db = d + t.patch0[b];
  const unsigned k = static_cast<unsigned>(t.ktail[b]);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // level 1 on the counts (written by the previous kernel: read through L2)
  for (int i = threadIdx.x; i < kTailBins; i += blockDim.x) bins[i] = __ldcg(&w->hist[i]);
  __syncthreads();
  select_from_top<kTailBins>(bins, k, sel, cred);
  const int tb = static_cast<int>(sel[0]);
  const unsigned cb = bins[tb];         // entries in the k-th largest's bucket
  const unsigned above_n = sel[1];      // entries in the buckets above it
  const bool listed = cb <= kTailList;
  // this CTA's chunk
  unsigned long long s_fix = 0ull;
  unsigned cnt = 0u;
  bool wrote = false;   // this thread listed a member
  const int i0 = static_cast<int>(blockIdx.x) * kTailChunk, i1 = min(N, i0 + kTailChunk);
  for (int base = i0; base < i1; base += blockDim.x) {   // uniform trip count: the ballot below
    const int i = base + static_cast<int>(threadIdx.x);
    const float v = i < i1 ? db[i] : 0.f;
    const int bk = i < i1 ? tail_bucket(v) : -1;
    if (bk > tb) {
      s_fix += fix32(v);
      ++cnt;
    }
    const bool member = listed && bk == tb;
    const unsigned ball = __ballot_sync(0xffffffffu, member);
    if (ball != 0u) {   // one slot reservation per warp
      unsigned slot = 0u;
      if (lane == 0) slot = atomicAdd(&w->list_n, static_cast<unsigned>(__popc(ball)));
      slot = __shfl_sync(0xffffffffu, slot, 0);
      if (member) {
        w->list[slot + __popc(ball & ((1u << lane) - 1u))] = __float_as_uint(v);
        wrote = true;
      }
    }
  }
  for (int o = 16; o > 0; o >>= 1) {
    cnt += __shfl_xor_sync(0xffffffffu, cnt, o);
    s_fix += __shfl_xor_sync(0xffffffffu, s_fix, o);
  }
  if (lane == 0) {
    cred[warp] = cnt;
    fred[warp] = s_fix;
  }
  if (wrote) __threadfence();   // this thread's list entries, before the CTA reports its chunk done
  __syncthreads();
  if (threadIdx.x == 0) {
    unsigned c = 0u;
    unsigned long long f = 0ull;
    for (int i = 0; i < static_cast<int>(blockDim.x >> 5); ++i) {
      c += cred[i];
      f += fred[i];
    }
    atomicAdd(&w->above_fix, f);
    atomicAdd(&w->above_cnt, c);
    __threadfence();
    last = atomicAdd(&w->done, 1u) == static_cast<unsigned>(nchunk - 1);
  }
  __syncthreads();
  if (!last) return;
  __threadfence();
  // the image's totals and rho_g, read now so that their latency overlaps level 2
  unsigned tot_cnt = 0u;
  unsigned long long tot_fix = 0ull;
  float rho_g = 0.f;
  if (threadIdx.x == 0) {
    tot_cnt = __ldcg(&w->above_cnt);
    tot_fix = __ldcg(&w->above_fix);
    rho_g = stats[t.b_base + b].rho_g;
  }
  // level 2 (the image's last CTA): T = the k-th largest distance; the members of the bucket
  // above T are summed in fixed point (c counts every distance above T)
  unsigned remaining = k - above_n;
  unsigned lo = __float_as_uint(static_cast<float>(tb) * (1.0f / 2048.0f));
  unsigned span = (tb == kTailBins - 1 ? 0x7F800001u : __float_as_uint(static_cast<float>(tb + 1) * (1.0f / 2048.0f))) - lo;
  const unsigned bucket_lo = lo, bucket_span = span;
  s_fix = 0ull;
  cnt = 0u;
  unsigned prefix;
  __syncthreads();   // everyone has read sel and bins[tb]
  if (listed) {
    for (int i = threadIdx.x; i < static_cast<int>(cb); i += blockDim.x) bins[i] = __ldcg(&w->list[i]);
    __syncthreads();
    if (cb <= blockDim.x) {
      // one member per thread, ranked against the whole list: a member with fewer than
      // `remaining` members at or above it lies above the k-th largest (and is summed); with fewer
      // than `remaining` above it but at least that many at or above it, it is the k-th largest
      int mi;
      unsigned gt, ge;
      if (rank_in_list(bins, cb, mi, gt, ge)) {
        const unsigned mine = bins[mi];
        if (ge < remaining) {
          s_fix += fix32(__uint_as_float(mine));
          ++cnt;
        } else if (gt < remaining) {
          sel[0] = mine;   // the same key from every member equal to it
        }
      }
      __syncthreads();
      prefix = sel[0];
    } else {
      while (true) {
        const int bits = 32 - __clz(span - 1u);
        const int shift = bits > 10 ? bits - 10 : 0;
        for (int i = threadIdx.x; i < kTailBins2; i += blockDim.x) hist2[i] = 0u;
        __syncthreads();
        for (int i = threadIdx.x; i < static_cast<int>(cb); i += blockDim.x) {
          const unsigned off = bins[i] - lo;   // wraps for keys below lo
          if (off < span) atomicAdd(&hist2[off >> shift], 1u);
        }
        __syncthreads();
        select_from_top<kTailBins2>(hist2, remaining, sel, cred);
        lo += sel[0] << shift;
        remaining -= sel[1];
        if (shift == 0) break;
        span = min(span - (sel[0] << shift), 1u << shift);
      }
      prefix = lo;
      for (int i = threadIdx.x; i < static_cast<int>(cb); i += blockDim.x) {
        const unsigned key = bins[i];
        if (key > prefix) {
          s_fix += fix32(__uint_as_float(key));
          ++cnt;
        }
      }
    }
  } else {
    // a crowded bucket: its members by key offset from its first key over the whole array,
    // 4096 offsets (2^shift keys each) at a time, until one key is left
    while (true) {
      const int bits = 32 - __clz(span - 1u);
      const int shift = bits > 12 ? bits - 12 : 0;
      __syncthreads();                               // everyone has read sel and the bins
      for (int i = threadIdx.x; i < kTailBins; i += blockDim.x) bins[i] = 0u;
      __syncthreads();
      for (int base = 0; base < N; base += blockDim.x) {   // uniform trip count: __match_any_sync below
        const int i = base + static_cast<int>(threadIdx.x);
        const unsigned off = i < N ? __float_as_uint(db[i]) - lo : span;   // wraps for keys below lo
        const bool in = off < span;
        const unsigned digit = in ? off >> shift : kTailBins;
        const unsigned members = __ballot_sync(0xffffffffu, in);
        if (__popc(members) > 4) {
          const unsigned peers = __match_any_sync(0xffffffffu, digit);
          if (in && lane == __ffs(peers) - 1) atomicAdd(&bins[digit], static_cast<unsigned>(__popc(peers)));
        } else if (in) {
          atomicAdd(&bins[digit], 1u);
        }
      }
      __syncthreads();
      select_from_top<kTailBins>(bins, remaining, sel, cred);
      lo += sel[0] << shift;
      remaining -= sel[1];
      if (shift == 0) break;
      span = min(span - (sel[0] << shift), 1u << shift);
    }
    prefix = lo;
    for (int i = threadIdx.x; i < N; i += blockDim.x) {   // the bucket's members above T
      const unsigned key = __float_as_uint(db[i]);
      if (key > prefix && key - bucket_lo < bucket_span) {
        s_fix += fix32(__uint_as_float(key));
        ++cnt;
      }
    }
  }
  for (int o = 16; o > 0; o >>= 1) {
    cnt += __shfl_xor_sync(0xffffffffu, cnt, o);
    s_fix += __shfl_xor_sync(0xffffffffu, s_fix, o);
  }
  __syncthreads();   // the level-2 reads of cred and sel are done
  if (lane == 0) {
    cred[warp] = cnt;
    fred[warp] = s_fix;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    unsigned c = tot_cnt;
    unsigned long long f = tot_fix;
    for (int i = 0; i < static_cast<int>(blockDim.x >> 5); ++i) {
      c += cred[i];
      f += fred[i];
    }
    const float T = __uint_as_float(prefix);   // k-th largest d
    const float tot = unfix32<false>(f, 1.0f) + static_cast<float>(k - c) * T;   // the rest equal T
    tail_finish(t, b, prm, stats, rho_g, tot / static_cast<float>(k));
  }
}


// ------------------------------------------------------------------------------------------------
// pixel-statistic previews (App. "Shallow Feature Preview Ablation"): one small token per patch,
// then Eq. 1-6 on those tokens
// ------------------------------------------------------------------------------------------------
// Token of patch i: kPixDim floats, zero-padded.  Feature codes as pace_apc_feature.
constexpr int kPixDim = 8;
constexpr int kFeatRgb = 0, kFeatEntropy = 1, kFeatEdge = 2, kFeatLaplacian = 3;
constexpr int kLumaR = 299, kLumaG = 587, kLumaB = 114;   // Y' = 299 R + 587 G + 114 B (BT.601, thousandths)
constexpr int kLumaScale = 255000;                         // Y' of white
constexpr long long kEdgeThr2 = 63750LL * 63750LL;         // (0.25 * 255000)^2: Sobel magnitude test in integers

__device__ __forceinline__ int warp_sum_i(int v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ long long warp_sum_ll(long long v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// One warp computes the feature token of the patch at `px` (staged strip, row pitch
// kStripRowBytes): out[0 .. kPixDim).  `luma` (196 ints) and `hist` (48 ints) are the warp's
// scratch in shared memory.
__device__ __forceinline__ void patch_feature(const uint8_t* px, int feature, int* luma, int* hist, float* out) {
  const int lane = threadIdx.x & 31;
  float tok[kPixDim] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  if (feature == kFeatRgb) {
    uint32_t s[3] = {0u, 0u, 0u}, q[3] = {0u, 0u, 0u};
    for (int i = lane; i < kPatch * kPatch; i += 32) {
      const uint8_t* p = px + (i / kPatch) * kStripRowBytes + (i % kPatch) * 3;
#pragma unroll
      for (int c = 0; c < 3; ++c) {
        const uint32_t v = p[c];
        s[c] += v;
        q[c] += v * v;
      }
    }
#pragma unroll
    for (int c = 0; c < 3; ++c) {
      const uint32_t S = static_cast<uint32_t>(warp_sum_i(static_cast<int>(s[c])));
      const uint32_t Q = static_cast<uint32_t>(warp_sum_i(static_cast<int>(q[c])));
      constexpr float kInv = 1.0f / (196.0f * 255.0f);
      tok[c] = static_cast<float>(S) * kInv;
      tok[3 + c] = sqrtf(static_cast<float>(196u * Q - S * S)) * kInv;   // 196 Q - S^2 >= 0, < 2^32
    }
    tok[6] = 1.f;
  } else if (feature == kFeatEntropy) {
    for (int i = lane; i < 48; i += 32) hist[i] = 0;
    __syncwarp();
    for (int i = lane; i < kPatch * kPatch; i += 32) {
      const uint8_t* p = px + (i / kPatch) * kStripRowBytes + (i % kPatch) * 3;
#pragma unroll
      for (int c = 0; c < 3; ++c) atomicAdd(&hist[c * 16 + (p[c] >> 4)], 1);
    }
    __syncwarp();
#pragma unroll
    for (int c = 0; c < 3; ++c) {
      float h = 0.f;
      if (lane < 16) {
        const int n = hist[c * 16 + lane];
        if (n > 0) {
          const float pr = static_cast<float>(n) * (1.0f / 196.0f);
          h = -pr * log2f(pr);
        }
      }
      h = warp_sum_f(h);
      tok[c] = h * 0.25f;
    }
    tok[3] = 1.f;
    __syncwarp();   // hist is rewritten by the warp's next patch
  } else {
    for (int i = lane; i < kPatch * kPatch; i += 32) {
      const uint8_t* p = px + (i / kPatch) * kStripRowBytes + (i % kPatch) * 3;
      luma[i] = kLumaR * p[0] + kLumaG * p[1] + kLumaB * p[2];
    }
    __syncwarp();
    int cnt = 0, sl = 0;
    long long sl2 = 0;
    for (int i = lane; i < 144; i += 32) {   // the 12 x 12 interior
      const int y = 1 + i / 12, x = 1 + i % 12;
      const int* r0 = luma + (y - 1) * kPatch + x;
      const int* r1 = r0 + kPatch;
      const int* r2 = r1 + kPatch;
      if (feature == kFeatEdge) {
        const long long gx = (r0[1] + 2 * r1[1] + r2[1]) - (r0[-1] + 2 * r1[-1] + r2[-1]);
        const long long gy = (r2[-1] + 2 * r2[0] + r2[1]) - (r0[-1] + 2 * r0[0] + r0[1]);
        cnt += (gx * gx + gy * gy > kEdgeThr2) ? 1 : 0;
      } else {
        const int l = r1[-1] + r1[1] + r0[0] + r2[0] - 4 * r1[0];
        sl += l;
        sl2 += static_cast<long long>(l) * l;
      }
    }
    if (feature == kFeatEdge) {
      tok[0] = static_cast<float>(warp_sum_i(cnt)) * (1.0f / 144.0f);
    } else {
      const long long S = static_cast<long long>(warp_sum_i(sl)), Q = warp_sum_ll(sl2);
      const long long num = 144 * Q - S * S;   // 144^2 var in Y'^2 units, exact
      tok[0] = sqrtf(static_cast<float>(num)) * (1.0f / (144.0f * static_cast<float>(kLumaScale)));
    }
    tok[1] = 1.f;
    __syncwarp();   // luma is rewritten by the warp's next patch
  }
  if (lane < kPixDim) {
    float v = tok[0];
#pragma unroll
    for (int k = 1; k < kPixDim; ++k)
      if (lane == k) v = tok[k];
    out[lane] = v;
  }
}

// Feature tokens of every patch: a resident grid over the strips (as the density passes),
// a warp per patch.
template <bool WIDE>
__global__ void __launch_bounds__(kApcThreads) apc_pix_features(const uint8_t* __restrict__ img,
                                                                const __grid_constant__ ApcTable t, int units,
                                                                int feature, float* __restrict__ tokens) {
  __shared__ __align__(16) uint8_t s2[2][kPatch * kStripRowBytes];
  __shared__ int luma[kApcThreads / 32][kPatch * kPatch];
  __shared__ int hist[kApcThreads / 32][48];
  int unit = blockIdx.x;
  if (unit >= units) return;
  const int warp = threadIdx.x >> 5;
  issue_strip<WIDE>(img, t, unit, s2[0]);
  for (int i = 0; unit < units; ++i, unit += gridDim.x) {
    const int next = unit + static_cast<int>(gridDim.x);
    if (next < units) {
      issue_strip<WIDE>(img, t, next, s2[(i + 1) & 1]);
      cp_async_wait_group<1>();
    } else {
      cp_async_wait_group<0>();
    }
    __syncthreads();
    const Strip q = strip_of(t, unit);
    const uint8_t* s = s2[i & 1];
    for (int p = warp; p < q.np; p += kApcThreads / 32)
      patch_feature(s + p * 42, feature, luma[warp], hist[warp],
                    tokens + (static_cast<int64_t>(t.patch0[q.b]) + q.py * t.gw[q.b] + q.px0 + p) * kPixDim);
    __syncthreads();   // this buffer is refilled two strips on
  }
}

// Density of kPixDim-float tokens, pass 1: t_hat in place and the chunk's column sums (2^-32
// fixed point, deterministic).  A CTA takes kApcThreads tokens of one image, a thread per token.
struct PixTable {
  int tok0[kApcMaxB];
  int n[kApcMaxB];
  int ktail[kApcMaxB];
  int unit_prefix[kApcMaxB + 1];
  int nb;
  int b_base;
};

__device__ __forceinline__ int find_pix_image(const PixTable& t, int unit) {
  int b = 0;
  while (b + 1 < t.nb && t.unit_prefix[b + 1] <= unit) ++b;
  return b;
}

__global__ void __launch_bounds__(kApcThreads) apc_pix_pass1(const __grid_constant__ PixTable t,
                                                             float* __restrict__ tokens,
                                                             unsigned long long* __restrict__ sums) {
  __shared__ float part[kApcThreads / 32][kPixDim];
  const int b = find_pix_image(t, blockIdx.x);
  const int i = (blockIdx.x - t.unit_prefix[b]) * kApcThreads + threadIdx.x;
  const bool live = i < t.n[b];
  float v[kPixDim] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  float4* row = reinterpret_cast<float4*>(tokens + (static_cast<int64_t>(t.tok0[b]) + (live ? i : 0)) * kPixDim);
  if (live) {
    const float4 a = row[0], c = row[1];
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = c.x; v[5] = c.y; v[6] = c.z; v[7] = c.w;
    float n2 = 0.f;
#pragma unroll
    for (int k = 0; k < kPixDim; ++k) n2 = fmaf(v[k], v[k], n2);
    const float iv = n2 > 0.f ? 1.0f / sqrtf(n2) : 0.f;
#pragma unroll
    for (int k = 0; k < kPixDim; ++k) v[k] *= iv;
    row[0] = make_float4(v[0], v[1], v[2], v[3]);
    row[1] = make_float4(v[4], v[5], v[6], v[7]);
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
#pragma unroll
  for (int k = 0; k < kPixDim; ++k) {
    const float w = warp_sum_f(v[k]);
    if (lane == 0) part[warp][k] = w;
  }
  __syncthreads();
  if (threadIdx.x < kPixDim) {
    float a = 0.f;
#pragma unroll
    for (int w = 0; w < kApcThreads / 32; ++w) a += part[w][threadIdx.x];
    atomicAdd(sums + static_cast<int64_t>(t.b_base + b) * kPixDim + threadIdx.x, fix32_signed(a));
  }
}

// Pass 2: c = sums / N, phi = |c|^2, c_hat = c / |c|, d_i = |t_hat_i - c_hat| (thread per token).
__global__ void __launch_bounds__(kApcThreads) apc_pix_pass2(const __grid_constant__ PixTable t,
                                                             const float* __restrict__ tokens,
                                                             const unsigned long long* __restrict__ sums,
                                                             float* __restrict__ d_out,
                                                             pace_apc_stats* __restrict__ stats,
                                                             TailWork* __restrict__ work) {
  const int b = find_pix_image(t, blockIdx.x);
  const int u = blockIdx.x - t.unit_prefix[b];
  const int i = u * kApcThreads + threadIdx.x;
  const int N = t.n[b];
  const float inv_n = 1.0f / static_cast<float>(N);
  float c[kPixDim];
  float phi = 0.f;
#pragma unroll
  for (int k = 0; k < kPixDim; ++k) {
    c[k] = unfix32<true>(sums[static_cast<int64_t>(t.b_base + b) * kPixDim + k], inv_n);
    phi = fmaf(c[k], c[k], phi);
  }
  const float inv_c = phi > 0.f ? 1.0f / sqrtf(phi) : 0.f;
  if (u == 0 && threadIdx.x == 0) {
    stats[t.b_base + b].phi = phi;
    stats[t.b_base + b].rho_g = 1.0f - phi;
    stats[t.b_base + b].n_patches = N;
    stats[t.b_base + b].k_tail = t.ktail[b];
  }
  if (i >= N) return;
  const float4* row = reinterpret_cast<const float4*>(tokens + (static_cast<int64_t>(t.tok0[b]) + i) * kPixDim);
  const float4 a = row[0], e = row[1];
  const float v[kPixDim] = {a.x, a.y, a.z, a.w, e.x, e.y, e.z, e.w};
  float acc = 0.f;
#pragma unroll
  for (int k = 0; k < kPixDim; ++k) {
    const float x = v[k] - c[k] * inv_c;
    acc = fmaf(x, x, acc);
  }
  const float dv = sqrtf(acc);
  d_out[t.tok0[b] + i] = dv;
  atomicAdd(&work[t.b_base + b].hist[tail_bucket(dv)], 1u);   // the tail's bucket counts
}

// ------------------------------------------------------------------------------------------------
// resample
// ------------------------------------------------------------------------------------------------
constexpr int kRsThreads = 256;  // threads of a resample CTA
constexpr int kRsTH = 8;         // output rows of a generic tile (kRsTH x kRsTW = kRsThreads)
constexpr int kRsTW = 32;        // output columns of a generic tile
constexpr int kRsChunk = 8;      // input rows filtered per step of the generic path

struct ResampleTable {
  int64_t src_off[kApcMaxB];
  int64_t dst_off[kApcMaxB];
  int H[kApcMaxB];
  int W[kApcMaxB];
  int Ho[kApcMaxB];  // used when stats == nullptr
  int Wo[kApcMaxB];
  int nb;
  int b_base;
};

__device__ __forceinline__ float cubic_w(float t) {
  // Keys' cubic convolution, a = -0.5
  t = fabsf(t);
  if (t < 1.0f) return (1.5f * t - 2.5f) * t * t + 1.0f;
  if (t < 2.0f) return ((-0.5f * t + 2.5f) * t - 4.0f) * t + 2.0f;
  return 0.0f;
}

__device__ __forceinline__ int64_t floor_div(int64_t x, int64_t d) { return x >= 0 ? x / d : -((-x + d - 1) / d); }
__device__ __forceinline__ int64_t ceil_div(int64_t x, int64_t d) { return x >= 0 ? (x + d - 1) / d : -((-x) / d); }

// Window of output index o (reading R5) in exact integer arithmetic.  With s = n_in / n_out
// and fs = max(s, 1), the centre is c = (2o + 1) n_in / (2 n_out), the taps are
// lo .. lo + n - 1 with lo = max(0, floor(c - 2 fs)) and lo + n = min(n_in, ceil(c + 2 fs)),
// and tap i sits at (lo + i + 0.5 - c) / fs = (num0 + i * step) * inv_den with integer
// num0 = (2 lo + 1) n_out - (2o + 1) n_in, step = 2 n_out and den = 2 n_out fs.
struct Win {
  int lo, n, num0, step;
  float inv_den;
};
__device__ __forceinline__ Win exact_window(int o, int n_in, int n_out) {
  const bool down = n_in > n_out;
  const int64_t cn = (2 * static_cast<int64_t>(o) + 1) * n_in;                   // c * 2 n_out
  const int64_t sup = 4 * static_cast<int64_t>(down ? n_in : n_out);           // 2 fs * 2 n_out
  const int64_t d = 2 * static_cast<int64_t>(n_out);
  int64_t a = floor_div(cn - sup, d), e = ceil_div(cn + sup, d);
  if (a < 0) a = 0;
  if (e > n_in) e = n_in;
  Win w;
  w.lo = static_cast<int>(a);
  w.n = static_cast<int>(e - a);
  w.num0 = static_cast<int>((2 * a + 1) * n_out - cn);
  w.step = 2 * n_out;
  w.inv_den = 1.0f / static_cast<float>(down ? 2 * n_in : 2 * n_out);
  return w;
}

// Window [lo, lo + n) of taps for output index o, the tap offset of lo, its step, 1/sum(weights).
__device__ __forceinline__ void window_1d(int o, int n_in, int n_out, int& lo, int& n, float& off0, float& ifs,
                                          float& inorm) {
  const Win w = exact_window(o, n_in, n_out);
  lo = w.lo;
  n = w.n;
  off0 = static_cast<float>(w.num0) * w.inv_den;
  ifs = static_cast<float>(w.step) * w.inv_den;
  float s = 0.f;
  for (int i = 0; i < n; ++i) s += cubic_w(static_cast<float>(w.num0 + i * w.step) * w.inv_den);
  inorm = 1.0f / s;
}

// Any downscale: one 4 x 32 output tile, weights evaluated per tap, input read through L1.
__device__ void resample_tile_generic(const uint8_t* __restrict__ img, int H, int W, int Ho, int Wo, int ox0,
                                      int oy0, uint8_t* __restrict__ out) {
  __shared__ int xlo[kRsTW], xn[kRsTW];
  __shared__ float xoff[kRsTW], xifs[kRsTW], xnorm[kRsTW];
  __shared__ int ylo[kRsTH], yn[kRsTH];
  __shared__ float yoff[kRsTH], yifs[kRsTH], ynorm[kRsTH];
  __shared__ float hbuf[kRsChunk][kRsTW][3];
  if (ox0 >= Wo || oy0 >= Ho) return;
  const int tid = threadIdx.x;
  if (tid < kRsTW) {
    const int ox = min(ox0 + tid, Wo - 1);
    window_1d(ox, W, Wo, xlo[tid], xn[tid], xoff[tid], xifs[tid], xnorm[tid]);
  } else if (tid >= 32 && tid < 32 + kRsTH) {
    const int i = tid - 32;
    const int oy = min(oy0 + i, Ho - 1);
    window_1d(oy, H, Ho, ylo[i], yn[i], yoff[i], yifs[i], ynorm[i]);
  }
  __syncthreads();
  const int nrows = min(kRsTH, Ho - oy0);
  const int iy_lo = ylo[0];
  const int iy_hi = ylo[nrows - 1] + yn[nrows - 1];  // exclusive
  const int64_t pitch = static_cast<int64_t>(W) * 3;
  // this thread's output pixel
  const int my_r = tid / kRsTW, my_c = tid % kRsTW;
  float acc0 = 0.f, acc1 = 0.f, acc2 = 0.f;
  for (int r0 = iy_lo; r0 < iy_hi; r0 += kRsChunk) {
    // horizontal pass: kRsChunk rows x 32 columns x 3 channels
    for (int v = tid; v < kRsChunk * kRsTW * 3; v += kRsThreads) {
      const int rr = v / (kRsTW * 3), rem = v - rr * (kRsTW * 3);
      const int cc = rem / 3, ch = rem - cc * 3;
      const int iy = r0 + rr;
      float h = 0.f;
      if (iy < iy_hi) {
        const uint8_t* row = img + iy * pitch + ch;
        const int lo = xlo[cc], n = xn[cc];
        const float off = xoff[cc], ifs = xifs[cc];
        for (int i = 0; i < n; ++i) h = fmaf(cubic_w(fmaf(static_cast<float>(i), ifs, off)),
                                             static_cast<float>(__ldg(row + 3 * (lo + i))), h);
        h *= xnorm[cc];
      }
      hbuf[rr][cc][ch] = h;
    }
    __syncthreads();
    if (my_r < nrows) {
      const int lo = ylo[my_r], n = yn[my_r];
      const float off = yoff[my_r], ifs = yifs[my_r];
      for (int rr = 0; rr < kRsChunk; ++rr) {
        const int i = r0 + rr - lo;
        if (i >= 0 && i < n) {
          const float w = cubic_w(fmaf(static_cast<float>(i), ifs, off));
          acc0 = fmaf(w, hbuf[rr][my_c][0], acc0);
          acc1 = fmaf(w, hbuf[rr][my_c][1], acc1);
          acc2 = fmaf(w, hbuf[rr][my_c][2], acc2);
        }
      }
    }
    __syncthreads();
  }
  const int oy = oy0 + my_r, ox = ox0 + my_c;
  if (my_r < nrows && ox < Wo) {
    const float nrm = ynorm[my_r];
    uint8_t* o = out + (static_cast<int64_t>(oy) * Wo + ox) * 3;
    o[0] = static_cast<uint8_t>(min(255, max(0, __float2int_rn(acc0 * nrm))));
    o[1] = static_cast<uint8_t>(min(255, max(0, __float2int_rn(acc1 * nrm))));
    o[2] = static_cast<uint8_t>(min(255, max(0, __float2int_rn(acc2 * nrm))));
  }
  __syncthreads();   // shared tile buffers are reused by the next call
}

// Downscale of at most 2.75 per side: one 16 x 32 output tile.  The CTA stages its whole
// input window in shared memory with 4-byte loads (every image starts 16-byte aligned and
// holds a multiple of 4 bytes, so the rounded loads stay inside it) and precomputes the
// normalised tap weights of its rows and columns; thread (column, channel) keeps its column's
// weights in registers, filters every staged row horizontally into a shared fp32 buffer and
// then its output column vertically.
constexpr int kFTH = 16, kFTW = 32, kFMaxTaps = 14;
// the fast path takes downscales of at most 2.75 = 11 / 4 per side (tested as 4 n_in <= 11 n_out)
constexpr int kFRows = 58;                   // >= 16 * 2.75 + 14 staged input rows
constexpr int kFCols = 118;                  // >= 32 * 2.75 + 14 window pixels + 14 read past it (weight 0)
constexpr int kFPitch = 368;                 // bytes per staged row: 3 * kFCols + 3 alignment slack, rounded
constexpr int kFLine = kFTW * 3;             // floats per row of the horizontal result
static_assert(kFPitch >= 3 * kFCols + 6 && kFPitch % 16 == 0, "staged row pitch");
static_assert(kFRows >= kFTH * 2.75 + 14 && kFCols >= kFTW * 2.75 + 14 + kFMaxTaps, "staged window");
static_assert(3 * kFTW <= kRsThreads / 2 && 64 + kFTH <= kRsThreads, "thread roles of the fast tile");
constexpr size_t kFSmem = static_cast<size_t>(kFRows) * kFPitch + static_cast<size_t>(kFRows) * kFLine * 4 +
                          (kFTW + kFTH) * kFMaxTaps * 4 + (2 * kFTW + 2 * kFTH + kFRows + 4) * 4;
constexpr int kRsCtasPerSm = 4;

// Normalised weights of the window of output index o (reading R5); returns the tap count.
__device__ __forceinline__ int window_weights(int o, int n_in, int n_out, int& lo, float* w) {
  const Win win = exact_window(o, n_in, n_out);
  if (win.n > kFMaxTaps) return win.n;
  float sum = 0.f;
  for (int i = 0; i < win.n; ++i) {
    w[i] = cubic_w(static_cast<float>(win.num0 + i * win.step) * win.inv_den);
    sum += w[i];
  }
  const float inv = 1.0f / sum;
  for (int i = 0; i < win.n; ++i) w[i] *= inv;
  lo = win.lo;
  return win.n;
}

template <int MAXT>
__device__ __forceinline__ void resample_tile_fast(const uint8_t* __restrict__ img, int H, int W, int Ho, int Wo,
                                                   int ox0, int oy0, uint8_t* __restrict__ out) {
  extern __shared__ __align__(16) unsigned char rs_smem[];
  unsigned char* sin = rs_smem;                                           // [kFRows][kFPitch] bytes
  float* sh = reinterpret_cast<float*>(sin + kFRows * kFPitch);            // [kFRows][kFTW * 3]
  float* wx = sh + kFRows * kFLine;                                        // [kFTW][kFMaxTaps]
  float* wy = wx + kFTW * kFMaxTaps;                                       // [kFTH][kFMaxTaps]
  int* xlo = reinterpret_cast<int*>(wy + kFTH * kFMaxTaps);
  int* xn = xlo + kFTW;
  int* ylo = xn + kFTW;
  int* yn = ylo + kFTH;
  int* shift = yn + kFTH;                                                  // [kFRows]
  const int tid = threadIdx.x;
  const int ncol = min(kFTW, Wo - ox0), nrow = min(kFTH, Ho - oy0);
  // with both scales <= 2.75 every window has <= 4 * 2.75 + 2 = 13 taps (min() is a guard)
  if (tid < ncol) xn[tid] = min(kFMaxTaps, window_weights(ox0 + tid, W, Wo, xlo[tid], wx + tid * kFMaxTaps));
  if (tid >= 64 && tid < 64 + nrow)
    yn[tid - 64] =
        min(kFMaxTaps, window_weights(oy0 + tid - 64, H, Ho, ylo[tid - 64], wy + (tid - 64) * kFMaxTaps));
  __syncthreads();
  const int x0 = xlo[0], x1 = xlo[ncol - 1] + xn[ncol - 1];
  const int y0 = ylo[0], y1 = ylo[nrow - 1] + yn[nrow - 1];
  const int nin_c = x1 - x0, nin_r = y1 - y0;
  // stage the input window (4-byte words covering each row segment), asynchronously: a warp per
  // row, every copy in flight at once
  const int64_t pitch = static_cast<int64_t>(W) * 3;
  const int64_t img_bytes = static_cast<int64_t>(H) * pitch;
  const int words = (nin_c * 3 + 3 + 3) >> 2;
  for (int r = tid >> 5; r < nin_r; r += kRsThreads / 32) {
    const int64_t start = (static_cast<int64_t>(y0 + r) * pitch + static_cast<int64_t>(x0) * 3);
    const int64_t a = start & ~int64_t{3};
    if ((tid & 31) == 0) shift[r] = static_cast<int>(start - a);
    for (int w = tid & 31; w < words; w += 32)
      if (a + 4 * w < img_bytes) cp_async4(sin + r * kFPitch + 4 * w, img + a + 4 * w);
  }
  cp_async_wait_all();
  __syncthreads();
  // the two halves of the CTA take the two halves of the rows; thread tt = (column, channel)
  const int half = tid / (kRsThreads / 2), tt = tid - half * (kRsThreads / 2);
  if (tt < 3 * ncol) {
    // horizontal pass: this half's staged rows, this thread's (column, channel)
    // (taps past the window have weight 0 and read staged bytes that exist: the staged row
    // holds kFCols >= the window of the last column + MAXT pixels)
    const int c = tt / 3, ch = tt - 3 * c;
    const int n = xn[c];
    // A byte b enters as the float 1 + b / 256 (b in the top 8 mantissa bits of 1.0, one integer
    // multiply-add), so sum_k w_k (1 + b_k / 256) = W + (sum_k w_k b_k) / 256 with W = sum_k w_k;
    // the accumulators stay in [1, 2) (fp32 steps of 2^-23, i.e. 3e-5 in pixel units after the
    // final 256 (acc - W)), and two rows share each packed FMA.
    float w[MAXT];
    float wsum = 0.f;
#pragma unroll
    for (int k = 0; k < MAXT; ++k) {
      w[k] = k < n ? wx[c * kFMaxTaps + k] : 0.f;
      wsum += w[k];
    }
    const float2 post = make_float2(-256.0f * wsum, -256.0f * wsum);
    const float2 k256 = make_float2(256.0f, 256.0f);
    auto unit = [](unsigned b) { return __uint_as_float(b * 32768u + 0x3F800000u); };
    const int base = (xlo[c] - x0) * 3 + ch;
    const int r_end = half ? nin_r : (nin_r + 1) / 2;
    int r = half ? (nin_r + 1) / 2 : 0;
    for (; r + 1 < r_end; r += 2) {   // two rows at a time: twice the independent work in flight
      const unsigned char* px0 = sin + r * kFPitch + shift[r] + base;
      const unsigned char* px1 = sin + (r + 1) * kFPitch + shift[r + 1] + base;
      float2 acc = make_float2(0.f, 0.f);
#pragma unroll
      for (int k = 0; k < MAXT; ++k)
        acc = ptx::ffma2(make_float2(w[k], w[k]), make_float2(unit(px0[3 * k]), unit(px1[3 * k])), acc);
      const float2 h = ptx::ffma2(acc, k256, post);
      sh[r * kFLine + tt] = h.x;
      sh[(r + 1) * kFLine + tt] = h.y;
    }
    if (r < r_end) {
      const unsigned char* px = sin + r * kFPitch + shift[r] + base;
      float acc = 0.f;
#pragma unroll
      for (int k = 0; k < MAXT; ++k) acc = fmaf(w[k], unit(px[3 * k]), acc);
      sh[r * kFLine + tt] = fmaf(acc, 256.0f, post.x);
    }
  }
  __syncthreads();
  // vertical pass and the uint8 store (a row of the tile is 3 * ncol consecutive bytes): thread
  // (g, p) of 4 x 48 filters line entries 2p and 2p + 1 of output rows g, g + 4, .. with one
  // 8-byte load and one packed FMA per tap (entry 3 * ncol, past the line when it is odd, holds
  // whatever the buffer held and is not stored)
  constexpr int kVPairs = kFLine / 2;
  static_assert(4 * kVPairs <= kRsThreads, "thread roles of the vertical pass");
  const int vg = tid / kVPairs, t0 = 2 * (tid - vg * kVPairs);
  if (vg < 4 && t0 < 3 * ncol) {
    const bool two = t0 + 1 < 3 * ncol;
    uint8_t* o = out + (static_cast<int64_t>(oy0) * Wo + ox0) * 3 + t0;
    for (int r = vg; r < nrow; r += 4) {
      const float* w = wy + r * kFMaxTaps;
      const float2* col = reinterpret_cast<const float2*>(sh + (ylo[r] - y0) * kFLine + t0);
      const int n = yn[r];
      float2 acc = make_float2(0.f, 0.f);
#pragma unroll 4
      for (int k = 0; k < n; ++k) acc = ptx::ffma2(make_float2(w[k], w[k]), col[k * kVPairs], acc);
      uint8_t* orow = o + static_cast<int64_t>(r) * Wo * 3;
      orow[0] = static_cast<uint8_t>(min(255, max(0, __float2int_rn(acc.x))));
      if (two) orow[1] = static_cast<uint8_t>(min(255, max(0, __float2int_rn(acc.y))));
    }
  }
  __syncthreads();   // the shared buffers are reused by the next tile
}

// Every CTA walks the output tiles of the whole batch (16 x 32 tiles; target sizes read from
// the density statistics on the device, or given), so the grid never holds empty CTAs.
__global__ void __launch_bounds__(kRsThreads) apc_resample(const uint8_t* __restrict__ src,
                                                           const __grid_constant__ ResampleTable t,
                                                           const pace_apc_stats* __restrict__ stats,
                                                           uint8_t* __restrict__ dst) {
  __shared__ int tile_prefix[kApcMaxB + 1];
  __shared__ int sho[kApcMaxB], swo[kApcMaxB];
  if (threadIdx.x == 0) {
    int acc = 0;
    for (int b = 0; b < t.nb; ++b) {
      int Ho = stats ? stats[t.b_base + b].h_out : t.Ho[b];
      int Wo = stats ? stats[t.b_base + b].w_out : t.Wo[b];
      if (Ho < 1 || Wo < 1 || Ho > t.H[b] || Wo > t.W[b]) Ho = Wo = 0;   // nothing to write
      sho[b] = Ho;
      swo[b] = Wo;
      tile_prefix[b] = acc;
      acc += ((Ho + kFTH - 1) / kFTH) * ((Wo + kFTW - 1) / kFTW);
    }
    tile_prefix[t.nb] = acc;
  }
  __syncthreads();
  const int total = tile_prefix[t.nb];
  for (int g = blockIdx.x; g < total; g += gridDim.x) {
    int b = 0;
    while (b + 1 < t.nb && tile_prefix[b + 1] <= g) ++b;
    const int Ho = sho[b], Wo = swo[b], H = t.H[b], W = t.W[b];
    const int tw = (Wo + kFTW - 1) / kFTW;
    const int l = g - tile_prefix[b];
    const int oy0 = (l / tw) * kFTH, ox0 = (l - (l / tw) * tw) * kFTW;
    const uint8_t* img = src + t.src_off[b];
    uint8_t* out = dst + t.dst_off[b];
    if (4 * W <= 11 * Wo && 4 * H <= 11 * Ho) {   // both scales <= 2.75 = 11 / 4
      if (4 * W <= 9 * Wo && 4 * H <= 9 * Ho) resample_tile_fast<10>(img, H, W, Ho, Wo, ox0, oy0, out);   // <= 10 taps
      else resample_tile_fast<kFMaxTaps>(img, H, W, Ho, Wo, ox0, oy0, out);
    } else {
        for (int sy = 0; sy < kFTH; sy += kRsTH)
        for (int sx = 0; sx < kFTW; sx += kRsTW) resample_tile_generic(img, H, W, Ho, Wo, ox0 + sx, oy0 + sy, out);
    }
  }
}

// ------------------------------------------------------------------------------------------------
// host side
// ------------------------------------------------------------------------------------------------
struct DensityLayout {
  size_t sums_off, work_off, zero_bytes, inv_off, d_off, total;   // [0, zero_bytes) is zeroed per call
  int64_t n_total;
};

DensityLayout density_layout(int B, const int32_t* H, const int32_t* W) {
  DensityLayout L{};
  int64_t n = 0;
  for (int b = 0; b < B; ++b) n += static_cast<int64_t>(H[b] / kPatch) * (W[b] / kPatch);
  L.n_total = n;
  L.sums_off = 0;
  L.work_off = align_up(static_cast<size_t>(B) * kTokDim * sizeof(unsigned long long), 256);
  L.zero_bytes = L.work_off + static_cast<size_t>(B) * sizeof(TailWork);
  L.inv_off = align_up(L.zero_bytes, 256);
  L.d_off = L.inv_off + align_up(static_cast<size_t>(n) * sizeof(float), 256);
  L.total = L.d_off + align_up(static_cast<size_t>(n) * sizeof(float), 256);
  return L;
}

// Grid of the strip passes: the CTAs that are resident at once (capped by the strips).
unsigned strip_grid(int units) {
  static std::atomic<int> cap[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) dev = 0;
  int c = cap[dev & 63].load(std::memory_order_relaxed);
  if (c == 0) {
    int nsm = 0, per = 0;
    cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per, apc_pass2<true>, kApcThreads, 0);
    c = std::max(1, nsm * std::max(per, 1));
    cap[dev & 63].store(c, std::memory_order_relaxed);
  }
  return static_cast<unsigned>(std::max(1, std::min(units, c)));
}

// Launches apc_tail_scan on one ApcTable: kTailChunk distances per CTA, the largest image's
// chunks per row of the grid (CTAs past a smaller image's chunks return at once).
void launch_tail_scan(const ApcTable& t, const float* d, TailParams tp, pace_apc_stats* stats, TailWork* work,
                      cudaStream_t stream) {
  int chunks = 1;
  for (int i = 0; i < t.nb; ++i) chunks = std::max(chunks, (t.n[i] + kTailChunk - 1) / kTailChunk);
  apc_tail_scan<<<dim3(static_cast<unsigned>(chunks), static_cast<unsigned>(t.nb)), 1024, 0, stream>>>(t, d, tp, stats,
                                                                                                     work);
}


pace_status_t check_images(const uint8_t* img, const int64_t* off, const int32_t* H, const int32_t* W, int B) {
  if (B < 0) return PACE_ERR_INVALID_ARG;
  if (B == 0) return PACE_OK;
  if (img == nullptr || off == nullptr || H == nullptr || W == nullptr) return PACE_ERR_INVALID_ARG;
  for (int b = 0; b < B; ++b) {
    if (H[b] < kPatch || W[b] < kPatch || H[b] % kPatch || W[b] % kPatch) return PACE_ERR_INVALID_ARG;
    if (off[b] < 0 || (reinterpret_cast<uintptr_t>(img) + off[b]) % 16) return PACE_ERR_INVALID_ARG;
    if (static_cast<int64_t>(H[b]) * W[b] > (int64_t{1} << 30)) return PACE_ERR_INVALID_ARG;
  }
  return PACE_OK;
}

}  // namespace
}  // namespace pace

using namespace pace;

extern "C" size_t pace_apc_density_workspace_size(int B, const int32_t* H, const int32_t* W) {
  if (B <= 0 || H == nullptr || W == nullptr) return 0;
  for (int b = 0; b < B; ++b)
    if (H[b] < kPatch || W[b] < kPatch) return 0;
  return density_layout(B, H, W).total;
}

extern "C" pace_status_t pace_apc_density(const uint8_t* img, const int64_t* img_off, const int32_t* H,
                                          const int32_t* W, int B, const pace_apc_params* params, float* d_out,
                                          pace_apc_stats* stats, void* ws, size_t ws_bytes,
                                          pace_stream_t stream) {
  PACE_CHECK(check_images(img, img_off, H, W, B));
  if (B == 0) return PACE_OK;
  if (stats == nullptr) return PACE_ERR_INVALID_ARG;
  pace_apc_params p;
  if (params) p = *params; else pace_apc_params_default(&p);
  if (!(p.tail_frac > 0.f && p.tail_frac <= 1.f) || !(p.gamma > 0.f) || !(p.alpha >= 0.f && p.alpha <= 1.f) ||
      !(p.r_min <= p.r_max) || p.align < 1)
    return PACE_ERR_INVALID_ARG;
  const DensityLayout L = density_layout(B, H, W);
  if (ws == nullptr || ws_bytes < L.total || reinterpret_cast<uintptr_t>(ws) % 16) return PACE_ERR_WORKSPACE;
  PACE_CHECK(check_device());
  uint8_t* w8 = static_cast<uint8_t*>(ws);
  auto* sums = reinterpret_cast<unsigned long long*>(w8 + L.sums_off);
  auto* work = reinterpret_cast<TailWork*>(w8 + L.work_off);
  auto* inv = reinterpret_cast<float*>(w8 + L.inv_off);
  float* d = d_out ? d_out : reinterpret_cast<float*>(w8 + L.d_off);
  PACE_CUDA(cudaMemsetAsync(w8, 0, L.zero_bytes, stream));   // column sums and tail scratch
  int patch0 = 0;
  for (int c0 = 0; c0 < B; c0 += kApcMaxB) {
    const int nb = (B - c0) < kApcMaxB ? (B - c0) : kApcMaxB;
    ApcTable t{};
    t.nb = nb;
    t.b_base = c0;
    t.unit_prefix[0] = 0;
    bool wide = true;
    for (int i = 0; i < nb; ++i) {
      const int b = c0 + i;
      t.off[i] = img_off[b];
      t.H[i] = H[b];
      t.W[i] = W[b];
      t.gw[i] = W[b] / kPatch;
      t.chunks[i] = (t.gw[i] + kStrip - 1) / kStrip;
      t.patch0[i] = patch0;
      const int N = (H[b] / kPatch) * t.gw[i];
      t.n[i] = N;
      double kt = std::floor(static_cast<double>(p.tail_frac) * N + 0.5);
      if (kt < 1) kt = 1;
      if (kt > N) kt = N;
      t.ktail[i] = static_cast<int>(kt);
      patch0 += N;
      t.unit_prefix[i + 1] = t.unit_prefix[i] + (H[b] / kPatch) * t.chunks[i];
      if ((static_cast<int64_t>(W[b]) * 3) % 4 != 0 || (t.gw[i] % 2) != 0 || (img_off[b] % 4) != 0) wide = false;
    }
    const int units = t.unit_prefix[nb];
    if (wide) apc_pass1<true><<<strip_grid(units), kApcThreads, 0, stream>>>(img, t, units, inv, sums);
    else apc_pass1<false><<<strip_grid(units), kApcThreads, 0, stream>>>(img, t, units, inv, sums);
    PACE_CHECK(check_launch());
    if (wide) apc_pass2<true><<<strip_grid(units), kApcThreads, 0, stream>>>(img, t, units, inv, sums, d, stats, work);
    else apc_pass2<false><<<strip_grid(units), kApcThreads, 0, stream>>>(img, t, units, inv, sums, d, stats, work);
    PACE_CHECK(check_launch());
    TailParams tp{p.alpha, p.gamma, p.r_min, p.r_max, p.align};
    launch_tail_scan(t, d, tp, stats, work, stream);
    PACE_CHECK(check_launch());
  }
  return PACE_OK;
}

static pace_status_t resample_impl(const uint8_t* src, const int64_t* src_off, const int32_t* H, const int32_t* W,
                                   const int32_t* Ho, const int32_t* Wo, const pace_apc_stats* stats,
                                   uint8_t* dst, const int64_t* dst_off, int B, pace_stream_t stream) {
  PACE_CHECK(check_images(src, src_off, H, W, B));
  if (B == 0) return PACE_OK;
  if (dst == nullptr || dst_off == nullptr) return PACE_ERR_INVALID_ARG;
  if (stats == nullptr) {
    if (Ho == nullptr || Wo == nullptr) return PACE_ERR_INVALID_ARG;
    for (int b = 0; b < B; ++b)
      if (Ho[b] < 1 || Wo[b] < 1 || Ho[b] > H[b] || Wo[b] > W[b]) return PACE_ERR_INVALID_ARG;
  }
  for (int b = 0; b < B; ++b)
    if (dst_off[b] < 0) return PACE_ERR_INVALID_ARG;
  PACE_CHECK(check_device());
  int sms = 1;
  {
    // opt in to the fast path's shared memory and read the SM count, once per device
    static DeviceOnce once;
    static std::atomic<int> sm_count[64];
    int dev = 0;
    PACE_CUDA(cudaGetDevice(&dev));
    if (!once.done(dev)) {
      int n = 0;
      PACE_CUDA(cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev));
      sm_count[dev & 63].store(n, std::memory_order_relaxed);
      PACE_CUDA(cudaFuncSetAttribute(apc_resample, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     static_cast<int>(kFSmem)));
      once.mark(dev);
    }
    sms = std::max(sm_count[dev & 63].load(std::memory_order_relaxed), 1);
  }
  for (int c0 = 0; c0 < B; c0 += kApcMaxB) {
    const int nb = (B - c0) < kApcMaxB ? (B - c0) : kApcMaxB;
    ResampleTable t{};
    t.nb = nb;
    t.b_base = c0;
    int hmax = 1, wmax = 1;
    for (int i = 0; i < nb; ++i) {
      const int b = c0 + i;
      t.src_off[i] = src_off[b];
      t.dst_off[i] = dst_off[b];
      t.H[i] = H[b];
      t.W[i] = W[b];
      t.Ho[i] = stats ? H[b] : Ho[b];
      t.Wo[i] = stats ? W[b] : Wo[b];
      if (t.Ho[i] > hmax) hmax = t.Ho[i];
      if (t.Wo[i] > wmax) wmax = t.Wo[i];
    }
    const int64_t tiles = static_cast<int64_t>((wmax + kFTW - 1) / kFTW) * ((hmax + kFTH - 1) / kFTH) * nb;
    const int grid = static_cast<int>(std::min<int64_t>(tiles, static_cast<int64_t>(kRsCtasPerSm) * sms));
    apc_resample<<<grid, kRsThreads, kFSmem, stream>>>(src, t, stats, dst);
    PACE_CHECK(check_launch());
  }
  return PACE_OK;
}

extern "C" pace_status_t pace_apc_resample(const uint8_t* src, const int64_t* src_off, const int32_t* H,
                                           const int32_t* W, const pace_apc_stats* stats, uint8_t* dst,
                                           const int64_t* dst_off, int B, pace_stream_t stream) {
  if (B > 0 && stats == nullptr) return PACE_ERR_INVALID_ARG;
  return resample_impl(src, src_off, H, W, nullptr, nullptr, stats, dst, dst_off, B, stream);
}

extern "C" pace_status_t pace_apc_resample_to(const uint8_t* src, const int64_t* src_off, const int32_t* H,
                                              const int32_t* W, const int32_t* H_out, const int32_t* W_out,
                                              uint8_t* dst, const int64_t* dst_off, int B, pace_stream_t stream) {
  return resample_impl(src, src_off, H, W, H_out, W_out, nullptr, dst, dst_off, B, stream);
}

// ------------------------------------------------------------------------------------------------
// pace_apc_density_static: the same density computation with library-owned scratch
// ------------------------------------------------------------------------------------------------
// Scratch of pace_apc_density_static, in a file-scope device array instead of caller memory:
// the per-image 589-entry fixed-point column sums, then the per-patch inverse token norms.
// Every GPU that loads the library holds this array until the process exits.
namespace pace {
namespace {
constexpr size_t kStaticSumsBytes =
    static_cast<size_t>(PACE_APC_STATIC_MAX_IMAGES) * kTokDim * sizeof(unsigned long long);
constexpr size_t kStaticWorkOff = (kStaticSumsBytes + 255) / 256 * 256;
constexpr size_t kStaticZeroBytes = kStaticWorkOff + static_cast<size_t>(PACE_APC_STATIC_MAX_IMAGES) * sizeof(TailWork);
constexpr size_t kStaticInvOff = (kStaticZeroBytes + 255) / 256 * 256;
constexpr size_t kStaticBytes = kStaticInvOff + static_cast<size_t>(PACE_APC_STATIC_MAX_PATCHES) * sizeof(float);

static __device__ __align__(256) unsigned char g_apc_static_scratch[kStaticBytes];

std::mutex g_static_mutex;
void* g_static_ptr[kMaxDevices] = {};
DeviceOnce g_static_once;

// Device address of the array for the current device.  The name g_apc_static_scratch in host
// code is only a host-side handle, so the address is looked up once per device and set-up
// generation (pace_init starts a new one, e.g. after cudaDeviceReset).
pace_status_t static_scratch(unsigned char** out) {
  int dev = -1;
  PACE_CUDA(cudaGetDevice(&dev));
  if (dev < 0 || dev >= kMaxDevices) return PACE_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> lk(g_static_mutex);
  if (!g_static_once.done(dev)) {
    void* p = nullptr;
    PACE_CUDA(cudaGetSymbolAddress(&p, g_apc_static_scratch));
    if (p == nullptr) return set_cuda_error(cudaErrorInvalidSymbol);
    g_static_ptr[dev] = p;
    g_static_once.mark(dev);
  }
  *out = static_cast<unsigned char*>(g_static_ptr[dev]);
  return PACE_OK;
}
}  // namespace
}  // namespace pace

extern "C" pace_status_t pace_apc_density_static(const uint8_t* img, const int64_t* img_off, const int32_t* H,
                                                 const int32_t* W, int B, const pace_apc_params* params,
                                                 float* d_out, pace_apc_stats* stats, pace_stream_t stream) {
  PACE_CHECK(check_images(img, img_off, H, W, B));
  if (B == 0) return PACE_OK;
  if (stats == nullptr || d_out == nullptr) return PACE_ERR_INVALID_ARG;
  if (B > PACE_APC_STATIC_MAX_IMAGES) return PACE_ERR_INVALID_ARG;
  int64_t n_total = 0;
  for (int b = 0; b < B; ++b) n_total += static_cast<int64_t>(H[b] / kPatch) * (W[b] / kPatch);
  if (n_total > PACE_APC_STATIC_MAX_PATCHES) return PACE_ERR_INVALID_ARG;
  pace_apc_params p;
  if (params) p = *params; else pace_apc_params_default(&p);
  if (!(p.tail_frac > 0.f && p.tail_frac <= 1.f) || !(p.gamma > 0.f) || !(p.alpha >= 0.f && p.alpha <= 1.f) ||
      !(p.r_min <= p.r_max) || p.align < 1)
    return PACE_ERR_INVALID_ARG;
  PACE_CHECK(check_device());
  unsigned char* scratch = nullptr;
  PACE_CHECK(static_scratch(&scratch));
  auto* sums = reinterpret_cast<unsigned long long*>(scratch);
  auto* work = reinterpret_cast<TailWork*>(scratch + kStaticWorkOff);
  auto* inv = reinterpret_cast<float*>(scratch + kStaticInvOff);
  // the array keeps the previous call's contents: the column sums and the tail scratch of the
  // call's images must start from zero
  PACE_CUDA(cudaMemsetAsync(sums, 0, static_cast<size_t>(B) * kTokDim * sizeof(unsigned long long), stream));
  PACE_CUDA(cudaMemsetAsync(work, 0, static_cast<size_t>(B) * sizeof(TailWork), stream));
  ApcTable t{};
  t.nb = B;
  t.b_base = 0;
  t.unit_prefix[0] = 0;
  bool wide = true;
  int patch0 = 0;
  for (int b = 0; b < B; ++b) {
    t.off[b] = img_off[b];
    t.H[b] = H[b];
    t.W[b] = W[b];
    t.gw[b] = W[b] / kPatch;
    t.chunks[b] = (t.gw[b] + kStrip - 1) / kStrip;
    t.patch0[b] = patch0;
    const int N = (H[b] / kPatch) * t.gw[b];
    t.n[b] = N;
    double kt = std::floor(static_cast<double>(p.tail_frac) * N + 0.5);
    if (kt < 1) kt = 1;
    if (kt > N) kt = N;
    t.ktail[b] = static_cast<int>(kt);
    patch0 += N;
    t.unit_prefix[b + 1] = t.unit_prefix[b] + (H[b] / kPatch) * t.chunks[b];
    if ((static_cast<int64_t>(W[b]) * 3) % 4 != 0 || (t.gw[b] % 2) != 0 || (img_off[b] % 4) != 0) wide = false;
  }
  const int units = t.unit_prefix[B];
  if (wide) apc_pass1<true><<<strip_grid(units), kApcThreads, 0, stream>>>(img, t, units, inv, sums);
  else apc_pass1<false><<<strip_grid(units), kApcThreads, 0, stream>>>(img, t, units, inv, sums);
  PACE_CHECK(check_launch());
  if (wide) apc_pass2<true><<<strip_grid(units), kApcThreads, 0, stream>>>(img, t, units, inv, sums, d_out, stats, work);
  else apc_pass2<false><<<strip_grid(units), kApcThreads, 0, stream>>>(img, t, units, inv, sums, d_out, stats, work);
  PACE_CHECK(check_launch());
  TailParams tp{p.alpha, p.gamma, p.r_min, p.r_max, p.align};
  launch_tail_scan(t, d_out, tp, stats, work, stream);
  return check_launch();
}

// ------------------------------------------------------------------------------------------------
// pace_apc_density_tokens: Eq. 1-6 on preview tokens
// ------------------------------------------------------------------------------------------------
namespace pace {
namespace {
// Opts pass 1 of the token density into two 40 KB stages (once per device).
pace_status_t tok_pass1_attr() {
  static DeviceOnce once;
  int dev = 0;
  PACE_CUDA(cudaGetDevice(&dev));
  if (once.done(dev)) return PACE_OK;
  PACE_CUDA(cudaFuncSetAttribute(apc_tok_pass1, cudaFuncAttributeMaxDynamicSharedMemorySize, 2 * kTok1StageBytes));
  once.mark(dev);
  return PACE_OK;
}

// Grid of pass 1: the CTAs resident at once (capped by the chunks).
unsigned tok_pass1_grid(int units) {
  static std::atomic<int> cap[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) dev = 0;
  int c = cap[dev & 63].load(std::memory_order_relaxed);
  if (c == 0) {
    int nsm = 0, per = 0;
    cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per, apc_tok_pass1, kApcThreads, 2 * kTok1StageBytes);
    c = std::max(1, nsm * std::max(per, 1));
    cap[dev & 63].store(c, std::memory_order_relaxed);
  }
  return static_cast<unsigned>(std::max(1, std::min(units, c)));
}

struct TokLayout {
  size_t sums_off, work_off, zero_bytes, inv_off, total;   // [0, zero_bytes) is zeroed per call
};
TokLayout tok_layout(int B, const int32_t* cu, int D) {
  TokLayout L{};
  L.sums_off = 0;
  L.work_off = align_up(static_cast<size_t>(B) * D * sizeof(unsigned long long), 256);
  L.zero_bytes = L.work_off + static_cast<size_t>(B) * sizeof(TailWork);
  L.inv_off = align_up(L.zero_bytes, 256);
  L.total = L.inv_off + align_up(static_cast<size_t>(cu[B]) * sizeof(float), 256);
  return L;
}
}  // namespace
}  // namespace pace

extern "C" size_t pace_apc_density_tokens_workspace_size(int B, const int32_t* cu_tokens, int D) {
  if (B <= 0 || cu_tokens == nullptr || D < 2) return 0;
  return tok_layout(B, cu_tokens, D).total;
}

extern "C" pace_status_t pace_apc_density_tokens(const void* T, const int32_t* cu_tokens, int B, int D,
                                                 const int32_t* H, const int32_t* W,
                                                 const pace_apc_params* params, float* d_out,
                                                 pace_apc_stats* stats, void* ws, size_t ws_bytes,
                                                 pace_stream_t stream) {
  if (B < 0) return PACE_ERR_INVALID_ARG;
  if (B == 0) return PACE_OK;
  if (T == nullptr || cu_tokens == nullptr || H == nullptr || W == nullptr || d_out == nullptr || stats == nullptr)
    return PACE_ERR_INVALID_ARG;
  if (D < 2 || D > kTokMaxD || D % 2 != 0 || reinterpret_cast<uintptr_t>(T) % 4 != 0) return PACE_ERR_INVALID_ARG;
  if (cu_tokens[0] != 0) return PACE_ERR_INVALID_ARG;
  for (int b = 0; b < B; ++b)
    if (cu_tokens[b + 1] - cu_tokens[b] < 1 || H[b] < 1 || W[b] < 1) return PACE_ERR_INVALID_ARG;
  pace_apc_params p;
  if (params) p = *params; else pace_apc_params_default(&p);
  if (!(p.tail_frac > 0.f && p.tail_frac <= 1.f) || !(p.gamma > 0.f) || !(p.alpha >= 0.f && p.alpha <= 1.f) ||
      !(p.r_min <= p.r_max) || p.align < 1)
    return PACE_ERR_INVALID_ARG;
  const TokLayout L = tok_layout(B, cu_tokens, D);
  if (ws == nullptr || ws_bytes < L.total || reinterpret_cast<uintptr_t>(ws) % 16) return PACE_ERR_WORKSPACE;
  PACE_CHECK(check_device());
  uint8_t* w8 = static_cast<uint8_t*>(ws);
  auto* sums = reinterpret_cast<unsigned long long*>(w8 + L.sums_off);
  auto* work = reinterpret_cast<TailWork*>(w8 + L.work_off);
  auto* inv = reinterpret_cast<float*>(w8 + L.inv_off);
  PACE_CUDA(cudaMemsetAsync(w8, 0, L.zero_bytes, stream));   // column sums and tail scratch
  const uint32_t* T32 = static_cast<const uint32_t*>(T);
  for (int c0 = 0; c0 < B; c0 += kApcMaxB) {
    const int nb = (B - c0) < kApcMaxB ? (B - c0) : kApcMaxB;
    TokTable tt{};
    ApcTable at{};   // what the tail kernel reads: sizes, token ranges, k_tail
    tt.nb = at.nb = nb;
    tt.b_base = at.b_base = c0;
    tt.D = D;
    tt.rows1 = std::max(1, std::min(32, kTok1StageBytes / (D * 2)));
    tt.unit_prefix[0] = 0;
    tt.unit_prefix1[0] = 0;
    for (int i = 0; i < nb; ++i) {
      const int b = c0 + i;
      const int N = cu_tokens[b + 1] - cu_tokens[b];
      tt.tok0[i] = cu_tokens[b];
      tt.n[i] = at.n[i] = N;
      double kt = std::floor(static_cast<double>(p.tail_frac) * N + 0.5);
      if (kt < 1) kt = 1;
      if (kt > N) kt = N;
      tt.ktail[i] = at.ktail[i] = static_cast<int>(kt);
      tt.unit_prefix[i + 1] = tt.unit_prefix[i] + (N + kTokChunk - 1) / kTokChunk;
      tt.unit_prefix1[i + 1] = tt.unit_prefix1[i] + (N + tt.rows1 - 1) / tt.rows1;
      at.H[i] = H[b];
      at.W[i] = W[b];
      at.patch0[i] = cu_tokens[b];
    }
    const int units = tt.unit_prefix[nb];
    const int units1 = tt.unit_prefix1[nb];
    const size_t smem1 = 2 * static_cast<size_t>(tt.rows1) * D * 2;
    PACE_CHECK(tok_pass1_attr());
    apc_tok_pass1<<<tok_pass1_grid(units1), kApcThreads, smem1, stream>>>(T32, tt, units1, inv, sums);
    PACE_CHECK(check_launch());
    apc_tok_pass2<<<units, kApcThreads, 0, stream>>>(T32, tt, inv, sums, d_out, stats, work);
    PACE_CHECK(check_launch());
    TailParams tp{p.alpha, p.gamma, p.r_min, p.r_max, p.align};
    launch_tail_scan(at, d_out, tp, stats, work, stream);
    PACE_CHECK(check_launch());
  }
  return PACE_OK;
}

// ------------------------------------------------------------------------------------------------
// pixel-statistic previews
// ------------------------------------------------------------------------------------------------
namespace pace {
namespace {

// Strip table of images c0 .. c0 + nb - 1 (as the density passes build it); false if an image
// is not laid out for 4-byte copies (then the narrow loader is used).
bool fill_strip_table(ApcTable& t, int c0, int nb, const int64_t* img_off, const int32_t* H, const int32_t* W,
                      float tail_frac, int& patch0) {
  bool wide = true;
  t = ApcTable{};
  t.nb = nb;
  t.b_base = c0;
  t.unit_prefix[0] = 0;
  for (int i = 0; i < nb; ++i) {
    const int b = c0 + i;
    t.off[i] = img_off[b];
    t.H[i] = H[b];
    t.W[i] = W[b];
    t.gw[i] = W[b] / kPatch;
    t.chunks[i] = (t.gw[i] + kStrip - 1) / kStrip;
    t.patch0[i] = patch0;
    const int N = (H[b] / kPatch) * t.gw[i];
    t.n[i] = N;
    double kt = std::floor(static_cast<double>(tail_frac) * N + 0.5);
    if (kt < 1) kt = 1;
    if (kt > N) kt = N;
    t.ktail[i] = static_cast<int>(kt);
    patch0 += N;
    t.unit_prefix[i + 1] = t.unit_prefix[i] + (H[b] / kPatch) * t.chunks[i];
    if ((static_cast<int64_t>(W[b]) * 3) % 4 != 0 || (t.gw[i] % 2) != 0 || (img_off[b] % 4) != 0) wide = false;
  }
  return wide;
}

pace_status_t launch_pix_features(const uint8_t* img, const ApcTable& t, bool wide, int feature, float* tokens,
                                  cudaStream_t stream) {
  const int units = t.unit_prefix[t.nb];
  if (wide) apc_pix_features<true><<<strip_grid(units), kApcThreads, 0, stream>>>(img, t, units, feature, tokens);
  else apc_pix_features<false><<<strip_grid(units), kApcThreads, 0, stream>>>(img, t, units, feature, tokens);
  return check_launch();
}

int64_t total_patches(int B, const int32_t* H, const int32_t* W) {
  int64_t n = 0;
  for (int b = 0; b < B; ++b) n += static_cast<int64_t>(H[b] / kPatch) * (W[b] / kPatch);
  return n;
}

}  // namespace
}  // namespace pace

extern "C" pace_status_t pace_apc_pixel_features(const uint8_t* img, const int64_t* img_off, const int32_t* H,
                                                 const int32_t* W, int B, int feature, float* tokens,
                                                 pace_stream_t stream) {
  PACE_CHECK(check_images(img, img_off, H, W, B));
  if (B == 0) return PACE_OK;
  if (feature < kFeatRgb || feature > kFeatLaplacian || tokens == nullptr || reinterpret_cast<uintptr_t>(tokens) % 16)
    return PACE_ERR_INVALID_ARG;
  PACE_CHECK(check_device());
  int patch0 = 0;
  for (int c0 = 0; c0 < B; c0 += kApcMaxB) {
    ApcTable t;
    const bool wide = fill_strip_table(t, c0, std::min(kApcMaxB, B - c0), img_off, H, W, 0.1f, patch0);
    PACE_CHECK(launch_pix_features(img, t, wide, feature, tokens, stream));
  }
  return PACE_OK;
}

extern "C" size_t pace_apc_density_pixel_workspace_size(int B, const int32_t* H, const int32_t* W) {
  if (B <= 0 || H == nullptr || W == nullptr) return 0;
  for (int b = 0; b < B; ++b)
    if (H[b] < kPatch || W[b] < kPatch) return 0;
  return align_up(static_cast<size_t>(total_patches(B, H, W)) * kPixDim * sizeof(float), 256) +
         align_up(static_cast<size_t>(B) * kPixDim * sizeof(unsigned long long), 256) +
         static_cast<size_t>(B) * sizeof(TailWork);
}

extern "C" pace_status_t pace_apc_density_pixel(const uint8_t* img, const int64_t* img_off, const int32_t* H,
                                                const int32_t* W, int B, int feature, const pace_apc_params* params,
                                                float* d_out, pace_apc_stats* stats, void* ws, size_t ws_bytes,
                                                pace_stream_t stream) {
  PACE_CHECK(check_images(img, img_off, H, W, B));
  if (B == 0) return PACE_OK;
  if (feature < kFeatRgb || feature > kFeatLaplacian || d_out == nullptr || stats == nullptr)
    return PACE_ERR_INVALID_ARG;
  pace_apc_params p;
  if (params) p = *params; else pace_apc_params_default(&p);
  if (!(p.tail_frac > 0.f && p.tail_frac <= 1.f) || !(p.gamma > 0.f) || !(p.alpha >= 0.f && p.alpha <= 1.f) ||
      !(p.r_min <= p.r_max) || p.align < 1)
    return PACE_ERR_INVALID_ARG;
  const size_t tok_bytes = align_up(static_cast<size_t>(total_patches(B, H, W)) * kPixDim * sizeof(float), 256);
  if (ws == nullptr || ws_bytes < pace_apc_density_pixel_workspace_size(B, H, W) ||
      reinterpret_cast<uintptr_t>(ws) % 16)
    return PACE_ERR_WORKSPACE;
  PACE_CHECK(check_device());
  auto* tokens = static_cast<float*>(ws);
  auto* sums = reinterpret_cast<unsigned long long*>(static_cast<uint8_t*>(ws) + tok_bytes);
  const size_t sums_bytes = align_up(static_cast<size_t>(B) * kPixDim * sizeof(unsigned long long), 256);
  auto* work = reinterpret_cast<TailWork*>(reinterpret_cast<uint8_t*>(sums) + sums_bytes);
  PACE_CUDA(cudaMemsetAsync(sums, 0, sums_bytes + static_cast<size_t>(B) * sizeof(TailWork), stream));   // sums, tail scratch
  int patch0 = 0;
  for (int c0 = 0; c0 < B; c0 += kApcMaxB) {
    const int nb = std::min(kApcMaxB, B - c0);
    ApcTable at;
    const bool wide = fill_strip_table(at, c0, nb, img_off, H, W, p.tail_frac, patch0);
    PACE_CHECK(launch_pix_features(img, at, wide, feature, tokens, stream));
    PixTable pt{};
    pt.nb = nb;
    pt.b_base = c0;
    pt.unit_prefix[0] = 0;
    for (int i = 0; i < nb; ++i) {
      pt.tok0[i] = at.patch0[i];
      pt.n[i] = at.n[i];
      pt.ktail[i] = at.ktail[i];
      pt.unit_prefix[i + 1] = pt.unit_prefix[i] + (at.n[i] + kApcThreads - 1) / kApcThreads;
    }
    const int units = pt.unit_prefix[nb];
    apc_pix_pass1<<<units, kApcThreads, 0, stream>>>(pt, tokens, sums);
    PACE_CHECK(check_launch());
    apc_pix_pass2<<<units, kApcThreads, 0, stream>>>(pt, tokens, sums, d_out, stats, work);
    PACE_CHECK(check_launch());
    TailParams tp{p.alpha, p.gamma, p.r_min, p.r_max, p.align};
    launch_tail_scan(at, d_out, tp, stats, work, stream);
    PACE_CHECK(check_launch());
  }
  return PACE_OK;
}
