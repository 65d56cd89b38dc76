// Extract: ViT received attention (S_vis) and LLM text->visual attention (S_llm), Sec. 3.3.
//
// Both maps are column sums of a row-softmax attention matrix, a_j = sum_i P_ij with
// P_ij = exp(s_ij - lse_i), s_ij = scale q_i . k_j.  They are computed flash-style in two
// passes so that the N x N score matrix is never stored:
//
//   pass 1  attn_row_lse   S = Q K^T on tcgen05 and, on the CUDA cores, the base-2 row
//           log-sum-exp L_i = log2 sum_j 2^(c s_ij), c = scale * log2(e).  Each row's shift
//           is fixed at the maximum of its first chunk of scores, so the common path has no
//           running maximum; a CTA whose rows overflowed that shift streams its keys a second
//           time with the exact online maximum.  Optionally split over key ranges (partial
//           (m, l) pairs merged by attn_lse_combine).  The result is stored as a 16-column
//           bf16 "shift row" per query: -L_i / c as hi + mid + lo, then zeros.
//   pass 2  attn_colsum    S^T = K Q^T with one extra K-step that multiplies the keys' ones
//           slice [1, 1, 1, 0, ...] by the queries' shift rows, so the accumulator already
//           holds s_ji - L_i / c.  Every TMEM lane is one key: each epilogue thread owns one key
//           and accumulates 2^(c a_ji) over the whole query stream in registers, with no
//           per-column loads, cross-thread reduction or atomics.
//   reduce  attn_reduce    sums the per-head (or per KV-head) partial maps and pools the
//           `merge` consecutive patches of each merged token.
//
// Every CTA works alone (one-SM MMA, local barriers only): it holds 128 resident rows and
// streams whole 256-row tiles, one 128 x 256 x 16 tcgen05.mma per K-step into a 128 x 256
// fp32 TMEM accumulator.  A work item is 256 resident rows, i.e. two CTAs.
//
// CTA layout (576 threads, one CTA per SM):
//   warp 0       TMA producer (one lane): the resident tile once, then every streamed tile
//                through a ring of stages
//   warp 1       TMEM allocation (512 columns = two 128 x 256 accumulators) and MMA issue
//                (one lane)
//   warps 2-17   four epilogue warpgroups; warpgroup e = 2p + hh reads columns hh*128.. of
//                accumulator p (stream tiles j with j % 2 == p); results of the four are
//                merged at the end
// Operands are K-major bf16 tiles staged by TMA: 64-column blocks with the 128-byte swizzle,
// and 16-column slices with the 32-byte swizzle (the tail of a head dimension that is not a
// multiple of 64, 80 = 64 + 16, and the shift slices of pass 2).  MMA descriptors are built
// once and advanced by immediates.
//
// GQA: query head h reads KV head h / G.  The ViT case is G = 1.
#include <algorithm>
#include <atomic>
#include <cmath>
#include <mutex>
#include <vector>

#include <cuda_bf16.h>
#include <cudaTypedefs.h>

#include "pace_common.cuh"
#include "pace_ptx.cuh"

namespace pace {
namespace {

using namespace ptx;

constexpr int kTile = 128;                // resident rows held by one CTA
constexpr int kPair = 256;                // rows of one work item (two CTAs, 128 rows each)
constexpr int kStream = 256;              // streamed rows per tile
constexpr int kEpiWarps = 16;
constexpr int kThreads = 64 + 32 * kEpiWarps;   // 576
constexpr int kAttnMaxB = 64;
constexpr uint32_t kTmemCols = 512;
constexpr float kShiftMargin = 90.f;      // pass 1: fixed shift = first chunk maximum + this (base 2)
constexpr int kNoMask = 1 << 29;          // diag of a non-causal image: every key is seen

// An operand tile of ROWS rows and head dimension D is stored as NB blocks of 64 columns
// (ROWS x 128 bytes, 128-byte swizzle) followed by R slices of 16 columns (ROWS x 32 bytes,
// 32-byte swizzle); D = 80: one block + one slice; D = 128: two blocks; D = 64: one block.
template <int D, int ROWS>
struct TileFmt {
  static constexpr int NB = D / 64;
  static constexpr int R = (D % 64) / 16;
  static constexpr int BLOCK = ROWS * 128;
  static constexpr int SLICE = ROWS * 32;
  static constexpr int BYTES = NB * BLOCK + R * SLICE;
  static_assert(D % 16 == 0 && BYTES % 1024 == 0 && ROWS % kTile == 0, "tile format");
};

template <int D>
struct Cfg {
  using A = TileFmt<D, kTile>;      // resident tile
  using B = TileFmt<D, kStream>;    // streamed tile
  static constexpr int STAGES = (D == 128) ? 2 : (D == 80) ? 4 : 5;
  static constexpr uint32_t IDESC = idesc_bf16_f32(kTile, kStream);
};

// Extra K slice of pass 2 (16 bf16 columns, 32 bytes per row).  Query row i carries the
// negated base-2 LSE divided by c, split into three bf16 terms hi + mid + lo (the rest of the
// 32 bytes zero); key rows carry [1, 1, 1, 0, ...].  One more K-step of the MMA then
// accumulates s_ji - L_i / c, so the epilogue needs no per-column shift.
constexpr int kShiftCols = 16;
constexpr uint16_t kBf16One = 0x3F80;
constexpr uint16_t kBf16NegHuge = 0xF180;   // -2^100: zero weight for padded query rows

struct alignas(256) OnesSlice {
  uint16_t v[kTile * kShiftCols];
  constexpr OnesSlice() : v() {
    for (int i = 0; i < kTile * kShiftCols; ++i) v[i] = (i % kShiftCols) < 3 ? kBf16One : 0;
  }
};
__device__ const OnesSlice g_ones_slice{};

// Writes the 32-byte shift row of one query: v = -L / c (or -inf for a padded row).
__device__ __forceinline__ void store_shift_row(uint16_t* row, float v) {
  uint32_t w0, w1;
  if (v > -INFINITY) {
    const __nv_bfloat16 hi = __float2bfloat16_rn(v);
    const float r1 = v - __bfloat162float(hi);
    const __nv_bfloat16 mid = __float2bfloat16_rn(r1);
    const __nv_bfloat16 lo = __float2bfloat16_rn(r1 - __bfloat162float(mid));
    w0 = static_cast<uint32_t>(__bfloat16_as_ushort(hi)) | (static_cast<uint32_t>(__bfloat16_as_ushort(mid)) << 16);
    w1 = static_cast<uint32_t>(__bfloat16_as_ushort(lo));
  } else {
    w0 = kBf16NegHuge;
    w1 = 0u;
  }
  uint4* p = reinterpret_cast<uint4*>(row);
  p[0] = make_uint4(w0, w1, 0u, 0u);
  p[1] = make_uint4(0u, 0u, 0u, 0u);
}

struct AttnTable {
  int q0[kAttnMaxB], nq[kAttnMaxB];   // query rows of image b
  int k0[kAttnMaxB], nk[kAttnMaxB];   // key rows of image b
  int diag[kAttnMaxB];                // causal mask: local key k is seen by local query i iff k <= i + diag
  int out0[kAttnMaxB];                // first part-map row of image b (pass 2)
  int lpad[kAttnMaxB];                // first padded L row of image b (multiple of 256)
  int pair_lo[kAttnMaxB], pair_n[kAttnMaxB];   // pass 1: the query pairs this launch takes
  int item_prefix[kAttnMaxB + 1];
  int nb;
  int H;        // query heads
  int G;        // query heads per KV head
  int splits;   // key splits of pass 1
  int prows;    // padded L rows per head
  int ktot;     // total key rows (part map row count)
};

__device__ __forceinline__ int find_image(const AttnTable& t, int item) {
  int b = 0;
  while (b + 1 < t.nb && t.item_prefix[b + 1] <= item) ++b;
  return b;
}

struct SmemCtl {
  uint64_t bars[40];
  uint32_t tmem_base;
  int abort;
  int redo;                  // pass 1: some row overflowed the fixed-shift round
  float xchg[3][2][kTile];   // hand-over between the four epilogue warpgroups
};

__device__ __forceinline__ void set_abort(SmemCtl* ctl, int* status, int kernel) {
  *reinterpret_cast<volatile int*>(&ctl->abort) = 1;
  record_error(status, PACE_ERR_TIMEOUT, kernel);
}
__device__ __forceinline__ bool aborted(const SmemCtl* ctl) {
  return *reinterpret_cast<const volatile int*>(&ctl->abort) != 0;
}

// TMA of ROWS rows (y .. y + ROWS - 1, columns x0 .. x0 + D) into dst in 128-row boxes;
// completion is counted on the barrier `bar`.
template <int D, int ROWS>
__device__ __forceinline__ void load_tile(uint8_t* dst, const CUtensorMap* m128, const CUtensorMap* m32, int x0,
                                          int y, uint32_t bar) {
  using F = TileFmt<D, ROWS>;
#pragma unroll
  for (int q = 0; q < ROWS / kTile; ++q) {
#pragma unroll
    for (int i = 0; i < F::NB; ++i)
      tma_load_2d(smem_u32(dst + i * F::BLOCK + q * kTile * 128), m128, x0 + 64 * i, y + q * kTile, bar);
#pragma unroll
    for (int r = 0; r < F::R; ++r)
      tma_load_2d(smem_u32(dst + F::NB * F::BLOCK + r * F::SLICE + q * kTile * 32), m32, x0 + 64 * F::NB + 16 * r,
                  y + q * kTile, bar);
  }
}

// Shared-memory descriptors of a tile: [0] for its 128-byte-swizzled blocks, [1] for its
// 32-byte-swizzled slices.  Adding (bytes >> 4) moves the start address.
template <int D, int ROWS>
__device__ __forceinline__ void tile_desc(const uint8_t* tile, uint64_t& d128, uint64_t& d32) {
  d128 = smem_desc_kmajor_sw128(smem_u32(tile));
  d32 = smem_desc_kmajor_sw32(smem_u32(tile + TileFmt<D, ROWS>::NB * TileFmt<D, ROWS>::BLOCK));
}

// MMA D[tmem] = A B^T (128 x 256) over the whole head dimension: 4 K-steps per 128-byte
// block, 1 per 32-byte slice.
template <int D>
__device__ __forceinline__ void mma_tile(uint32_t d, uint64_t a128, uint64_t a32, uint64_t b128, uint64_t b32) {
  using FA = typename Cfg<D>::A;
  using FB = typename Cfg<D>::B;
#pragma unroll
  for (int i = 0; i < FA::NB; ++i)
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const uint64_t oa = static_cast<uint64_t>(i * (FA::BLOCK >> 4) + k * 2);
      const uint64_t ob = static_cast<uint64_t>(i * (FB::BLOCK >> 4) + k * 2);
      mma_bf16_ss(d, a128 + oa, b128 + ob, Cfg<D>::IDESC, (i | k) != 0);
    }
#pragma unroll
  for (int r = 0; r < FA::R; ++r)
    mma_bf16_ss(d, a32 + static_cast<uint64_t>(r * (FA::SLICE >> 4)), b32 + static_cast<uint64_t>(r * (FB::SLICE >> 4)),
                Cfg<D>::IDESC, (FA::NB | r) != 0);
}

// 64 TMEM columns of this warp's 32 lanes -> v[0..63] (fp32 bit patterns), ready to use.
__device__ __forceinline__ void load_cols64(uint32_t taddr, uint32_t (&v)[64]) {
  tmem_ld_32x32b_x64(taddr, v);
  tmem_wait_ld();
  reg_fence64(v);
}

// Online (max, sum of exp2) update of one row with 64 new scores (raw dot products);
// entries at and beyond `valid` are ignored.
__device__ __forceinline__ void lse_update64(const uint32_t (&v)[64], int valid, float c, float& m_run,
                                             float& l_run) {
  if (valid <= 0) return;
  float s[64];
#pragma unroll
  for (int e = 0; e < 64; ++e) s[e] = __uint_as_float(v[e]);
  if (valid < 64) {
#pragma unroll
    for (int e = 0; e < 64; ++e)
      if (e >= valid) s[e] = -INFINITY;
  }
  float mx0 = -INFINITY, mx1 = -INFINITY, mx2 = -INFINITY, mx3 = -INFINITY;
#pragma unroll
  for (int e = 0; e < 64; e += 8) {
    mx0 = max3(mx0, s[e + 0], s[e + 1]);
    mx1 = max3(mx1, s[e + 2], s[e + 3]);
    mx2 = max3(mx2, s[e + 4], s[e + 5]);
    mx3 = max3(mx3, s[e + 6], s[e + 7]);
  }
  const float mt = fmaxf(fmaxf(mx0, mx1), fmaxf(mx2, mx3)) * c;
  if (mt > m_run) {
    l_run *= ex2_approx(m_run - mt);
    m_run = mt;
  }
  const float2 cc = make_float2(c, c);
  const float2 nm = make_float2(-m_run, -m_run);
  float2 a0 = make_float2(0.f, 0.f), a1 = a0;
#pragma unroll
  for (int e = 0; e < 64; e += 4) {
    const float2 x0 = ffma2(make_float2(s[e], s[e + 1]), cc, nm);
    const float2 x1 = ffma2(make_float2(s[e + 2], s[e + 3]), cc, nm);
    a0 = fadd2(a0, make_float2(ex2_approx(x0.x), ex2_approx(x0.y)));
    a1 = fadd2(a1, make_float2(ex2_approx(x1.x), ex2_approx(x1.y)));
  }
  const float2 a = fadd2(a0, a1);
  l_run += a.x + a.y;
}

// Fixed-shift row update with 64 new scores: the shift m is the base-2 maximum of the row's
// first chunk plus a margin of kShiftMargin, and then never moves, so there is no maximum in the
// common path.  Every term 2^(c s - m) above 2^-126 is computed to full relative precision, and
// the largest term of the row is >= 2^-kShiftMargin, so the terms flushed to zero weigh at most
// N 2^(kShiftMargin - 126) of the sum (2^-16 for N = 2^20).  The only failure is overflow (a
// score more than about 127 + kShiftMargin - log2(N) above the first chunk's maximum), which
// leaves l = inf or NaN and is caught by the caller.
template <bool FIRST>
__device__ __forceinline__ void lse_fixed64(const uint32_t (&v)[64], int valid, float c, float& m_run,
                                            float& l_run) {
  float s[64];
#pragma unroll
  for (int e = 0; e < 64; ++e) s[e] = __uint_as_float(v[e]);
  if (valid < 64) {
#pragma unroll
    for (int e = 0; e < 64; ++e)
      if (e >= valid) s[e] = -INFINITY;
  }
  if (FIRST) {
    float mx0 = -INFINITY, mx1 = -INFINITY, mx2 = -INFINITY, mx3 = -INFINITY;
#pragma unroll
    for (int e = 0; e < 64; e += 8) {
      mx0 = max3(mx0, s[e + 0], s[e + 1]);
      mx1 = max3(mx1, s[e + 2], s[e + 3]);
      mx2 = max3(mx2, s[e + 4], s[e + 5]);
      mx3 = max3(mx3, s[e + 6], s[e + 7]);
    }
    m_run = fmaf(fmaxf(fmaxf(mx0, mx1), fmaxf(mx2, mx3)), c, kShiftMargin);
  }
  const float2 cc = make_float2(c, c);
  const float2 nm = make_float2(-m_run, -m_run);
  float2 a0 = make_float2(0.f, 0.f), a1 = a0;
#pragma unroll
  for (int e = 0; e < 64; e += 4) {
    const float2 x0 = ffma2(make_float2(s[e], s[e + 1]), cc, nm);
    const float2 x1 = ffma2(make_float2(s[e + 2], s[e + 3]), cc, nm);
    a0 = fadd2(a0, make_float2(ex2_approx(x0.x), ex2_approx(x0.y)));
    a1 = fadd2(a1, make_float2(ex2_approx(x1.x), ex2_approx(x1.y)));
  }
  const float2 a = fadd2(a0, a1);
  l_run += a.x + a.y;
}

// Fixed-shift update of a full chunk once the shift is set (no masking, no maximum); the sum
// stays in two packed partial sums that the caller folds into l once, after its last chunk.
__device__ __forceinline__ void lse_fixed_full(const uint32_t (&v)[64], float c, float m_run, float2& a0,
                                               float2& a1) {
  const float2 cc = make_float2(c, c);
  const float2 nm = make_float2(-m_run, -m_run);
#pragma unroll
  for (int e = 0; e < 64; e += 4) {
    const float2 x0 = ffma2(make_float2(__uint_as_float(v[e]), __uint_as_float(v[e + 1])), cc, nm);
    const float2 x1 = ffma2(make_float2(__uint_as_float(v[e + 2]), __uint_as_float(v[e + 3])), cc, nm);
    a0 = fadd2(a0, make_float2(ex2_approx(x0.x), ex2_approx(x0.y)));
    a1 = fadd2(a1, make_float2(ex2_approx(x1.x), ex2_approx(x1.y)));
  }
}

// Dispatch of the fixed-shift update: the first chunk with keys sets the shift.  The two
// cases are separate instantiations so that the maximum is not issued (predicated off) for
// every chunk.
__device__ __forceinline__ void lse_fixed(const uint32_t (&v)[64], int valid, float c, float& m_run, float& l_run) {
  if (valid <= 0) return;
  if (m_run == -INFINITY) lse_fixed64<true>(v, valid, c, m_run, l_run);
  else lse_fixed64<false>(v, valid, c, m_run, l_run);
}

// (a0, a1) += sum_e 2^(c a_e) over 64 columns, a_e = s_e - L / c straight from the MMA, as two
// packed partial sums carried across chunks.
__device__ __forceinline__ void colsum64(const uint32_t (&v)[64], float c, float2& a0, float2& a1) {
  const float2 cc = make_float2(c, c);
  const float2 zero = make_float2(0.f, 0.f);
#pragma unroll
  for (int e = 0; e < 64; e += 4) {
    const float2 x0 = ffma2(make_float2(__uint_as_float(v[e]), __uint_as_float(v[e + 1])), cc, zero);
    const float2 x1 = ffma2(make_float2(__uint_as_float(v[e + 2]), __uint_as_float(v[e + 3])), cc, zero);
    a0 = fadd2(a0, make_float2(ex2_approx(x0.x), ex2_approx(x0.y)));
    a1 = fadd2(a1, make_float2(ex2_approx(x1.x), ex2_approx(x1.y)));
  }
}

// colsum64 over the columns e >= lo only (the causal mask of pass 2).
__device__ __forceinline__ void colsum64_from(const uint32_t (&v)[64], int lo, float c, float2& a0, float2& a1) {
  uint32_t w[64];
#pragma unroll
  for (int e = 0; e < 64; ++e) w[e] = e < lo ? 0xFF800000u : v[e];   // -inf: 2^(c * -inf) = 0
  colsum64(w, c, a0, a1);
}

// Overwrites query rows rows .. kStream - 1 of a staged pass-2 tile with zeros: the 128-byte rows
// of its 64-column blocks and the 32-byte rows of its 16-column slices (a swizzle only moves
// 16-byte pieces within their own row), by the 32 lanes of a warp.  The shift slice keeps the
// padded rows' -2^100, so these rows add exactly 0 to every key's sum.
template <int D>
__device__ __forceinline__ void zero_stage_rows(uint8_t* st, int rows) {
  using F = TileFmt<D, kStream>;
  constexpr int PIECES = F::NB * 8 + F::R * 2;   // 16-byte pieces per row
  const int lane = threadIdx.x & 31;
  const uint4 z = make_uint4(0u, 0u, 0u, 0u);
  for (int i = lane; i < (kStream - rows) * PIECES; i += 32) {
    const int row = rows + i / PIECES, pc = i % PIECES;
    uint8_t* dst = pc < F::NB * 8 ? st + (pc >> 3) * F::BLOCK + row * 128 + (pc & 7) * 16
                                  : st + F::NB * F::BLOCK + ((pc - F::NB * 8) >> 1) * F::SLICE + row * 32 +
                                        ((pc - F::NB * 8) & 1) * 16;
    *reinterpret_cast<uint4*>(dst) = z;
  }
}

// Brings the CTA to a quiet point: waits for its MMAs (phase `done_phase` of b_done) and lets
// in-flight copies land after an abort; TMEM stays allocated.
__device__ __forceinline__ void cta_quiesce(SmemCtl* ctl, uint32_t b_done, uint32_t done_phase, int* status,
                                            int kernel) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  tc_fence_before_sync();
  __syncthreads();
  if (warp == 1 && lane == 0) {
    if (!mbar_wait(b_done, done_phase, kWaitLimitNs)) record_error(status, PACE_ERR_TIMEOUT, kernel);
  }
  if (threadIdx.x == 0 && aborted(ctl)) {   // give outstanding TMA copies time to land
    const uint64_t t0 = globaltimer_ns();
    while (globaltimer_ns() - t0 < 100000ull) {
    }
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
}

// Releases the CTA's TMEM (after cta_quiesce).
__device__ __forceinline__ void cta_release_tmem(uint32_t tmem) {
  if ((threadIdx.x >> 5) == 1) tmem_dealloc(tmem, kTmemCols);
}

// ------------------------------------------------------------------------------------------------
// pass 1: row log-sum-exp
// ------------------------------------------------------------------------------------------------
template <int D, bool CAUSAL>
__global__ void __launch_bounds__(kThreads, 1) attn_row_lse(const __grid_constant__ CUtensorMap tmq,
                                                            const __grid_constant__ CUtensorMap tmq32,
                                                            const __grid_constant__ CUtensorMap tmk,
                                                            const __grid_constant__ CUtensorMap tmk32,
                                                            const __grid_constant__ AttnTable t, float c,
                                                            uint16_t* __restrict__ shift_out,
                                                            float2* __restrict__ ml_out, int* status) {
  using C = Cfg<D>;
  constexpr int ST = C::STAGES;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = smem;                                // this CTA's resident query tile
  uint8_t* sK = sQ + C::A::BYTES;                    // ST stages of a key tile
  SmemCtl* ctl = reinterpret_cast<SmemCtl*>(sK + ST * C::B::BYTES);
  const uint32_t b_qfull = smem_u32(&ctl->bars[0]);     // query tile landed
  const uint32_t b_done = smem_u32(&ctl->bars[1]);      // all MMAs of a round finished
  auto b_kfull = [&](int s) { return smem_u32(&ctl->bars[2 + s]); };
  auto b_kempty = [&](int s) { return smem_u32(&ctl->bars[2 + ST + s]); };
  auto b_sfull = [&](int p) { return smem_u32(&ctl->bars[2 + 2 * ST + p]); };
  auto b_sfree = [&](int p) { return smem_u32(&ctl->bars[4 + 2 * ST + p]); };

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = blockIdx.x & 1u;       // which 128-row half of the item
  const int item = blockIdx.x >> 1;
  const int b = find_image(t, item);
  int r = item - t.item_prefix[b];
  const int split = r % t.splits;
  r /= t.splits;
  const int npair = t.pair_n[b];
  const int diag = t.diag[b];
  // causal images: the last query rows see the most keys, so they are scheduled first
  const int pair = t.pair_lo[b] + (CAUSAL ? npair - 1 - r % npair : r % npair);
  const int h = r / npair;
  const int g = h / t.G;
  const int qrow0 = pair * kPair + kTile * static_cast<int>(rank);     // this CTA's first local query row
  const int nkt_all = (t.nk[b] + kStream - 1) / kStream;
  const int kt0 = static_cast<int>((static_cast<int64_t>(split) * nkt_all) / t.splits);
  // causal: key tiles past the one holding key qrow0 + 127 + diag are masked for every row (diag >= 0)
  const int kt1_all = static_cast<int>((static_cast<int64_t>(split + 1) * nkt_all) / t.splits);
  const int kt1 = CAUSAL ? min(kt1_all, (diag + qrow0 + kTile - 1) / kStream + 1) : kt1_all;
  const int nj = max(kt1 - kt0, 0);
  const int pre = min(nj, ST);   // key stages issued in the prologue (round 0, first use of each stage)

  if (threadIdx.x == 0) {
    mbar_init(b_qfull, 1);
    mbar_init(b_done, 1);
    for (int s = 0; s < ST; ++s) {
      mbar_init(b_kfull(s), 1);
      mbar_init(b_kempty(s), 1);
    }
    for (int p = 0; p < 2; ++p) {
      mbar_init(b_sfull(p), 1);
      mbar_init(b_sfree(p), 8);   // the eight warps of warpgroup pair p
    }
    ctl->abort = 0;
    ctl->redo = 0;
    fence_mbar_init();
    // The query tile and the first key stages are requested before the CTA-wide barrier below,
    // so their latency overlaps the TMEM allocation (the barriers are initialised and fenced
    // by this thread; nobody else touches them before that barrier).
    prefetch_tensormap(&tmq);
    prefetch_tensormap(&tmk);
    if (C::A::R > 0) {
      prefetch_tensormap(&tmq32);
      prefetch_tensormap(&tmk32);
    }
    mbar_arrive_expect_tx(b_qfull, C::A::BYTES);
    load_tile<D, kTile>(sQ, &tmq, &tmq32, h * D, t.q0[b] + qrow0, b_qfull);
    for (int j = 0; j < pre; ++j) {
      mbar_arrive_expect_tx(b_kfull(j), C::B::BYTES);
      load_tile<D, kStream>(sK + j * C::B::BYTES, &tmk, &tmk32, g * D, t.k0[b] + (kt0 + j) * kStream, b_kfull(j));
    }
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&ctl->tmem_base), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem = ctl->tmem_base;

  // Round 0 uses the fixed-shift update; if any row of the CTA overflowed it, round 1
  // streams the keys again with the exact online-maximum update.  Stream tiles are counted
  // across rounds (it = round * nj + j), so every barrier keeps its phase sequence.
  const int e = (warp - 2) >> 2;            // epilogue warpgroup (warps 2..17)
  const int p = e >> 1, hh = e & 1;
  const int quad = warp & 3;
  const int rr = quad * 32 + lane;
  auto run_round = [&](int round) {
    const int it0 = round * nj;
    if (warp == 0) {
      if (lane == 0) {
        for (int j = round == 0 ? pre : 0; j < nj; ++j) {
          const int it = it0 + j;
          const int s = it % ST, u = it / ST;
          if (u > 0 && !mbar_wait(b_kempty(s), (u - 1) & 1, kWaitLimitNs)) {
            set_abort(ctl, status, K_ATTN_ROW_LSE);
            break;
          }
          if (aborted(ctl)) break;
          mbar_arrive_expect_tx(b_kfull(s), C::B::BYTES);
          load_tile<D, kStream>(sK + s * C::B::BYTES, &tmk, &tmk32, g * D, t.k0[b] + (kt0 + j) * kStream, b_kfull(s));
        }
      }
    } else if (warp == 1) {
      if (lane == 0) {
        uint64_t aq128, aq32, bk128, bk32;
        tile_desc<D, kTile>(sQ, aq128, aq32);
        tile_desc<D, kStream>(sK, bk128, bk32);
        const bool ok = mbar_wait(b_qfull, 0, kWaitLimitNs);
        if (!ok) set_abort(ctl, status, K_ATTN_ROW_LSE);
        for (int j = 0; ok && j < nj; ++j) {
          const int it = it0 + j;
          const int s = it % ST, u = it / ST;
          const int pa = it & 1, v = it >> 1;
          if (!mbar_wait(b_kfull(s), u & 1, kWaitLimitNs) ||
              (v > 0 && !mbar_wait(b_sfree(pa), (v - 1) & 1, kWaitLimitNs)) || aborted(ctl)) {
            set_abort(ctl, status, K_ATTN_ROW_LSE);
            break;
          }
          tc_fence_after_sync();
          const uint64_t so = static_cast<uint64_t>(s * (C::B::BYTES >> 4));
          mma_tile<D>(tmem + pa * 256, aq128, aq32, bk128 + so, bk32 + so);
          mma_commit(b_sfull(pa));
          mma_commit(b_kempty(s));
        }
        mma_commit(b_done);
      }
      __syncwarp();
    } else {
      // epilogue warpgroup e = 2p + hh: accumulator p (stream tiles it % 2 == p), columns hh * 128 ..
      float m_run = -INFINITY, l_run = 0.f;
      float2 la0 = make_float2(0.f, 0.f), la1 = la0;   // the full chunks' sums (round 0 only)
      const uint32_t tbuf = tmem + (static_cast<uint32_t>(quad * 32) << 16) + p * 256 + hh * 128;
      for (int j = (p - it0) & 1; j < nj; j += 2) {
        const int it = it0 + j;
        const int v = it >> 1;
        const bool ok = __all_sync(0xffffffffu, mbar_wait(b_sfull(p), v & 1, kWaitLimitNs));
        // warp-uniform exit: the tcgen05.ld below is warp-wide.  The epilogue does not poll the
        // abort flag per tile: an abort elsewhere reaches it through its own bounded wait.
        if (!ok) {
          set_abort(ctl, status, K_ATTN_ROW_LSE);
          break;
        }
        tc_fence_after_sync();
        // keys of these columns that the row sees: inside the image and, if causal, k <= row + diag
        const int cs = (kt0 + j) * kStream + hh * 128;
        const int valid = CAUSAL ? min(t.nk[b] - cs, diag + qrow0 + rr - cs + 1) : t.nk[b] - cs;
        uint32_t sv[64];
        load_cols64(tbuf, sv);
        // Warp-uniform by construction (both branches hold warp-wide TMEM loads): with a causal
        // mask the lanes vote; without one, valid is the same for every lane and the shift is set
        // once this pair's first tile is done (tested on j, not on m_run, which a NaN in a row's
        // scores would make differ between lanes).
        const bool lean = CAUSAL ? __all_sync(0xffffffffu, round == 0 && valid >= 128 && m_run > -INFINITY)
                                 : (round == 0 && valid >= 128 && j != ((p - it0) & 1));
        if (lean) {   // the common tile: both chunks full, shift already fixed
          lse_fixed_full(sv, c, m_run, la0, la1);
          load_cols64(tbuf + 64, sv);
          tc_fence_before_sync();
          __syncwarp();
          if (lane == 0) mbar_arrive(b_sfree(p));
          lse_fixed_full(sv, c, m_run, la0, la1);
          continue;
        }
        if (round == 0) lse_fixed(sv, valid, c, m_run, l_run);
        else lse_update64(sv, valid, c, m_run, l_run);
        load_cols64(tbuf + 64, sv);
        tc_fence_before_sync();
        __syncwarp();
        if (lane == 0) mbar_arrive(b_sfree(p));
        if (round == 0) lse_fixed(sv, valid - 64, c, m_run, l_run);
        else if (valid > 64) lse_update64(sv, valid - 64, c, m_run, l_run);
      }
      {
        const float2 a = fadd2(la0, la1);
        l_run += a.x + a.y;
      }
      // inf or NaN in a row of the image: it needs the exact round (rows past the image are
      // ignored, so whatever their Q rows hold cannot change the valid rows' results)
      if (!(l_run < INFINITY) && qrow0 + rr < t.nq[b]) ctl->redo = 1;
      // merge the four warpgroups' (m, l) of each row
      if (e > 0) {
        ctl->xchg[e - 1][0][rr] = m_run;
        ctl->xchg[e - 1][1][rr] = l_run;
      }
      named_barrier_sync(1, 32 * kEpiWarps);
      if (e == 0) {
        float M = m_run;
#pragma unroll
        for (int i = 0; i < 3; ++i) M = fmaxf(M, ctl->xchg[i][0][rr]);
        float l = l_run > 0.f ? l_run * ex2_approx(m_run - M) : 0.f;
#pragma unroll
        for (int i = 0; i < 3; ++i) {
          const float li = ctl->xchg[i][1][rr];
          if (li > 0.f) l += li * ex2_approx(ctl->xchg[i][0][rr] - M);
        }
        const int row = qrow0 + rr;                       // local query row
        const int64_t prow = static_cast<int64_t>(h) * t.prows + t.lpad[b] + row;
        if (t.splits == 1) {
          store_shift_row(shift_out + prow * kShiftCols, row < t.nq[b] ? -(M + log2f(l)) / c : -INFINITY);
        } else {
          ml_out[static_cast<int64_t>(split) * t.H * t.prows + prow] =
              (row < t.nq[b] && l > 0.f) ? make_float2(M, l) : make_float2(-INFINITY, 0.f);
        }
      }
    }
  };

  run_round(0);
  cta_quiesce(ctl, b_done, 0, status, K_ATTN_ROW_LSE);
  // If a row overflowed the fixed shift, the CTA streams the keys again with the exact update
  // and overwrites its outputs (stream tiles continue at it = nj ..).
  if (ctl->redo != 0 && !aborted(ctl)) {
    __syncthreads();   // every thread has read the flags before round 1 can change them
    run_round(1);
    cta_quiesce(ctl, b_done, 1, status, K_ATTN_ROW_LSE);
  }
  cta_release_tmem(tmem);
}

// Merges per-split (m, l) pairs into the shift row of -L / c, L = m + log2(l); rows past the
// image get the padded-row shift.
__global__ void __launch_bounds__(128) attn_lse_combine(const __grid_constant__ AttnTable t, float c,
                                                        const float2* __restrict__ ml, uint16_t* __restrict__ shift_out) {
  // blockIdx.x = (image, 128-row tile of its padded rows) flattened
  int rem = blockIdx.x;
  const int h = blockIdx.y;
  int b = 0;
  for (; b < t.nb; ++b) {
    const int nt = (t.nq[b] + kPair - 1) / kPair * 2;
    if (rem < nt) break;
    rem -= nt;
  }
  if (b >= t.nb) return;
  const int row = rem * kTile + threadIdx.x;
  const int64_t prow = static_cast<int64_t>(h) * t.prows + t.lpad[b] + row;
  if (row >= t.nq[b]) {
    store_shift_row(shift_out + prow * kShiftCols, -INFINITY);
    return;
  }
  float M = -INFINITY;
  for (int s = 0; s < t.splits; ++s) M = fmaxf(M, ml[static_cast<int64_t>(s) * t.H * t.prows + prow].x);
  float l = 0.f;
  for (int s = 0; s < t.splits; ++s) {
    const float2 p = ml[static_cast<int64_t>(s) * t.H * t.prows + prow];
    if (p.y > 0.f) l += p.y * ex2_approx(p.x - M);
  }
  store_shift_row(shift_out + prow * kShiftCols, -(M + log2f(l)) / c);
}

// ------------------------------------------------------------------------------------------------
// pass 2: column sums of 2^(c s - L)
// ------------------------------------------------------------------------------------------------
template <int D, bool CAUSAL>
__global__ void __launch_bounds__(kThreads, 1) attn_colsum(const __grid_constant__ CUtensorMap tmq,
                                                           const __grid_constant__ CUtensorMap tmq32,
                                                           const __grid_constant__ CUtensorMap tmk,
                                                           const __grid_constant__ CUtensorMap tmk32,
                                                           const __grid_constant__ CUtensorMap tmshift,
                                                           const __grid_constant__ CUtensorMap tmones,
                                                           const __grid_constant__ AttnTable t, float c,
                                                           float* __restrict__ part, int* status) {
  using C = Cfg<D>;
  constexpr int ST = C::STAGES;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;                                 // this CTA's resident key tile
  constexpr int A2 = C::A::BYTES + kTile * kShiftCols * 2;        // key tile + ones slice
  constexpr int B2 = C::B::BYTES + kStream * kShiftCols * 2;      // query tile + shift slice
  uint8_t* sQ = sA + A2;                               // ST stages of a query tile
  SmemCtl* ctl = reinterpret_cast<SmemCtl*>(sQ + ST * B2);
  const uint32_t b_afull = smem_u32(&ctl->bars[0]);
  const uint32_t b_done = smem_u32(&ctl->bars[1]);
  auto b_qfull = [&](int s) { return smem_u32(&ctl->bars[2 + s]); };
  auto b_qempty = [&](int s) { return smem_u32(&ctl->bars[2 + ST + s]); };
  auto b_sfull = [&](int p) { return smem_u32(&ctl->bars[2 + 2 * ST + p]); };
  auto b_sfree = [&](int p) { return smem_u32(&ctl->bars[4 + 2 * ST + p]); };
  // stage s holds an image's ragged last query tile with the rows past the image zeroed: one
  // arrival per ragged use of the stage (the other tiles need only their copy)
  auto b_fixed = [&](int s) { return smem_u32(&ctl->bars[6 + 2 * ST + s]); };

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = blockIdx.x & 1u;       // which 128-row half of the item
  const int item = blockIdx.x >> 1;
  const int b = find_image(t, item);
  const int r = item - t.item_prefix[b];
  const int nkp = (t.nk[b] + kPair - 1) / kPair;
  const int kp = r % nkp;
  const int g = r / nkp;
  const int krow0 = kp * kPair + kTile * static_cast<int>(rank);     // this CTA's first local key row
  const int diag = t.diag[b];
  const int nqt = (t.nq[b] + kStream - 1) / kStream;
  // causal images: query tiles that end before row krow0 - diag see none of this CTA's keys
  const int qt_min = CAUSAL && krow0 > diag ? (krow0 - diag) / kStream : 0;
  const int nspan = max(nqt - qt_min, 0);
  const int nj = t.G * nspan;                                         // stream: (head in group, query tile)
  // query rows of stream tile j that lie inside the image (kStream unless it is the image's last
  // tile and the image ends inside it)
  auto ragged_rows = [&](int j) { return min(kStream, t.nq[b] - (qt_min + j % nspan) * kStream); };
  // the ragged tiles are j = nspan - 1, 2 nspan - 1, .. (when the image ends inside its last query
  // tile); the phase of b_fixed(j % ST) that ragged tile j completes = how many earlier ragged tiles
  // used the same stage
  auto ragged_phase = [&](int j) {
    int k = 0;
    for (int j2 = nspan - 1; j2 < j; j2 += nspan) k += (j2 % ST) == (j % ST);
    return k & 1;
  };

  if (threadIdx.x == 0) {
    mbar_init(b_afull, 1);
    mbar_init(b_done, 1);
    for (int s = 0; s < ST; ++s) {
      mbar_init(b_qfull(s), 1);
      mbar_init(b_qempty(s), 1);
    }
    for (int p = 0; p < 2; ++p) {
      mbar_init(b_sfull(p), 1);
      mbar_init(b_sfree(p), 8);
    }
    for (int s = 0; s < ST; ++s) mbar_init(b_fixed(s), 1);
    ctl->abort = 0;
    fence_mbar_init();
  }
  // stage s of stream item j: query tile (head in group, query tile) plus its shift slice
  auto issue_stage = [&](int j, int s) {
    const int hq = j / nspan, qt = qt_min + j - hq * nspan;
    const int h = g * t.G + hq;
    uint8_t* st = sQ + s * B2;
    mbar_arrive_expect_tx(b_qfull(s), B2);
    load_tile<D, kStream>(st, &tmq, &tmq32, h * D, t.q0[b] + qt * kStream, b_qfull(s));
    const int srow = h * t.prows + t.lpad[b] + qt * kStream;
#pragma unroll
    for (int q = 0; q < kStream / kTile; ++q)
      tma_load_2d(smem_u32(st + C::B::BYTES + q * kTile * kShiftCols * 2), &tmshift, 0, srow + q * kTile,
                  b_qfull(s));
  };
  const int pre = min(nj, ST);   // query stages issued in the prologue (first use of each stage)
  if (threadIdx.x == 0) {
    // the resident key tile and the first query stages are requested before the CTA-wide
    // barrier, so their latency overlaps the TMEM allocation
    prefetch_tensormap(&tmq);
    prefetch_tensormap(&tmk);
    if (C::A::R > 0) {
      prefetch_tensormap(&tmq32);
      prefetch_tensormap(&tmk32);
    }
    prefetch_tensormap(&tmshift);
    mbar_arrive_expect_tx(b_afull, A2);
    load_tile<D, kTile>(sA, &tmk, &tmk32, g * D, t.k0[b] + krow0, b_afull);
    tma_load_2d(smem_u32(sA + C::A::BYTES), &tmones, 0, 0, b_afull);
    for (int j = 0; j < pre; ++j) issue_stage(j, j);
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&ctl->tmem_base), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem = ctl->tmem_base;

  if (warp == 0) {
    // The whole warp walks the stream: lane 0 issues the copies; on an image's last query tile,
    // when it holds rows past the image, all lanes overwrite those rows with zeros once the copy
    // has landed (they belong to the next image and may hold inf or NaN, which the -2^100 shift of
    // a padded row would not cancel), and then release the tile to the MMA.
    for (int j = 0; j < nj; ++j) {
      const int s = j % ST, u = j / ST;
      int ok = 1;
      if (j >= pre && lane == 0) {
        if (u > 0 && !mbar_wait(b_qempty(s), (u - 1) & 1, kWaitLimitNs)) {
          set_abort(ctl, status, K_ATTN_COLSUM);
          ok = 0;
        } else if (aborted(ctl)) {
          ok = 0;
        } else {
          issue_stage(j, s);
        }
      }
      const int rows = ragged_rows(j);
      if (rows < kStream) {
        if (lane == 0 && ok && !mbar_wait(b_qfull(s), u & 1, kWaitLimitNs)) {
          set_abort(ctl, status, K_ATTN_COLSUM);
          ok = 0;
        }
        if (__shfl_sync(0xffffffffu, ok, 0)) {
          zero_stage_rows<D>(sQ + s * B2, rows);
          fence_proxy_async_shared();
          __syncwarp();
          if (lane == 0) mbar_arrive(b_fixed(s));
        }
      }
      if (!__shfl_sync(0xffffffffu, ok, 0)) break;
    }
  } else if (warp == 1) {
    if (lane == 0) {
      uint64_t ak128, ak32, bq128, bq32;
      tile_desc<D, kTile>(sA, ak128, ak32);
      tile_desc<D, kStream>(sQ, bq128, bq32);
      const uint64_t aone = smem_desc_kmajor_sw32(smem_u32(sA + C::A::BYTES));
      const uint64_t bshift = smem_desc_kmajor_sw32(smem_u32(sQ + C::B::BYTES));
      bool ok = mbar_wait(b_afull, 0, kWaitLimitNs);
      if (!ok) set_abort(ctl, status, K_ATTN_COLSUM);
      for (int j = 0; ok && j < nj; ++j) {
        const int s = j % ST, u = j / ST;
        const int p = j & 1, v = j >> 1;
        if (!mbar_wait(b_qfull(s), u & 1, kWaitLimitNs) ||
            (v > 0 && !mbar_wait(b_sfree(p), (v - 1) & 1, kWaitLimitNs)) || aborted(ctl)) {
          set_abort(ctl, status, K_ATTN_COLSUM);
          break;
        }
        if (ragged_rows(j) < kStream && !mbar_wait(b_fixed(s), ragged_phase(j), kWaitLimitNs)) {
          set_abort(ctl, status, K_ATTN_COLSUM);
          break;
        }
        tc_fence_after_sync();
        const uint64_t so = static_cast<uint64_t>(s * (B2 >> 4));
        mma_tile<D>(tmem + p * 256, ak128, ak32, bq128 + so, bq32 + so);
        mma_bf16_ss(tmem + p * 256, aone, bshift + so, C::IDESC, 1);   // + (-L_i / c)
        mma_commit(b_sfull(p));
        mma_commit(b_qempty(s));
      }
      mma_commit(b_done);
    }
    __syncwarp();
  } else {
    // epilogue warpgroup e = 2p + hh: accumulator p (stream tiles j % 2 == p), query columns hh * 128 ..
    const int e = (warp - 2) >> 2;
    const int p = e >> 1, hh = e & 1;
    const int quad = warp & 3;
    const int rr = quad * 32 + lane;
    float2 acc = make_float2(0.f, 0.f), acc1 = acc;
    const uint32_t tbuf = tmem + (static_cast<uint32_t>(quad * 32) << 16) + p * 256 + hh * 128;
    const int key = krow0 + rr;
    for (int j = p; j < nj; j += 2) {
      const int v = j >> 1;
      const bool ok = __all_sync(0xffffffffu, mbar_wait(b_sfull(p), v & 1, kWaitLimitNs));
      if (!ok) {   // warp-uniform exit (see pass 1): the tcgen05.ld below is warp-wide
        set_abort(ctl, status, K_ATTN_COLSUM);
        break;
      }
      tc_fence_after_sync();
      // causal mask: query columns before `lo` do not see this thread's key
      int lo = 0;
      bool masked = false;
      if (CAUSAL) {
        lo = key - diag - ((qt_min + j % nspan) * kStream + hh * 128);
        masked = __any_sync(0xffffffffu, lo > 0);
      }
      uint32_t sv[64];
      load_cols64(tbuf, sv);
      if (masked) colsum64_from(sv, lo, c, acc, acc1);
      else colsum64(sv, c, acc, acc1);
      load_cols64(tbuf + 64, sv);
      tc_fence_before_sync();
      __syncwarp();
      if (lane == 0) mbar_arrive(b_sfree(p));
      if (masked) colsum64_from(sv, lo - 64, c, acc, acc1);
      else colsum64(sv, c, acc, acc1);
    }
    acc = fadd2(acc, acc1);
    const float a = acc.x + acc.y;
    if (e > 0) ctl->xchg[e - 1][0][rr] = a;
    named_barrier_sync(1, 32 * kEpiWarps);
    if (e == 0) {
      if (key < t.nk[b])
        part[static_cast<int64_t>(g) * t.ktot + t.out0[b] + key] =
            (a + ctl->xchg[0][0][rr]) + (ctl->xchg[1][0][rr] + ctl->xchg[2][0][rr]);
    }
  }
  cta_quiesce(ctl, b_done, 0, status, K_ATTN_COLSUM);
  cta_release_tmem(tmem);
}

// out[m] = sum over groups and the `merge` rows of token m of part[group][row].  Four lanes per
// output: lane j sums groups j, j + 4, .. in order, then the four partial sums are added by a
// fixed shuffle tree (the same bits for any launch), so 4x more loads are in flight than with
// one thread per output.
constexpr int kReduceLanes = 4;
__global__ void __launch_bounds__(256) attn_reduce(const float* __restrict__ part, int groups, int ktot, int merge,
                                                   float* __restrict__ out) {
  const int tid = blockIdx.x * blockDim.x + threadIdx.x;
  const int m = tid / kReduceLanes, j = tid % kReduceLanes;
  const int nout = ktot / merge;
  float s = 0.f;
  if (m < nout) {
    for (int g = j; g < groups; g += kReduceLanes) {
      const float* p = part + static_cast<int64_t>(g) * ktot + static_cast<int64_t>(m) * merge;
      float gs;
      if (merge == 4 && (ktot & 3) == 0) {   // 16-byte aligned rows of four
        const float4 v = __ldg(reinterpret_cast<const float4*>(p));
        gs = (v.x + v.y) + (v.z + v.w);
      } else {
        gs = 0.f;
        for (int q = 0; q < merge; ++q) gs += p[q];
      }
      s += gs;
    }
  }
  s += __shfl_xor_sync(0xffffffffu, s, 1);
  s += __shfl_xor_sync(0xffffffffu, s, 2);
  if (j == 0 && m < nout) out[m] = s;
}

// ------------------------------------------------------------------------------------------------
// host side
// ------------------------------------------------------------------------------------------------
PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static std::once_flag once;
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// 2-D map over a row-major bf16 matrix [rows, cols]; box = 64 columns (128-byte swizzle) or
// 16 columns (32-byte swizzle) x 128 rows.
pace_status_t make_map(CUtensorMap* m, const void* ptr, int64_t rows, int64_t cols, bool wide) {
  auto enc = tensor_map_encoder();
  if (enc == nullptr) return set_cuda_error(cudaErrorNotSupported);
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(cols * 2)};
  cuuint32_t box[2] = {wide ? 64u : 16u, static_cast<cuuint32_t>(kTile)};
  cuuint32_t es[2] = {1, 1};
  CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, es,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, wide ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_32B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return PACE_ERR_INVALID_ARG;
  return PACE_OK;
}

// One image of a call.  Pass 1: queries q0 .. q0 + nq - 1 of Q against keys k0 .. k0 + nk - 1
// of K, key k seen by query i iff k <= i + diag (diag >= 0).  Pass 2: the same queries against
// the scored keys v0 .. v0 + nv - 1 (rows of K), key j seen by query i iff j <= i + vdiag;
// scores go to output rows out0 .. out0 + nv - 1.
struct Seg {
  int q0, nq, k0, nk, diag;
  int v0, nv, vdiag, out0;
};

struct AttnLayout {
  int splits;
  int64_t prows, ktot;
  size_t L_off, part_off, ml_off, total;
};

// Key splits of pass 1.  A CTA costs about kSplitOverheadTiles streamed tiles of start-up and
// drain on top of its key tiles, and CTAs run in rounds of kPlanSms (one per SM), so the split
// count that minimises rounds x (tiles per CTA + overhead) is taken (the smallest on ties).  The
// GB300's SM count is a planning constant here, so that the workspace size queries need no device.
constexpr int kPlanSms = 152;
constexpr double kSplitOverheadTiles = 4.4;

int choose_splits(const std::vector<Seg>& segs, int H) {
  int64_t items = 0;
  int max_kt = 1;
  for (const Seg& sg : segs) {
    items += static_cast<int64_t>(H) * ((sg.nq + kPair - 1) / kPair);
    max_kt = std::max(max_kt, (sg.nk + kStream - 1) / kStream);
  }
  if (items == 0) return 1;
  int best = 1;
  double best_cost = 0.0;
  for (int s = 1; s <= std::min(max_kt, 32); ++s) {
    const int64_t rounds = (2 * items * s + kPlanSms - 1) / kPlanSms;
    const double cost = static_cast<double>(rounds) * ((max_kt + s - 1) / s + kSplitOverheadTiles);
    if (s == 1 || cost < best_cost) {
      best = s;
      best_cost = cost;
    }
  }
  return best;
}

AttnLayout attn_layout(const std::vector<Seg>& segs, int H, int groups) {
  AttnLayout L{};
  L.splits = choose_splits(segs, H);
  int64_t pr = 0, kt = 0;
  for (const Seg& sg : segs) {
    pr += static_cast<int64_t>((sg.nq + kPair - 1) / kPair) * kPair;
    kt += sg.nv;
  }
  L.prows = pr;   // every image's L rows start on a 256-row (1 KB) boundary
  L.ktot = kt;
  L.L_off = 0;
  L.part_off = align_up(static_cast<size_t>(H) * L.prows * kShiftCols * 2, 256);
  L.ml_off = L.part_off + align_up(static_cast<size_t>(groups) * L.ktot * sizeof(float), 256);
  L.total = L.ml_off;
  if (L.splits > 1) L.total += align_up(static_cast<size_t>(L.splits) * H * L.prows * sizeof(float2), 256);
  return L;
}

// Non-causal images: queries cu_q[b] .. against keys cu_k[b] .. in both passes.
std::vector<Seg> cross_segs(int B, const int32_t* cu_q, const int32_t* cu_k) {
  std::vector<Seg> segs(static_cast<size_t>(std::max(B, 0)));
  for (int b = 0; b < B; ++b) {
    const int nq = cu_q[b + 1] - cu_q[b], nk = cu_k[b + 1] - cu_k[b];
    segs[b] = Seg{cu_q[b], nq, cu_k[b], nk, kNoMask, cu_k[b], nk, kNoMask, cu_k[b]};
  }
  return segs;
}

// Causal sequences (full-sequence S_llm): image b is positions cu_seq[b] .. cu_seq[b+1] - 1 of Q
// and K, its visual tokens at local positions v .. v + nv - 1, queries from local position q_lo
// (the query set) to the end.
std::vector<Seg> sequence_segs(int B, const int32_t* cu_seq, const int32_t* vis_start, const int32_t* n_vis,
                               int query_set) {
  std::vector<Seg> segs(static_cast<size_t>(std::max(B, 0)));
  int out0 = 0;
  for (int b = 0; b < B; ++b) {
    const int S = cu_seq[b + 1] - cu_seq[b], v = vis_start[b], nv = n_vis[b];
    const int q_lo = query_set == PACE_QUERY_VISION_TEXT ? v : query_set == PACE_QUERY_TEXT ? v + nv : S - 1;
    segs[b] = Seg{cu_seq[b] + q_lo, S - q_lo, cu_seq[b], S, q_lo, cu_seq[b] + v, nv, q_lo - v, out0};
    out0 += nv;
  }
  return segs;
}

pace_status_t check_segments(int B, const int32_t* cu, int multiple) {
  if (cu == nullptr || cu[0] != 0) return PACE_ERR_INVALID_ARG;
  for (int b = 0; b < B; ++b) {
    const int n = cu[b + 1] - cu[b];
    if (n < 1 || n % multiple != 0 || cu[b] % multiple != 0) return PACE_ERR_INVALID_ARG;
  }
  return PACE_OK;
}

// Opts the two passes into their shared-memory size, once per device (so that later
// calls, including ones made during stream capture, only launch).
template <int D, bool CAUSAL>
pace_status_t set_smem_attrs(size_t* s1, size_t* s2) {
  using C = Cfg<D>;
  *s1 = 1024 + C::A::BYTES + C::STAGES * C::B::BYTES + sizeof(SmemCtl);
  *s2 = 1024 + C::A::BYTES + kTile * kShiftCols * 2 + C::STAGES * (C::B::BYTES + kStream * kShiftCols * 2) +
        sizeof(SmemCtl);
  static DeviceOnce once;
  int dev = 0;
  PACE_CUDA(cudaGetDevice(&dev));
  if (once.done(dev)) return PACE_OK;
  PACE_CUDA(cudaFuncSetAttribute(attn_row_lse<D, CAUSAL>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 static_cast<int>(*s1)));
  PACE_CUDA(cudaFuncSetAttribute(attn_colsum<D, CAUSAL>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 static_cast<int>(*s2)));
  once.mark(dev);
  return PACE_OK;
}

// Launches `items` work items of two independent CTAs each.
template <typename... Params, typename... Args>
pace_status_t launch_pairs(void (*kernel)(Params...), int items, size_t smem, cudaStream_t stream, Args... args) {
  if (items <= 0) return PACE_OK;
  kernel<<<dim3(2 * static_cast<unsigned>(items)), dim3(kThreads), smem, stream>>>(args...);
  return check_launch();
}

// Pass 1 in pieces: piece c waits for event ready[c] and takes the query pairs whose last row
// (a global row of Q) is below end_row[c] (and not below end_row[c - 1]).
struct QueryChunks {
  int n = 0;
  const int64_t* end_row = nullptr;
  cudaEvent_t const* ready = nullptr;
};

template <int D, bool CAUSAL>
pace_status_t run_importance(const void* Q, const void* K, int64_t qrows, int64_t krows,
                             const std::vector<Seg>& segs, int Hq, int Hkv, float scale, int merge, float* out,
                             void* ws, cudaStream_t stream, const QueryChunks& chunks = QueryChunks{}) {
  const int B = static_cast<int>(segs.size());
  const int G = Hq / Hkv;
  const AttnLayout Lay = attn_layout(segs, Hq, Hkv);
  uint8_t* w8 = static_cast<uint8_t*>(ws);
  uint16_t* Lw = reinterpret_cast<uint16_t*>(w8 + Lay.L_off);
  float* part = reinterpret_cast<float*>(w8 + Lay.part_off);
  float2* ml = Lay.splits > 1 ? reinterpret_cast<float2*>(w8 + Lay.ml_off) : nullptr;
  int* status = device_status_word();
  CUtensorMap mq, mq32, mk, mk32;
  qrows = std::max<int64_t>(qrows, 1);
  krows = std::max<int64_t>(krows, 1);
  PACE_CHECK(make_map(&mq, Q, qrows, static_cast<int64_t>(Hq) * D, true));
  PACE_CHECK(make_map(&mk, K, krows, static_cast<int64_t>(Hkv) * D, true));
  PACE_CHECK(make_map(&mq32, Q, qrows, static_cast<int64_t>(Hq) * D, false));
  PACE_CHECK(make_map(&mk32, K, krows, static_cast<int64_t>(Hkv) * D, false));
  CUtensorMap mshift, mones;
  PACE_CHECK(make_map(&mshift, Lw, std::max<int64_t>(static_cast<int64_t>(Hq) * Lay.prows, 1), kShiftCols, false));
  const void* ones = nullptr;
  PACE_CUDA(cudaGetSymbolAddress(const_cast<void**>(&ones), g_ones_slice));
  PACE_CHECK(make_map(&mones, ones, kTile, kShiftCols, false));
  size_t s1 = 0, s2 = 0;
  PACE_CHECK((set_smem_attrs<D, CAUSAL>(&s1, &s2)));
  const float c = static_cast<float>(static_cast<double>(scale) * 1.4426950408889634);
  int lpad = 0;
  for (int c0 = 0; c0 < B; c0 += kAttnMaxB) {
    const int nb = std::min(kAttnMaxB, B - c0);
    AttnTable t{};
    t.nb = nb;
    t.H = Hq;
    t.G = G;
    t.splits = Lay.splits;
    t.prows = static_cast<int>(Lay.prows);
    t.ktot = static_cast<int>(Lay.ktot);
    int items1 = 0, ctiles = 0;
    t.item_prefix[0] = 0;
    for (int i = 0; i < nb; ++i) {
      const Seg& sg = segs[c0 + i];
      t.q0[i] = sg.q0;
      t.nq[i] = sg.nq;
      t.k0[i] = sg.k0;
      t.nk[i] = sg.nk;
      t.diag[i] = sg.diag;
      t.lpad[i] = lpad;
      lpad += (sg.nq + kPair - 1) / kPair * kPair;
      items1 += Hq * ((sg.nq + kPair - 1) / kPair) * Lay.splits;
      t.item_prefix[i + 1] = items1;
      ctiles += (sg.nq + kPair - 1) / kPair * 2;
    }
    const int pieces = chunks.n > 0 ? chunks.n : 1;
    for (int pc = 0; pc < pieces; ++pc) {
      int items_pc = 0;
      t.item_prefix[0] = 0;
      for (int i = 0; i < nb; ++i) {
        const Seg& sg = segs[c0 + i];
        const int npair = (sg.nq + kPair - 1) / kPair;
        int lo = 0, hi = npair;
        if (chunks.n > 0) {   // pairs whose last row falls in [end_row[pc - 1], end_row[pc])
          auto last_row = [&](int pr) { return static_cast<int64_t>(sg.q0) + std::min((pr + 1) * kPair, sg.nq) - 1; };
          const int64_t from = pc > 0 ? chunks.end_row[pc - 1] : INT64_MIN, to = chunks.end_row[pc];
          while (lo < npair && last_row(lo) < from) ++lo;
          hi = lo;
          while (hi < npair && last_row(hi) < to) ++hi;
        }
        t.pair_lo[i] = lo;
        t.pair_n[i] = hi - lo;
        items_pc += Hq * (hi - lo) * Lay.splits;
        t.item_prefix[i + 1] = items_pc;
      }
      if (chunks.n > 0) PACE_CUDA(cudaStreamWaitEvent(stream, chunks.ready[pc], 0));
      PACE_CHECK(launch_pairs(attn_row_lse<D, CAUSAL>, items_pc, s1, stream, mq, mq32, mk, mk32, t, c, Lw, ml, status));
    }
    (void)items1;
    if (Lay.splits > 1 && ctiles > 0) {
      attn_lse_combine<<<dim3(ctiles, Hq), kTile, 0, stream>>>(t, c, ml, Lw);
      PACE_CHECK(check_launch());
    }
    // pass 2 streams the same query rows (and L rows) against the scored keys
    int items2 = 0;
    for (int i = 0; i < nb; ++i) {
      const Seg& sg = segs[c0 + i];
      t.k0[i] = sg.v0;
      t.nk[i] = sg.nv;
      t.diag[i] = sg.vdiag;
      t.out0[i] = sg.out0;
      items2 += Hkv * ((sg.nv + kPair - 1) / kPair);
      t.item_prefix[i + 1] = items2;
    }
    PACE_CHECK(launch_pairs(attn_colsum<D, CAUSAL>, items2, s2, stream, mq, mq32, mk, mk32, mshift, mones, t, c, part,
                            status));
  }
  const int nout = static_cast<int>(Lay.ktot / merge);
  if (nout > 0) {
    attn_reduce<<<(nout * kReduceLanes + 255) / 256, 256, 0, stream>>>(part, Hkv, static_cast<int>(Lay.ktot), merge,
                                                                         out);
    PACE_CHECK(check_launch());
  }
  return PACE_OK;
}

pace_status_t check_heads(int Hq, int Hkv, int D, float scale, const void* Q, const void* K) {
  if (Q == nullptr || K == nullptr) return PACE_ERR_INVALID_ARG;
  if (Hq < 1 || Hkv < 1 || Hq % Hkv != 0 || Hq > 256) return PACE_ERR_INVALID_ARG;
  if (D != 64 && D != 80 && D != 128) return PACE_ERR_INVALID_ARG;
  if (!(scale > 0.f) || !std::isfinite(scale)) return PACE_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(Q) | reinterpret_cast<uintptr_t>(K)) % 16) return PACE_ERR_INVALID_ARG;
  return PACE_OK;
}

template <bool CAUSAL>
pace_status_t dispatch(const void* Q, const void* K, int64_t qrows, int64_t krows, const std::vector<Seg>& segs,
                       int Hq, int Hkv, int D, float scale, int merge, float* out, void* ws, size_t ws_bytes,
                       cudaStream_t stream, const QueryChunks& chunks = QueryChunks{}) {
  const AttnLayout Lay = attn_layout(segs, Hq, Hkv);
  if (ws == nullptr || ws_bytes < Lay.total || reinterpret_cast<uintptr_t>(ws) % 16) return PACE_ERR_WORKSPACE;
  PACE_CHECK(check_device());
  switch (D) {
    case 64: return run_importance<64, CAUSAL>(Q, K, qrows, krows, segs, Hq, Hkv, scale, merge, out, ws, stream, chunks);
    case 80: return run_importance<80, CAUSAL>(Q, K, qrows, krows, segs, Hq, Hkv, scale, merge, out, ws, stream, chunks);
    default: return run_importance<128, CAUSAL>(Q, K, qrows, krows, segs, Hq, Hkv, scale, merge, out, ws, stream, chunks);
  }
}

pace_status_t importance(const void* Q, const void* K, const int32_t* cu_q, const int32_t* cu_k, int B, int Hq,
                         int Hkv, int D, float scale, int merge, float* out, void* ws, size_t ws_bytes,
                         cudaStream_t stream, const QueryChunks& chunks = QueryChunks{}) {
  if (B < 0) return PACE_ERR_INVALID_ARG;
  if (B == 0) return PACE_OK;
  if (out == nullptr) return PACE_ERR_INVALID_ARG;
  PACE_CHECK(check_heads(Hq, Hkv, D, scale, Q, K));
  PACE_CHECK(check_segments(B, cu_q, cu_q == cu_k ? merge : 1));
  if (cu_k != cu_q) PACE_CHECK(check_segments(B, cu_k, merge));
  if (static_cast<int64_t>(cu_q[B]) + static_cast<int64_t>(kTile) * B > (int64_t{1} << 30)) return PACE_ERR_INVALID_ARG;
  return dispatch<false>(Q, K, cu_q[B], cu_k[B], cross_segs(B, cu_q, cu_k), Hq, Hkv, D, scale, merge, out, ws, ws_bytes,
                  stream, chunks);
}

// Checks the sequence layout of the full-sequence S_llm.
pace_status_t check_sequences(int B, const int32_t* cu_seq, const int32_t* vis_start, const int32_t* n_vis,
                              int query_set) {
  if (cu_seq == nullptr || vis_start == nullptr || n_vis == nullptr || cu_seq[0] != 0) return PACE_ERR_INVALID_ARG;
  if (query_set != PACE_QUERY_VISION_TEXT && query_set != PACE_QUERY_TEXT && query_set != PACE_QUERY_LAST)
    return PACE_ERR_INVALID_ARG;
  for (int b = 0; b < B; ++b) {
    const int64_t S = static_cast<int64_t>(cu_seq[b + 1]) - cu_seq[b];
    if (S < 1 || vis_start[b] < 0 || n_vis[b] < 1 || static_cast<int64_t>(vis_start[b]) + n_vis[b] > S)
      return PACE_ERR_INVALID_ARG;
  }
  if (static_cast<int64_t>(cu_seq[B]) + static_cast<int64_t>(kTile) * B > (int64_t{1} << 30)) return PACE_ERR_INVALID_ARG;
  return PACE_OK;
}

}  // namespace
}  // namespace pace

using namespace pace;

extern "C" size_t pace_vit_attn_importance_workspace_size(int B, const int32_t* cu_seqlens, int n_heads) {
  if (B <= 0 || cu_seqlens == nullptr || n_heads < 1) return 0;
  return attn_layout(cross_segs(B, cu_seqlens, cu_seqlens), n_heads, n_heads).total;
}

extern "C" pace_status_t pace_vit_attn_importance(const void* Q, const void* K, const int32_t* cu_seqlens, int B,
                                                  int n_heads, int head_dim, float scale, int merge,
                                                  float* s_vis_raw, void* ws, size_t ws_bytes,
                                                  pace_stream_t stream) {
  if (merge != 1 && merge != 2 && merge != 4) return PACE_ERR_INVALID_ARG;
  return importance(Q, K, cu_seqlens, cu_seqlens, B, n_heads, n_heads, head_dim, scale, merge, s_vis_raw, ws,
                    ws_bytes, stream);
}

extern "C" size_t pace_llm_text_visual_importance_workspace_size(int B, const int32_t* cu_q, const int32_t* cu_k,
                                                                 int n_q_heads, int n_kv_heads) {
  if (B <= 0 || cu_q == nullptr || cu_k == nullptr || n_q_heads < 1 || n_kv_heads < 1) return 0;
  return attn_layout(cross_segs(B, cu_q, cu_k), n_q_heads, n_kv_heads).total;
}

extern "C" pace_status_t pace_llm_text_visual_importance(const void* Q, const void* K, const int32_t* cu_q,
                                                         const int32_t* cu_k, int B, int n_q_heads,
                                                         int n_kv_heads, int head_dim, float scale,
                                                         float* s_llm_raw, void* ws, size_t ws_bytes,
                                                         pace_stream_t stream) {
  return importance(Q, K, cu_q, cu_k, B, n_q_heads, n_kv_heads, head_dim, scale, 1, s_llm_raw, ws, ws_bytes,
                    stream);
}

extern "C" size_t pace_llm_sequence_importance_workspace_size(int B, const int32_t* cu_seq, const int32_t* vis_start,
                                                              const int32_t* n_vis, int n_q_heads, int n_kv_heads,
                                                              int query_set) {
  if (B <= 0 || n_q_heads < 1 || n_kv_heads < 1) return 0;
  if (check_sequences(B, cu_seq, vis_start, n_vis, query_set) != PACE_OK) return 0;
  return attn_layout(sequence_segs(B, cu_seq, vis_start, n_vis, query_set), n_q_heads, n_kv_heads).total;
}

extern "C" pace_status_t pace_llm_sequence_importance(const void* Q, const void* K, const int32_t* cu_seq,
                                                      const int32_t* vis_start, const int32_t* n_vis, int B,
                                                      int n_q_heads, int n_kv_heads, int head_dim, float scale,
                                                      int query_set, float* s_llm_raw, void* ws, size_t ws_bytes,
                                                      pace_stream_t stream) {
  if (B < 0) return PACE_ERR_INVALID_ARG;
  if (B == 0) return PACE_OK;
  if (s_llm_raw == nullptr) return PACE_ERR_INVALID_ARG;
  PACE_CHECK(check_heads(n_q_heads, n_kv_heads, head_dim, scale, Q, K));
  PACE_CHECK(check_sequences(B, cu_seq, vis_start, n_vis, query_set));
  return dispatch<true>(Q, K, cu_seq[B], cu_seq[B], sequence_segs(B, cu_seq, vis_start, n_vis, query_set), n_q_heads,
                  n_kv_heads, head_dim, scale, 1, s_llm_raw, ws, ws_bytes, stream);
}

extern "C" pace_status_t pace_vit_attn_importance_chunked(const void* Q, const void* K, const int32_t* cu_seqlens,
                                                          int B, int n_heads, int head_dim, float scale, int merge,
                                                          float* s_vis_raw, void* ws, size_t ws_bytes, int n_chunks,
                                                          const int64_t* chunk_end_rows, void* const* chunk_ready,
                                                          pace_stream_t stream) {
  if (merge != 1 && merge != 2 && merge != 4) return PACE_ERR_INVALID_ARG;
  if (B < 0) return PACE_ERR_INVALID_ARG;
  if (B == 0) return PACE_OK;
  if (cu_seqlens == nullptr || n_chunks < 1 || n_chunks > 64 || chunk_end_rows == nullptr || chunk_ready == nullptr)
    return PACE_ERR_INVALID_ARG;
  for (int c = 0; c < n_chunks; ++c) {
    if (chunk_ready[c] == nullptr || chunk_end_rows[c] < 0) return PACE_ERR_INVALID_ARG;
    if (c > 0 && chunk_end_rows[c] < chunk_end_rows[c - 1]) return PACE_ERR_INVALID_ARG;
  }
  if (chunk_end_rows[n_chunks - 1] != cu_seqlens[B]) return PACE_ERR_INVALID_ARG;
  QueryChunks ch;
  ch.n = n_chunks;
  ch.end_row = chunk_end_rows;
  ch.ready = reinterpret_cast<cudaEvent_t const*>(chunk_ready);
  return importance(Q, K, cu_seqlens, cu_seqlens, B, n_heads, n_heads, head_dim, scale, merge, s_vis_raw, ws,
                    ws_bytes, stream, ch);
}
