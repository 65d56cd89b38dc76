// Extract: ViT received attention (S_vis) and LLM text->visual attention (S_llm), Sec. 3.3.
//
// Both maps are column sums of a row-softmax attention matrix, a_j = sum_i P_ij with
// P_ij = exp(s_ij - lse_i), s_ij = scale q_i . k_j.  They are computed flash-style in two
// passes so that the N x N score matrix is never stored:
//
//   pass 1  attn_row_lse   S = Q K^T tile by tile on tcgen05 (M = 128 query rows, N = 128
//           keys), online row max / sum of exp2 on the CUDA cores, giving the base-2
//           log-sum-exp L_i = log2 sum_j 2^(c s_ij), c = scale * log2(e).  Optionally split
//           over key ranges (partial (m, l) pairs merged by attn_lse_combine).
//   pass 2  attn_colsum    S^T = K Q^T (M = 128 keys, N = 128 queries): every TMEM lane is one
//           key, so each epilogue thread owns one key and accumulates 2^(c s_ji - L_i) over
//           the whole query stream in registers; no cross-thread reduction and no atomics.
//   reduce  attn_reduce    sums the per-head (or per KV-head) partial maps and pools the
//           `merge` consecutive patches of each merged token.
//
// CTA layout of both passes (320 threads):
//   warp 0      TMA producer (one lane): resident operand tiles once, then a 4-6 stage ring
//   warp 1      TMEM allocation (512 columns) and MMA issue (one lane)
//   warps 2-9   two epilogue warpgroups; warpgroup w owns resident tile w (two query tiles
//               in pass 1, two key tiles in pass 2) and its two TMEM accumulators
//               (double-buffered: columns w*256 + {0, 128})
// Operands are K-major bf16 tiles staged by TMA with the 32-byte swizzle (16 elements of the
// head dimension per row), one tile per 16-wide slice of the head dimension.
//
// GQA: query head h reads KV head h / G.  The ViT case is G = 1.
#include <atomic>
#include <cmath>
#include <mutex>

#include <cudaTypedefs.h>

#include "pace_common.cuh"
#include "pace_ptx.cuh"

namespace pace {
namespace {

using namespace ptx;

constexpr int kTile = 128;
constexpr int kThreads = 320;
constexpr int kAttnMaxB = 64;
constexpr int kSliceBytes = kTile * 32;   // one 128-row x 16-element bf16 slice
constexpr uint32_t kTmemCols = 512;
constexpr int kTargetItems = 304;         // 2 CTAs' worth per SM on 152 SMs

template <int D>
struct Cfg {
  static constexpr int KC = D / 16;                       // slices of the head dimension
  static constexpr int STAGES = (D == 128) ? 4 : (D == 80 ? 4 : 6);
  static constexpr int TILE_BYTES = KC * kSliceBytes;
  static constexpr uint32_t IDESC = idesc_bf16_f32(128, 128);
};

struct AttnTable {
  int q0[kAttnMaxB], nq[kAttnMaxB];   // query rows of image b
  int k0[kAttnMaxB], nk[kAttnMaxB];   // key rows of image b
  int lpad[kAttnMaxB];                // first padded L row of image b
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
  uint64_t bars[32];
  uint32_t tmem_base;
  int abort;
};

__device__ __forceinline__ void set_abort(SmemCtl* ctl, int* status, int kernel) {
  *reinterpret_cast<volatile int*>(&ctl->abort) = 1;
  record_error(status, PACE_ERR_TIMEOUT, kernel);
}
__device__ __forceinline__ bool aborted(const SmemCtl* ctl) {
  return *reinterpret_cast<const volatile int*>(&ctl->abort) != 0;
}

// Loads 4 x 32 TMEM columns of this warp's 32 lanes into v[0..127] (fp32 bit patterns).
__device__ __forceinline__ void load_row128(uint32_t taddr, uint32_t (&v)[4][32]) {
  tmem_ld_32x32b_x32(taddr + 0, v[0]);
  tmem_ld_32x32b_x32(taddr + 32, v[1]);
  tmem_ld_32x32b_x32(taddr + 64, v[2]);
  tmem_ld_32x32b_x32(taddr + 96, v[3]);
  tmem_wait_ld();
  reg_fence32(v[0]);
  reg_fence32(v[1]);
  reg_fence32(v[2]);
  reg_fence32(v[3]);
}

// ------------------------------------------------------------------------------------------------
// pass 1: row log-sum-exp
// ------------------------------------------------------------------------------------------------
template <int D>
__global__ void __launch_bounds__(kThreads, 1) attn_row_lse(const __grid_constant__ CUtensorMap tmq,
                                                            const __grid_constant__ CUtensorMap tmk,
                                                            const __grid_constant__ AttnTable t, float c,
                                                            float* __restrict__ L_out,
                                                            float2* __restrict__ ml_out, int* status) {
  using C = Cfg<D>;
  constexpr int KC = C::KC, ST = C::STAGES;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = smem;                                // 2 resident query tiles
  uint8_t* sK = sQ + 2 * C::TILE_BYTES;              // ST key stages
  SmemCtl* ctl = reinterpret_cast<SmemCtl*>(sK + ST * C::TILE_BYTES);
  const uint32_t b_qfull = smem_u32(&ctl->bars[0]);
  const uint32_t b_done = smem_u32(&ctl->bars[1]);
  auto b_kfull = [&](int s) { return smem_u32(&ctl->bars[2 + s]); };
  auto b_kempty = [&](int s) { return smem_u32(&ctl->bars[2 + ST + s]); };
  auto b_sfull = [&](int i) { return smem_u32(&ctl->bars[2 + 2 * ST + i]); };
  auto b_sfree = [&](int i) { return smem_u32(&ctl->bars[2 + 2 * ST + 4 + i]); };

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int item = blockIdx.x;
  const int b = find_image(t, item);
  int r = item - t.item_prefix[b];
  const int split = r % t.splits;
  r /= t.splits;
  const int npair = (t.nq[b] + 2 * kTile - 1) / (2 * kTile);
  const int pair = r % npair;
  const int h = r / npair;
  const int g = h / t.G;
  const int qrow0 = pair * 2 * kTile;                               // local query row of tile 0
  const int nqt = min(2, (t.nq[b] - qrow0 + kTile - 1) / kTile);    // 1 or 2 valid query tiles
  const int nkt_all = (t.nk[b] + kTile - 1) / kTile;
  const int kt0 = static_cast<int>((static_cast<int64_t>(split) * nkt_all) / t.splits);
  const int kt1 = static_cast<int>((static_cast<int64_t>(split + 1) * nkt_all) / t.splits);
  const int nj = kt1 - kt0;

  if (threadIdx.x == 0) {
    mbar_init(b_qfull, 1);
    mbar_init(b_done, 1);
    for (int s = 0; s < ST; ++s) {
      mbar_init(b_kfull(s), 1);
      mbar_init(b_kempty(s), 1);
    }
    for (int i = 0; i < 4; ++i) {
      mbar_init(b_sfull(i), 1);
      mbar_init(b_sfree(i), 4);
    }
    ctl->abort = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&ctl->tmem_base), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem = ctl->tmem_base;
  int issued = 0;

  if (warp == 0) {
    if (lane == 0) {
      prefetch_tensormap(&tmq);
      prefetch_tensormap(&tmk);
      mbar_arrive_expect_tx(b_qfull, nqt * C::TILE_BYTES);
      for (int qt = 0; qt < nqt; ++qt)
        for (int kc = 0; kc < KC; ++kc)
          tma_load_2d(smem_u32(sQ + (qt * KC + kc) * kSliceBytes), &tmq, h * D + kc * 16,
                      t.q0[b] + qrow0 + qt * kTile, b_qfull);
      for (int j = 0; j < nj; ++j) {
        const int s = j % ST, u = j / ST;
        if (u > 0 && !mbar_wait(b_kempty(s), (u - 1) & 1, kWaitLimitNs)) {
          set_abort(ctl, status, K_ATTN_ROW_LSE);
          break;
        }
        if (aborted(ctl)) break;
        mbar_arrive_expect_tx(b_kfull(s), C::TILE_BYTES);
        const int krow = t.k0[b] + (kt0 + j) * kTile;
        for (int kc = 0; kc < KC; ++kc)
          tma_load_2d(smem_u32(sK + (s * KC + kc) * kSliceBytes), &tmk, g * D + kc * 16, krow, b_kfull(s));
        issued = j + 1;
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      bool ok = mbar_wait(b_qfull, 0, kWaitLimitNs);
      if (!ok) set_abort(ctl, status, K_ATTN_ROW_LSE);
      for (int j = 0; ok && j < nj; ++j) {
        const int s = j % ST, u = j / ST;
        if (!mbar_wait(b_kfull(s), u & 1, kWaitLimitNs) || aborted(ctl)) {
          set_abort(ctl, status, K_ATTN_ROW_LSE);
          break;
        }
        tc_fence_after_sync();
        const int buf = j & 1, v = j >> 1;
        for (int qt = 0; qt < nqt; ++qt) {
          if (v > 0 && !mbar_wait(b_sfree(qt * 2 + buf), (v - 1) & 1, kWaitLimitNs)) {
            set_abort(ctl, status, K_ATTN_ROW_LSE);
            ok = false;
            break;
          }
          tc_fence_after_sync();
          const uint32_t d = tmem + qt * 256 + buf * 128;
#pragma unroll
          for (int kc = 0; kc < KC; ++kc)
            mma_bf16_ss(d, smem_desc_kmajor_sw32(smem_u32(sQ + (qt * KC + kc) * kSliceBytes)),
                        smem_desc_kmajor_sw32(smem_u32(sK + (s * KC + kc) * kSliceBytes)), C::IDESC, kc > 0);
          mma_commit(b_sfull(qt * 2 + buf));
        }
        mma_commit(b_kempty(s));
      }
      mma_commit(b_done);
      if (!mbar_wait(b_done, 0, kWaitLimitNs)) record_error(status, PACE_ERR_TIMEOUT, K_ATTN_ROW_LSE);
    }
    __syncwarp();
  } else {
    // epilogue: warpgroup qt = (warp - 2) / 4, TMEM lane quadrant = warp % 4
    const int qt = (warp - 2) >> 2;
    const int quad = warp & 3;
    const int rr = quad * 32 + lane;
    if (qt < nqt) {
      float m_run = -INFINITY, l_run = 0.f;
      const uint32_t trow = tmem + (static_cast<uint32_t>(quad * 32) << 16) + qt * 256;
      for (int j = 0; j < nj; ++j) {
        const int buf = j & 1, v = j >> 1;
        const bool ok = __all_sync(0xffffffffu, mbar_wait(b_sfull(qt * 2 + buf), v & 1, kWaitLimitNs));
        if (!ok || aborted(ctl)) {   // warp-uniform exit: the tcgen05.ld below is warp-wide
          set_abort(ctl, status, K_ATTN_ROW_LSE);
          break;
        }
        tc_fence_after_sync();
        uint32_t sv[4][32];
        load_row128(trow + buf * 128, sv);
        tc_fence_before_sync();
        __syncwarp();
        if (lane == 0) mbar_arrive(b_sfree(qt * 2 + buf));
        const int valid = t.nk[b] - (kt0 + j) * kTile;   // keys of this tile inside the image
        if (valid < kTile) {
#pragma unroll
          for (int a = 0; a < 4; ++a)
#pragma unroll
            for (int e = 0; e < 32; ++e)
              if (a * 32 + e >= valid) sv[a][e] = __float_as_uint(-INFINITY);
        }
        float mx0 = -INFINITY, mx1 = -INFINITY, mx2 = -INFINITY, mx3 = -INFINITY;
#pragma unroll
        for (int e = 0; e < 32; e += 2) {
          mx0 = max3(mx0, __uint_as_float(sv[0][e]), __uint_as_float(sv[0][e + 1]));
          mx1 = max3(mx1, __uint_as_float(sv[1][e]), __uint_as_float(sv[1][e + 1]));
          mx2 = max3(mx2, __uint_as_float(sv[2][e]), __uint_as_float(sv[2][e + 1]));
          mx3 = max3(mx3, __uint_as_float(sv[3][e]), __uint_as_float(sv[3][e + 1]));
        }
        const float mt = fmaxf(fmaxf(mx0, mx1), fmaxf(mx2, mx3)) * c;
        if (mt > m_run) {
          l_run *= ex2_approx(m_run - mt);
          m_run = mt;
        }
        const float nm = -m_run;
        float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
#pragma unroll
        for (int e = 0; e < 32; ++e) {
          a0 += ex2_approx(fmaf(__uint_as_float(sv[0][e]), c, nm));
          a1 += ex2_approx(fmaf(__uint_as_float(sv[1][e]), c, nm));
          a2 += ex2_approx(fmaf(__uint_as_float(sv[2][e]), c, nm));
          a3 += ex2_approx(fmaf(__uint_as_float(sv[3][e]), c, nm));
        }
        l_run += (a0 + a1) + (a2 + a3);
      }
      const int row = qrow0 + qt * kTile + rr;          // local query row
      const int64_t prow = static_cast<int64_t>(h) * t.prows + t.lpad[b] + row;
      if (t.splits == 1) {
        L_out[prow] = row < t.nq[b] ? m_run + log2f(l_run) : INFINITY;
      } else {
        ml_out[static_cast<int64_t>(split) * t.H * t.prows + prow] =
            row < t.nq[b] ? make_float2(m_run, l_run) : make_float2(-INFINITY, 0.f);
      }
    }
  }

  // teardown: every wait above is bounded, so all threads arrive here
  tc_fence_before_sync();
  __syncthreads();
  if (warp == 0 && lane == 0 && aborted(ctl)) {
    // let in-flight TMA loads land before the CTA's shared memory is released
    mbar_wait(b_qfull, 0, kWaitLimitNs);
    for (int j = max(0, issued - ST); j < issued; ++j) mbar_wait(b_kfull(j % ST), (j / ST) & 1, kWaitLimitNs);
  }
  tc_fence_after_sync();
  if (warp == 1) tmem_dealloc(tmem, kTmemCols);
}

// Merges per-split (m, l) pairs into L = m + log2(l); rows past the image get +inf.
__global__ void __launch_bounds__(128) attn_lse_combine(const __grid_constant__ AttnTable t,
                                                        const float2* __restrict__ ml, float* __restrict__ L_out) {
  // blockIdx.x = (h, image, tile) flattened through per-image tile counts
  int rem = blockIdx.x;
  const int h = blockIdx.y;
  int b = 0;
  for (; b < t.nb; ++b) {
    const int nt = (t.nq[b] + kTile - 1) / kTile;
    if (rem < nt) break;
    rem -= nt;
  }
  if (b >= t.nb) return;
  const int row = rem * kTile + threadIdx.x;
  const int64_t prow = static_cast<int64_t>(h) * t.prows + t.lpad[b] + row;
  if (row >= t.nq[b]) {
    L_out[prow] = INFINITY;
    return;
  }
  float M = -INFINITY;
  for (int s = 0; s < t.splits; ++s) M = fmaxf(M, ml[static_cast<int64_t>(s) * t.H * t.prows + prow].x);
  float l = 0.f;
  for (int s = 0; s < t.splits; ++s) {
    const float2 p = ml[static_cast<int64_t>(s) * t.H * t.prows + prow];
    if (p.y > 0.f) l += p.y * ex2_approx(p.x - M);
  }
  L_out[prow] = M + log2f(l);
}

// ------------------------------------------------------------------------------------------------
// pass 2: column sums of 2^(c s - L)
// ------------------------------------------------------------------------------------------------
template <int D>
__global__ void __launch_bounds__(kThreads, 1) attn_colsum(const __grid_constant__ CUtensorMap tmq,
                                                           const __grid_constant__ CUtensorMap tmk,
                                                           const __grid_constant__ AttnTable t, float c,
                                                           const float* __restrict__ L, float* __restrict__ part,
                                                           int* status) {
  using C = Cfg<D>;
  constexpr int KC = C::KC, ST = C::STAGES;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;                                 // 2 resident key tiles
  uint8_t* sQ = sA + 2 * C::TILE_BYTES;               // ST query stages
  float* sL = reinterpret_cast<float*>(sQ + ST * C::TILE_BYTES);   // ST x 128 floats
  SmemCtl* ctl = reinterpret_cast<SmemCtl*>(sL + ST * kTile);
  const uint32_t b_afull = smem_u32(&ctl->bars[0]);
  const uint32_t b_done = smem_u32(&ctl->bars[1]);
  auto b_qfull = [&](int s) { return smem_u32(&ctl->bars[2 + s]); };
  auto b_qempty = [&](int s) { return smem_u32(&ctl->bars[2 + ST + s]); };
  auto b_sfull = [&](int i) { return smem_u32(&ctl->bars[2 + 2 * ST + i]); };
  auto b_sfree = [&](int i) { return smem_u32(&ctl->bars[2 + 2 * ST + 4 + i]); };

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int item = blockIdx.x;
  const int b = find_image(t, item);
  const int r = item - t.item_prefix[b];
  const int nkp = (t.nk[b] + 2 * kTile - 1) / (2 * kTile);
  const int kp = r % nkp;
  const int g = r / nkp;
  const int krow0 = kp * 2 * kTile;                                   // local key row of tile 0
  const int nkt = min(2, (t.nk[b] - krow0 + kTile - 1) / kTile);
  const int nqt = (t.nq[b] + kTile - 1) / kTile;
  const int nj = t.G * nqt;                                           // stream: (head in group, query tile)

  if (threadIdx.x == 0) {
    mbar_init(b_afull, 1);
    mbar_init(b_done, 1);
    for (int s = 0; s < ST; ++s) {
      mbar_init(b_qfull(s), 1);
      mbar_init(b_qempty(s), 1 + 4 * nkt);
    }
    for (int i = 0; i < 4; ++i) {
      mbar_init(b_sfull(i), 1);
      mbar_init(b_sfree(i), 4);
    }
    ctl->abort = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&ctl->tmem_base), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem = ctl->tmem_base;
  int issued = 0;

  if (warp == 0) {
    if (lane == 0) {
      prefetch_tensormap(&tmq);
      prefetch_tensormap(&tmk);
      mbar_arrive_expect_tx(b_afull, nkt * C::TILE_BYTES);
      for (int kt = 0; kt < nkt; ++kt)
        for (int kc = 0; kc < KC; ++kc)
          tma_load_2d(smem_u32(sA + (kt * KC + kc) * kSliceBytes), &tmk, g * D + kc * 16,
                      t.k0[b] + krow0 + kt * kTile, b_afull);
      for (int j = 0; j < nj; ++j) {
        const int s = j % ST, u = j / ST;
        if (u > 0 && !mbar_wait(b_qempty(s), (u - 1) & 1, kWaitLimitNs)) {
          set_abort(ctl, status, K_ATTN_COLSUM);
          break;
        }
        if (aborted(ctl)) break;
        const int hh = j / nqt, qt = j - hh * nqt;
        const int h = g * t.G + hh;
        mbar_arrive_expect_tx(b_qfull(s), C::TILE_BYTES + kTile * 4);
        for (int kc = 0; kc < KC; ++kc)
          tma_load_2d(smem_u32(sQ + (s * KC + kc) * kSliceBytes), &tmq, h * D + kc * 16, t.q0[b] + qt * kTile,
                      b_qfull(s));
        bulk_load(smem_u32(sL + s * kTile), L + static_cast<int64_t>(h) * t.prows + t.lpad[b] + qt * kTile,
                  kTile * 4, b_qfull(s));
        issued = j + 1;
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      bool ok = mbar_wait(b_afull, 0, kWaitLimitNs);
      if (!ok) set_abort(ctl, status, K_ATTN_COLSUM);
      for (int j = 0; ok && j < nj; ++j) {
        const int s = j % ST, u = j / ST;
        if (!mbar_wait(b_qfull(s), u & 1, kWaitLimitNs) || aborted(ctl)) {
          set_abort(ctl, status, K_ATTN_COLSUM);
          break;
        }
        tc_fence_after_sync();
        const int buf = j & 1, v = j >> 1;
        for (int kt = 0; kt < nkt; ++kt) {
          if (v > 0 && !mbar_wait(b_sfree(kt * 2 + buf), (v - 1) & 1, kWaitLimitNs)) {
            set_abort(ctl, status, K_ATTN_COLSUM);
            ok = false;
            break;
          }
          tc_fence_after_sync();
          const uint32_t d = tmem + kt * 256 + buf * 128;
#pragma unroll
          for (int kc = 0; kc < KC; ++kc)
            mma_bf16_ss(d, smem_desc_kmajor_sw32(smem_u32(sA + (kt * KC + kc) * kSliceBytes)),
                        smem_desc_kmajor_sw32(smem_u32(sQ + (s * KC + kc) * kSliceBytes)), C::IDESC, kc > 0);
          mma_commit(b_sfull(kt * 2 + buf));
        }
        mma_commit(b_qempty(s));
      }
      mma_commit(b_done);
      if (!mbar_wait(b_done, 0, kWaitLimitNs)) record_error(status, PACE_ERR_TIMEOUT, K_ATTN_COLSUM);
    }
    __syncwarp();
  } else {
    const int kt = (warp - 2) >> 2;
    const int quad = warp & 3;
    const int rr = quad * 32 + lane;
    if (kt < nkt) {
      float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
      const uint32_t trow = tmem + (static_cast<uint32_t>(quad * 32) << 16) + kt * 256;
      for (int j = 0; j < nj; ++j) {
        const int buf = j & 1, v = j >> 1;
        const int s = j % ST, u = j / ST;
        const bool ok = __all_sync(0xffffffffu, mbar_wait(b_sfull(kt * 2 + buf), v & 1, kWaitLimitNs));
        if (!ok || aborted(ctl)) {   // warp-uniform exit: the tcgen05.ld below is warp-wide
          set_abort(ctl, status, K_ATTN_COLSUM);
          break;
        }
        tc_fence_after_sync();
        uint32_t sv[4][32];
        load_row128(trow + buf * 128, sv);
        tc_fence_before_sync();
        __syncwarp();
        if (lane == 0) mbar_arrive(b_sfree(kt * 2 + buf));
        if (!__all_sync(0xffffffffu, mbar_wait(b_qfull(s), u & 1, kWaitLimitNs))) {   // L of this stage (landed)
          set_abort(ctl, status, K_ATTN_COLSUM);
          break;
        }
        const float4* Lp = reinterpret_cast<const float4*>(sL + s * kTile);
#pragma unroll
        for (int a = 0; a < 4; ++a) {
#pragma unroll
          for (int e = 0; e < 32; e += 4) {
            const float4 l4 = Lp[a * 8 + e / 4];
            a0 += ex2_approx(fmaf(__uint_as_float(sv[a][e + 0]), c, -l4.x));
            a1 += ex2_approx(fmaf(__uint_as_float(sv[a][e + 1]), c, -l4.y));
            a2 += ex2_approx(fmaf(__uint_as_float(sv[a][e + 2]), c, -l4.z));
            a3 += ex2_approx(fmaf(__uint_as_float(sv[a][e + 3]), c, -l4.w));
          }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(b_qempty(s));
      }
      const int key = krow0 + kt * kTile + rr;
      if (key < t.nk[b]) part[static_cast<int64_t>(g) * t.ktot + t.k0[b] + key] = (a0 + a1) + (a2 + a3);
    }
  }

  tc_fence_before_sync();
  __syncthreads();
  if (warp == 0 && lane == 0 && aborted(ctl)) {
    // let in-flight TMA loads land before the CTA's shared memory is released
    mbar_wait(b_afull, 0, kWaitLimitNs);
    for (int j = max(0, issued - ST); j < issued; ++j) mbar_wait(b_qfull(j % ST), (j / ST) & 1, kWaitLimitNs);
  }
  tc_fence_after_sync();
  if (warp == 1) tmem_dealloc(tmem, kTmemCols);
}

// out[m] = sum over groups and the `merge` rows of token m of part[group][row].
__global__ void __launch_bounds__(256) attn_reduce(const float* __restrict__ part, int groups, int ktot, int merge,
                                                   float* __restrict__ out) {
  const int m = blockIdx.x * blockDim.x + threadIdx.x;
  const int nout = ktot / merge;
  if (m >= nout) return;
  float s = 0.f;
  for (int g = 0; g < groups; ++g) {
    const float* p = part + static_cast<int64_t>(g) * ktot + static_cast<int64_t>(m) * merge;
    float gs = 0.f;
    for (int q = 0; q < merge; ++q) gs += p[q];
    s += gs;
  }
  out[m] = s;
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

// 2-D map over a row-major bf16 matrix [rows, cols]; box = 16 columns x 128 rows, 32-byte swizzle.
pace_status_t make_map(CUtensorMap* m, const void* ptr, int64_t rows, int64_t cols) {
  auto enc = tensor_map_encoder();
  if (enc == nullptr) return set_cuda_error(cudaErrorNotSupported);
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(cols * 2)};
  cuuint32_t box[2] = {16, kTile};
  cuuint32_t es[2] = {1, 1};
  CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, es,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_32B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return PACE_ERR_INVALID_ARG;
  return PACE_OK;
}

struct AttnLayout {
  int splits;
  int64_t prows, ktot, qtot;
  size_t L_off, part_off, ml_off, total;
};

// Key splits of pass 1: enough items to cover the GPU about twice.
int choose_splits(int B, const int32_t* cu_q, const int32_t* cu_k, int H) {
  int64_t items = 0;
  int max_kt = 1;
  for (int b = 0; b < B; ++b) {
    const int nq = cu_q[b + 1] - cu_q[b], nk = cu_k[b + 1] - cu_k[b];
    items += static_cast<int64_t>(H) * ((nq + 2 * kTile - 1) / (2 * kTile));
    max_kt = std::max(max_kt, (nk + kTile - 1) / kTile);
  }
  if (items >= kTargetItems || items == 0) return 1;
  int s = static_cast<int>((kTargetItems + items - 1) / items);
  s = std::min(s, std::min(max_kt, 32));
  return std::max(s, 1);
}

AttnLayout attn_layout(int B, const int32_t* cu_q, const int32_t* cu_k, int H, int groups) {
  AttnLayout L{};
  L.splits = choose_splits(B, cu_q, cu_k, H);
  L.qtot = cu_q[B];
  L.ktot = cu_k[B];
  int64_t pr = 0;
  for (int b = 0; b < B; ++b) pr += static_cast<int64_t>((cu_q[b + 1] - cu_q[b] + kTile - 1) / kTile) * kTile;
  L.prows = pr;   // every image's L rows start on a 128-row (512-byte) boundary
  L.L_off = 0;
  L.part_off = align_up(static_cast<size_t>(H) * L.prows * sizeof(float), 256);
  L.ml_off = L.part_off + align_up(static_cast<size_t>(groups) * L.ktot * sizeof(float), 256);
  L.total = L.ml_off;
  if (L.splits > 1) L.total += align_up(static_cast<size_t>(L.splits) * H * L.prows * sizeof(float2), 256);
  return L;
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
template <int D>
pace_status_t set_smem_attrs(size_t* s1, size_t* s2) {
  using C = Cfg<D>;
  *s1 = 1024 + 2 * C::TILE_BYTES + C::STAGES * C::TILE_BYTES + sizeof(SmemCtl);
  *s2 = 1024 + 2 * C::TILE_BYTES + C::STAGES * C::TILE_BYTES + C::STAGES * kTile * 4 + sizeof(SmemCtl);
  static std::atomic<uint64_t> done{0};
  int dev = 0;
  PACE_CUDA(cudaGetDevice(&dev));
  const uint64_t bit = uint64_t{1} << (dev & 63);
  if (done.load(std::memory_order_acquire) & bit) return PACE_OK;
  PACE_CUDA(cudaFuncSetAttribute(attn_row_lse<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(*s1)));
  PACE_CUDA(cudaFuncSetAttribute(attn_colsum<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(*s2)));
  done.fetch_or(bit, std::memory_order_acq_rel);
  return PACE_OK;
}

template <int D>
pace_status_t run_importance(const void* Q, const void* K, const int32_t* cu_q, const int32_t* cu_k, int B, int Hq,
                             int Hkv, float scale, int merge, float* out, void* ws, cudaStream_t stream) {
  const int G = Hq / Hkv;
  const AttnLayout Lay = attn_layout(B, cu_q, cu_k, Hq, Hkv);
  uint8_t* w8 = static_cast<uint8_t*>(ws);
  float* Lw = reinterpret_cast<float*>(w8 + Lay.L_off);
  float* part = reinterpret_cast<float*>(w8 + Lay.part_off);
  float2* ml = Lay.splits > 1 ? reinterpret_cast<float2*>(w8 + Lay.ml_off) : nullptr;
  int* status = device_status_word();
  CUtensorMap mq, mk;
  PACE_CHECK(make_map(&mq, Q, std::max<int64_t>(Lay.qtot, 1), static_cast<int64_t>(Hq) * D));
  PACE_CHECK(make_map(&mk, K, std::max<int64_t>(Lay.ktot, 1), static_cast<int64_t>(Hkv) * D));
  size_t s1 = 0, s2 = 0;
  PACE_CHECK(set_smem_attrs<D>(&s1, &s2));
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
      const int b = c0 + i;
      t.q0[i] = cu_q[b];
      t.nq[i] = cu_q[b + 1] - cu_q[b];
      t.k0[i] = cu_k[b];
      t.nk[i] = cu_k[b + 1] - cu_k[b];
      t.lpad[i] = lpad;
      lpad += (t.nq[i] + kTile - 1) / kTile * kTile;
      items1 += Hq * ((t.nq[i] + 2 * kTile - 1) / (2 * kTile)) * Lay.splits;
      t.item_prefix[i + 1] = items1;
      ctiles += (t.nq[i] + kTile - 1) / kTile;
    }
    attn_row_lse<D><<<items1, kThreads, s1, stream>>>(mq, mk, t, c, Lw, ml, status);
    PACE_CHECK(check_launch());
    if (Lay.splits > 1) {
      attn_lse_combine<<<dim3(ctiles, Hq), kTile, 0, stream>>>(t, ml, Lw);
      PACE_CHECK(check_launch());
    }
    int items2 = 0;
    for (int i = 0; i < nb; ++i) {
      items2 += Hkv * ((t.nk[i] + 2 * kTile - 1) / (2 * kTile));
      t.item_prefix[i + 1] = items2;
    }
    attn_colsum<D><<<items2, kThreads, s2, stream>>>(mq, mk, t, c, Lw, part, status);
    PACE_CHECK(check_launch());
  }
  const int nout = static_cast<int>(Lay.ktot / merge);
  attn_reduce<<<(nout + 255) / 256, 256, 0, stream>>>(part, Hkv, static_cast<int>(Lay.ktot), merge, out);
  return check_launch();
}

pace_status_t importance(const void* Q, const void* K, const int32_t* cu_q, const int32_t* cu_k, int B, int Hq,
                         int Hkv, int D, float scale, int merge, float* out, void* ws, size_t ws_bytes,
                         cudaStream_t stream) {
  if (B < 0) return PACE_ERR_INVALID_ARG;
  if (B == 0) return PACE_OK;
  if (Q == nullptr || K == nullptr || out == nullptr) return PACE_ERR_INVALID_ARG;
  if (Hq < 1 || Hkv < 1 || Hq % Hkv != 0 || Hq > 256) return PACE_ERR_INVALID_ARG;
  if (D != 64 && D != 80 && D != 128) return PACE_ERR_INVALID_ARG;
  if (!(scale > 0.f) || !std::isfinite(scale)) return PACE_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(Q) | reinterpret_cast<uintptr_t>(K)) % 16) return PACE_ERR_INVALID_ARG;
  PACE_CHECK(check_segments(B, cu_q, cu_q == cu_k ? merge : 1));
  if (cu_k != cu_q) PACE_CHECK(check_segments(B, cu_k, merge));
  if (static_cast<int64_t>(cu_q[B]) + static_cast<int64_t>(kTile) * B > (int64_t{1} << 30)) return PACE_ERR_INVALID_ARG;
  const AttnLayout Lay = attn_layout(B, cu_q, cu_k, Hq, Hkv);
  if (ws == nullptr || ws_bytes < Lay.total || reinterpret_cast<uintptr_t>(ws) % 16) return PACE_ERR_WORKSPACE;
  PACE_CHECK(check_device());
  switch (D) {
    case 64: return run_importance<64>(Q, K, cu_q, cu_k, B, Hq, Hkv, scale, merge, out, ws, stream);
    case 80: return run_importance<80>(Q, K, cu_q, cu_k, B, Hq, Hkv, scale, merge, out, ws, stream);
    default: return run_importance<128>(Q, K, cu_q, cu_k, B, Hq, Hkv, scale, merge, out, ws, stream);
  }
}

}  // namespace
}  // namespace pace

using namespace pace;

extern "C" size_t pace_vit_attn_importance_workspace_size(int B, const int32_t* cu_seqlens, int n_heads) {
  if (B <= 0 || cu_seqlens == nullptr || n_heads < 1) return 0;
  return attn_layout(B, cu_seqlens, cu_seqlens, n_heads, n_heads).total;
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
  return attn_layout(B, cu_q, cu_k, n_q_heads, n_kv_heads).total;
}

extern "C" pace_status_t pace_llm_text_visual_importance(const void* Q, const void* K, const int32_t* cu_q,
                                                         const int32_t* cu_k, int B, int n_q_heads,
                                                         int n_kv_heads, int head_dim, float scale,
                                                         float* s_llm_raw, void* ws, size_t ws_bytes,
                                                         pace_stream_t stream) {
  return importance(Q, K, cu_q, cu_k, B, n_q_heads, n_kv_heads, head_dim, scale, 1, s_llm_raw, ws, ws_bytes,
                    stream);
}
