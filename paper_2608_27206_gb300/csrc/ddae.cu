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
#include "pace_select.cuh"

namespace pace {
namespace {

constexpr int kSelThreads = 1024;
constexpr int kSelMaxB = 256;

struct SelectTable {
  int v0[kSelMaxB];  // first global row of image b
  int nv[kSelMaxB];  // visual tokens of image b
  int k0[kSelMaxB];  // first output slot of image b
  int nk[kSelMaxB];  // tokens kept for image b
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

// Block-wide reduction of two values; every thread gets the result.  `red` holds 2*32 floats.
template <int OP>  // 0 = sum, 1 = min, 2 = max
__device__ __forceinline__ float2 block_reduce2(float a, float b, float* red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (OP == 0) { a = warp_sum(a); b = warp_sum(b); }
  if (OP == 1) { a = warp_min(a); b = warp_min(b); }
  if (OP == 2) { a = warp_max(a); b = warp_max(b); }
  __syncthreads();
  if (lane == 0) { red[warp] = a; red[32 + warp] = b; }
  __syncthreads();
  if (warp == 0) {
    a = red[lane];
    b = red[32 + lane];
    if (OP == 0) { a = warp_sum(a); b = warp_sum(b); }
    if (OP == 1) { a = warp_min(a); b = warp_min(b); }
    if (OP == 2) { a = warp_max(a); b = warp_max(b); }
    if (lane == 0) { red[0] = a; red[32] = b; }
  }
  __syncthreads();
  return make_float2(red[0], red[32]);
}

__global__ void __launch_bounds__(kSelThreads) ddae_select_kernel(const float* __restrict__ s_llm,
                                                                  const float* __restrict__ s_vis,
                                                                  const __grid_constant__ SelectTable tab,
                                                                  float tau, int fusion, float* __restrict__ s_final,
                                                                  float* __restrict__ weights,
                                                                  int32_t* __restrict__ kept, int b_base) {
  extern __shared__ float sm[];
  __shared__ float red[64];
  __shared__ int wsum[33];
  __shared__ unsigned hist[256];
  __shared__ unsigned sel[2];
  const int b = blockIdx.x;
  const int nv = tab.nv[b], v0 = tab.v0[b];
  float* A = sm;        // S_llm raw -> normalised -> S_final
  float* V = sm + nv;   // S_vis raw -> normalised
  const int tid = threadIdx.x;

  // 1. stage both maps, min / max
  float amin = FLT_MAX, amax = -FLT_MAX, vmin = FLT_MAX, vmax = -FLT_MAX;
  for (int i = tid; i < nv; i += kSelThreads) {
    const float a = s_llm[v0 + i], v = s_vis[v0 + i];
    A[i] = a;
    V[i] = v;
    amin = fminf(amin, a); amax = fmaxf(amax, a);
    vmin = fminf(vmin, v); vmax = fmaxf(vmax, v);
  }
  const float2 mn = block_reduce2<1>(amin, vmin, red);
  const float2 mx = block_reduce2<2>(amax, vmax, red);
  const float ar = mx.x - mn.x, vr = mx.y - mn.y;

  // 2. min-max normalisation (a constant map becomes 0) and the means
  float sa = 0.f, sv = 0.f;
  for (int i = tid; i < nv; i += kSelThreads) {
    const float a = ar > 0.f ? __fdiv_rn(A[i] - mn.x, ar) : 0.f;
    const float v = vr > 0.f ? __fdiv_rn(V[i] - mn.y, vr) : 0.f;
    A[i] = a;
    V[i] = v;
    sa += a;
    sv += v;
  }
  const float2 sums = block_reduce2<0>(sa, sv, red);
  const float ma = sums.x / nv, mv = sums.y / nv;
  float qa = 0.f, qv = 0.f;
  for (int i = tid; i < nv; i += kSelThreads) {
    const float da = A[i] - ma, dv = V[i] - mv;
    qa = fmaf(da, da, qa);
    qv = fmaf(dv, dv, qv);
  }
  const float2 sq = block_reduce2<0>(qa, qv, red);
  const float sig_a = sqrtf(sq.x / nv), sig_v = sqrtf(sq.y / nv);

  // 3. Eq. 7: confidence-weighted softmax fusion (or a fixed-weight ablation)
  float wa, wv;
  if (fusion == PACE_DDAE_ONLY_LLM) {
    wa = 1.f;
    wv = 0.f;
  } else if (fusion == PACE_DDAE_ONLY_VIT) {
    wa = 0.f;
    wv = 1.f;
  } else if (fusion == PACE_DDAE_FIXED) {
    wa = wv = 0.5f;
  } else {
    const float za = sig_a / tau, zv = sig_v / tau, zm = fmaxf(za, zv);
    const float ea = expf(za - zm), ev = expf(zv - zm);
    wa = ea / (ea + ev);
    wv = ev / (ea + ev);
  }
  if (tid == 0 && weights != nullptr) {
    weights[2 * (b_base + b)] = wa;
    weights[2 * (b_base + b) + 1] = wv;
  }
  for (int i = tid; i < nv; i += kSelThreads) {
    const float f = fmaf(wa, A[i], wv * V[i]);
    A[i] = f;
    if (s_final != nullptr) s_final[v0 + i] = f;
  }
  __syncthreads();

  // 4. top-K threshold by radix select on the fp32 bits
  const int K = tab.nk[b], k0 = tab.k0[b];
  if (K <= 0) return;
  if (K >= nv) {
    for (int i = tid; i < nv; i += kSelThreads) kept[k0 + i] = v0 + i;
    return;
  }
  unsigned prefix = 0u, mask = 0u;
  unsigned remaining = static_cast<unsigned>(K);
  const int lane = tid & 31;
  for (int shift = 24; shift >= 0; shift -= 8) {
    for (int i = tid; i < 256; i += kSelThreads) hist[i] = 0u;
    __syncthreads();
    // histogram of the next digit; lanes holding the same digit are combined first, so a
    // narrow value range costs one shared atomic per distinct digit per warp
    for (int base = 0; base < nv; base += kSelThreads) {
      const int i = base + tid;
      const unsigned key = i < nv ? __float_as_uint(A[i]) : 0u;
      const bool in = i < nv && (key & mask) == prefix;
      const unsigned digit = in ? ((key >> shift) & 255u) : 256u;
      const unsigned peers = __match_any_sync(0xffffffffu, digit);
      if (in && lane == __ffs(peers) - 1) atomicAdd(&hist[digit], static_cast<unsigned>(__popc(peers)));
    }
    __syncthreads();
    if (tid < 32) warp_digit_search(hist, remaining, sel);
    __syncthreads();
    prefix |= sel[0] << shift;
    mask |= 255u << shift;
    remaining -= sel[1];
    __syncthreads();
  }
  const unsigned T = prefix;  // bit pattern of the K-th largest S_final
  // `remaining` = how many keys equal to T are kept (lowest indices first)

  // 5. ascending compaction: the kept tokens before index i are the keys > T before i plus
  // min(keys == T before i, remaining), so one packed prefix count per chunk places them
  int gt_run = 0, eq_run = 0;
  const unsigned lt_mask = (1u << lane) - 1u;
  const int warp = tid >> 5;
  for (int base = 0; base < nv; base += kSelThreads) {
    const int i = base + tid;
    const unsigned key = i < nv ? __float_as_uint(A[i]) : 0u;
    const bool gt = i < nv && key > T;
    const bool eq = i < nv && key == T;
    const unsigned bg = __ballot_sync(0xffffffffu, gt), be = __ballot_sync(0xffffffffu, eq);
    if (lane == 0) wsum[warp] = static_cast<int>(__popc(bg) | (__popc(be) << 16));
    __syncthreads();
    if (warp == 0) {
      const int v = wsum[lane];
      int incl = v;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int n = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += n;
      }
      wsum[lane] = incl - v;
      if (lane == 31) wsum[32] = incl;
    }
    __syncthreads();
    const int wp = wsum[warp];
    const int gt_before = gt_run + (wp & 0xffff) + __popc(bg & lt_mask);
    const int eq_before = eq_run + (wp >> 16) + __popc(be & lt_mask);
    if (gt || (eq && static_cast<unsigned>(eq_before) < remaining))
      kept[k0 + gt_before + min(eq_before, static_cast<int>(remaining))] = v0 + i;
    gt_run += wsum[32] & 0xffff;
    eq_run += wsum[32] >> 16;
    __syncthreads();
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
    if (nv < 1 || nv > PACE_DDAE_MAX_TOKENS || nk < 0 || nk > nv) return PACE_ERR_INVALID_ARG;
    if (nv > max_nv) max_nv = nv;
  }
  if (cu_keep[B] > 0 && kept == nullptr) return PACE_ERR_INVALID_ARG;
  const float tau = params ? params->tau : 0.5f;
  const int fusion = params ? params->fusion : PACE_DDAE_ADAPTIVE;
  if (!(tau > 0.f) || !std::isfinite(tau)) return PACE_ERR_INVALID_ARG;
  if (fusion < PACE_DDAE_ADAPTIVE || fusion > PACE_DDAE_FIXED) return PACE_ERR_INVALID_ARG;
  PACE_CHECK(check_device());
  const size_t smem = static_cast<size_t>(2 * max_nv) * sizeof(float);
  {
    // opt in to the largest size once per device
    static DeviceOnce once;
    int dev = 0;
    PACE_CUDA(cudaGetDevice(&dev));
    if (!once.done(dev)) {
      PACE_CUDA(cudaFuncSetAttribute(ddae_select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     static_cast<int>(2 * PACE_DDAE_MAX_TOKENS * sizeof(float))));
      once.mark(dev);
    }
  }
  for (int c0 = 0; c0 < B; c0 += kSelMaxB) {
    const int nb = (B - c0) < kSelMaxB ? (B - c0) : kSelMaxB;
    SelectTable t;
    for (int i = 0; i < nb; ++i) {
      const int b = c0 + i;
      t.v0[i] = cu_v[b];
      t.nv[i] = cu_v[b + 1] - cu_v[b];
      t.k0[i] = cu_keep[b];
      t.nk[i] = cu_keep[b + 1] - cu_keep[b];
    }
    ddae_select_kernel<<<nb, kSelThreads, smem, stream>>>(s_llm_raw, s_vis_raw, t, tau, fusion, s_final, weights, kept,
                                                           c0);
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
