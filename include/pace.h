/*
 * libpace — C ABI of the GB300 (sm_103a) condense-and-extract hot path of PACE
 * (arxiv 2608.27206, "PACE: A Unified Condense-and-Extract Paradigm for Fast
 * VLM Inference").
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 *  - Every call returns a pace_status_t.  Arguments are checked on the host
 *    before anything is launched; a rejected call launches nothing.
 *  - "device" pointers are caller-owned device memory on the current CUDA
 *    device; "host" arrays are read during the call only (they are copied into
 *    kernel parameters), so they may be freed or reused as soon as it returns.
 *  - Nothing is allocated or freed inside a call.  Scratch memory comes from the
 *    caller as (ws, ws_bytes), sized by the matching *_workspace_size query;
 *    a too-small workspace returns PACE_ERR_WORKSPACE.
 *  - All work is enqueued on `stream` (a cudaStream_t; NULL = legacy default
 *    stream) and runs asynchronously.  Launch failures return PACE_ERR_CUDA
 *    and the CUDA error code is kept for pace_last_cuda_error().
 *  - Device-side waits are bounded.  A kernel whose wait runs out records
 *    PACE_ERR_TIMEOUT in the device status word (pace_device_status) and
 *    returns early; its outputs are then undefined.
 *  - The library runs only on sm_103 devices (GB300); elsewhere every compute
 *    call returns PACE_ERR_UNSUPPORTED_ARCH.  There is no CPU fallback.
 *  - bf16 tensors are passed as `const void*` holding IEEE bfloat16 values.
 */
#ifndef PACE_H_
#define PACE_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#if defined(__GNUC__)
#define PACE_API __attribute__((visibility("default")))
#else
#define PACE_API
#endif

typedef struct CUstream_st* pace_stream_t; /* same type as cudaStream_t */

typedef enum pace_status_t {
  PACE_OK = 0,
  PACE_ERR_INVALID_ARG = 1,      /* a size, pointer or parameter is out of range */
  PACE_ERR_UNSUPPORTED_ARCH = 2, /* the current device is not an sm_103 GPU */
  PACE_ERR_WORKSPACE = 3,        /* ws_bytes smaller than the size query returned */
  PACE_ERR_CUDA = 4,             /* a CUDA runtime call or launch failed */
  PACE_ERR_TIMEOUT = 5           /* a bounded device-side wait ran out (device status word) */
} pace_status_t;

/* Human-readable name of a status code (static string). */
PACE_API const char* pace_status_string(pace_status_t status);

/* CUDA error code (cudaError_t) of the last PACE_ERR_CUDA on the calling thread. */
PACE_API int pace_last_cuda_error(void);

/* Checks that `device` is an sm_103 GPU and prepares per-device state (device
 * status word).  Optional: every entry point does the same check lazily.
 * Each call starts the device's set-up afresh: the status word is cleared and its
 * address, the addresses of the library's device arrays and the kernels' shared-memory
 * opt-ins are looked up again on the next call that needs them.  After cudaDeviceReset
 * (or anything else that destroys the device's primary context) call pace_init again
 * before any other call on that device; the cached values of the old context are stale.
 * Call it while no other libpace call is in flight on that device. */
PACE_API pace_status_t pace_init(int device);

/* Reads the device status word of the current device (synchronises the device).
 * *code = PACE_OK or PACE_ERR_TIMEOUT; *where = the kernel that recorded it
 * (0 if none).  With clear != 0 the word is reset to PACE_OK afterwards. */
PACE_API pace_status_t pace_device_status(int* code, int* where, int clear);

/* Exercises the bounded-wait path: launches one CTA that waits on a barrier nothing ever
 * arrives at.  After limit_us microseconds (1 .. 1000000) the wait gives up, the kernel
 * records PACE_ERR_TIMEOUT (kernel id 11) in the device status word and returns; the CUDA
 * context stays usable.  For failure-detection tests of callers. */
PACE_API pace_status_t pace_selftest_wait_timeout(uint32_t limit_us, pace_stream_t stream);

/* Number of CUDA kernels this library has launched in the calling process (all threads,
 * all devices).  Instrumentation for benchmarks: counts launches, not completed work. */
PACE_API uint64_t pace_kernel_launch_count(void);

/* ==============================================================================
 * Condense — Adaptive Pixel Compressor (APC), Sec. 3.2, Eq. 1-6; App. B.3.
 * ============================================================================== */

typedef struct pace_apc_params {
  float alpha;     /* weight of rho_g in rho = alpha rho_g + (1-alpha) rho_d (Eq. 6); 0.6 */
  float gamma;     /* local contrast scale of rho_d = min(d_top / gamma, 1) (Eq. 5); 1.5  */
  float tail_frac; /* fraction of tokens averaged into d_top; 0.10                         */
  float r_min;     /* lower clamp of the retention ratio r; 0                             */
  float r_max;     /* hard budget cap of r (Sec. 3.2, Adaptive Condensation); 1           */
  int32_t align;   /* output sides are multiples of this (merge unit); 28                 */
} pace_apc_params;

/* Per-image result of pace_apc_density (written on the device). */
typedef struct pace_apc_stats {
  float phi;         /* mean pairwise cosine of the preview tokens (Eq. 1) */
  float rho_g;       /* 1 - phi (Eq. 2) */
  float d_top;       /* mean of the k_tail largest d_i */
  float rho_d;       /* min(d_top / gamma, 1) (Eq. 5) */
  float rho;         /* alpha rho_g + (1 - alpha) rho_d (Eq. 6) */
  float r;           /* min(max(rho, r_min), r_max): retained area ratio */
  int32_t n_patches; /* N = (H/14) (W/14) */
  int32_t k_tail;    /* max(1, floor(tail_frac N + 0.5)) */
  int32_t h_out;     /* min(H, max(align, align * floor(H sqrt(r) / align + 0.5))) */
  int32_t w_out;     /* same for W */
} pace_apc_stats;

/* Fills the paper's defaults: alpha 0.6, gamma 1.5, tail 10 %, r in [0, 1], align 28. */
PACE_API void pace_apc_params_default(pace_apc_params* params);

/* Scratch bytes needed by pace_apc_density for these images (host arrays H, W). */
PACE_API size_t pace_apc_density_workspace_size(int B, const int32_t* H, const int32_t* W);

/*
 * APC information density of B images (Sec. 3.2, Eq. 1-6, "per-region density on
 * raw pixels").  The preview token of 14x14 patch i is the stand-in
 * T_i = [x_i / 255 ; 1] (x_i = the patch's 588 bytes in row, column, channel
 * order); t_i = T_i / |T_i|; c = mean t_i; phi = |c|^2 (equal to Eq. 1's double
 * sum); c_hat = c / |c|; d_i = |t_i - c_hat| (Eq. 4).
 *
 *  img      device  uint8 HWC images; image b starts at byte img_off[b], 16-byte aligned
 *  img_off  host    int64 [B]
 *  H, W     host    int32 [B]; multiples of 14, >= 14
 *  params   host    NULL for the defaults
 *  d_out    device  float [sum N_b]: d_i of every patch, images in order, patches in
 *                   raster order (may be NULL)
 *  stats    device  pace_apc_stats [B]
 *  ws       device  >= pace_apc_density_workspace_size(B, H, W) bytes, 16-byte aligned
 */
PACE_API pace_status_t pace_apc_density(const uint8_t* img, const int64_t* img_off, const int32_t* H, const int32_t* W,
                               int B, const pace_apc_params* params, float* d_out, pace_apc_stats* stats,
                               void* ws, size_t ws_bytes, pace_stream_t stream);

/*
 * pace_apc_density without caller scratch.  The paper has no counterpart to this call:
 * it exists for callers that cannot allocate device memory themselves, such as a plugin
 * running inside a host framework that owns every allocation, or a latency-critical path
 * where cudaMalloc (which may synchronise the device) is not allowed.  It computes exactly
 * what pace_apc_density computes, with the same kernels, but its scratch lives in one
 * file-scope device array owned by the library (about 860 KB on every GPU that loads the
 * library, held until the process exits).  It allocates and frees nothing.
 *
 *  - At most PACE_APC_STATIC_MAX_IMAGES images and PACE_APC_STATIC_MAX_PATCHES patches
 *    (14x14) in total per call; larger calls return PACE_ERR_INVALID_ARG and launch nothing.
 *  - d_out is required (the per-patch distances are an output, not scratch).
 *  - The first call on a device looks up the array's device address (cudaGetSymbolAddress)
 *    with that device current; make that first call before any stream capture.  The
 *    address is kept until pace_init(device) is called again, which a device reset
 *    requires (the old address belongs to the destroyed context).
 *  - Every call shares the one array and it keeps the last call's contents (the call clears
 *    the part that must start at zero).  Calls whose work overlaps on the GPU — on different
 *    streams, or from different threads — race on it; serialise them.
 * Other arguments are as for pace_apc_density.
 */
#define PACE_APC_STATIC_MAX_IMAGES 16
#define PACE_APC_STATIC_MAX_PATCHES 65536
PACE_API pace_status_t pace_apc_density_static(const uint8_t* img, const int64_t* img_off, const int32_t* H,
                                               const int32_t* W, int B, const pace_apc_params* params,
                                               float* d_out, pace_apc_stats* stats, pace_stream_t stream);

/*
 * APC density on preview tokens (Sec. 3.2 "Shallow Feature Preview", Eq. 1-6): the paper's
 * own input, the token embeddings T_v of the first ViT block, instead of the pixel stand-in.
 * Per image b with tokens T_i (rows cu_tokens[b] .. cu_tokens[b+1]-1): t_hat_i = T_i / |T_i|
 * (a zero token counts as t_hat = 0), c = mean t_hat, phi = |c|^2 (= Eq. 1), rho_g = 1 - phi,
 * c_hat = c / |c| (0 when c = 0), d_i = |t_hat_i - c_hat|, then the same tail mean, rho_d,
 * rho, r and target size as pace_apc_density (the target size from the image's H, W).
 *
 *  T          device  bf16 [cu_tokens[B], D] row-major, 4-byte aligned; D even, 2 <= D <= 4096
 *  cu_tokens  host    int32 [B+1] prefix, cu_tokens[0] = 0, at least one token per image
 *  H, W       host    int32 [B] size of each image in pixels (for h_out, w_out)
 *  params     host    NULL for the paper's defaults
 *  d_out      device  float [cu_tokens[B]], one distance per token
 *  stats      device  pace_apc_stats [B] (n_patches = the token count)
 *  ws         device  >= pace_apc_density_tokens_workspace_size(B, cu_tokens, D) bytes, 16-B aligned
 */
PACE_API size_t pace_apc_density_tokens_workspace_size(int B, const int32_t* cu_tokens, int D);
PACE_API pace_status_t pace_apc_density_tokens(const void* T, const int32_t* cu_tokens, int B, int D,
                                               const int32_t* H, const int32_t* W, const pace_apc_params* params,
                                               float* d_out, pace_apc_stats* stats, void* ws, size_t ws_bytes,
                                               pace_stream_t stream);

/* Pixel-statistic previews: the four training-free statistics that the preview ablation
 * (App. "Shallow Feature Preview Ablation") puts in place of the ViT feature.  The paper names
 * them without a definition; these are the readings used here, per 14 x 14 patch, with integer
 * luma Y' = 299 R + 587 G + 114 B (Y = Y' / 255000) and the patch's 12 x 12 interior for the
 * 3 x 3 operators:
 *   RGB_STATS      [mean_R, mean_G, mean_B, std_R, std_G, std_B, 1] of x / 255 (population std)
 *   COLOR_ENTROPY  [H_R, H_G, H_B, 4] / 4, H_c the entropy in bits of the 16-bin histogram
 *                  (value >> 4) of channel c
 *   EDGE_DENSITY   [e, 1], e the fraction of interior pixels whose Sobel magnitude of Y > 0.25
 *                  (decided exactly, in integers)
 *   LAPLACIAN      [s, 1], s the population std of the 4-neighbour Laplacian of Y
 * A token is stored as 8 floats, zero-padded. */
typedef enum pace_apc_feature {
  PACE_APC_FEATURE_RGB_STATS = 0,
  PACE_APC_FEATURE_COLOR_ENTROPY = 1,
  PACE_APC_FEATURE_EDGE_DENSITY = 2,
  PACE_APC_FEATURE_LAPLACIAN = 3
} pace_apc_feature;

/*
 * The feature tokens of every patch (raster order per image, images packed).
 *
 *  img, img_off, H, W, B  as for pace_apc_density
 *  feature   pace_apc_feature
 *  tokens    device  float [sum N_b][8], 16-byte aligned
 *  Invalid arguments: PACE_ERR_INVALID_ARG before any launch.
 */
PACE_API pace_status_t pace_apc_pixel_features(const uint8_t* img, const int64_t* img_off, const int32_t* H,
                                       const int32_t* W, int B, int feature, float* tokens,
                                       pace_stream_t stream);

/* Scratch bytes for pace_apc_density_pixel (host H, W [B]). */
PACE_API size_t pace_apc_density_pixel_workspace_size(int B, const int32_t* H, const int32_t* W);

/*
 * APC (Sec. 3.2, Eq. 1-6, r and the target size) with a pixel-statistic preview in place of
 * T_v: the feature tokens above, l2-normalised, through the same statistics and tail as
 * pace_apc_density.  Arguments as for pace_apc_density plus `feature`; ws holds the tokens.
 */
PACE_API pace_status_t pace_apc_density_pixel(const uint8_t* img, const int64_t* img_off, const int32_t* H,
                                      const int32_t* W, int B, int feature, const pace_apc_params* params,
                                      float* d_out, pace_apc_stats* stats, void* ws, size_t ws_bytes,
                                      pace_stream_t stream);

/*
 * APC resize (Sec. 3.2 "Adaptive Condensation"; App. B.3: width and height scaled by
 * sqrt(r), bicubic).  Separable cubic convolution (a = -0.5) with centre-aligned
 * sampling, support widened by the downscale factor (antialias), the window clipped
 * at the border and renormalised; fp32 weights, round half to even, clamp to [0,255].
 * The target size (h_out, w_out) of image b is read from stats[b] on the device, so no
 * host synchronisation is needed between density and resize.
 *
 *  src, src_off, H, W  as for pace_apc_density
 *  stats    device  pace_apc_stats [B] from pace_apc_density (h_out <= H, w_out <= W)
 *  dst      device  uint8; image b is written as h_out x w_out x 3 at byte dst_off[b];
 *                   the caller reserves H*W*3 bytes there (the largest possible size)
 *  dst_off  host    int64 [B]
 */
PACE_API pace_status_t pace_apc_resample(const uint8_t* src, const int64_t* src_off, const int32_t* H, const int32_t* W,
                                const pace_apc_stats* stats, uint8_t* dst, const int64_t* dst_off, int B,
                                pace_stream_t stream);

/* Same resize to explicit host-given sizes H_out[b] x W_out[b] (1 <= H_out <= H, 1 <= W_out <= W). */
PACE_API pace_status_t pace_apc_resample_to(const uint8_t* src, const int64_t* src_off, const int32_t* H, const int32_t* W,
                                   const int32_t* H_out, const int32_t* W_out, uint8_t* dst,
                                   const int64_t* dst_off, int B, pace_stream_t stream);

/* ==============================================================================
 * Extract — Dynamic Dual-Attention Extractor (DDAE), Sec. 3.3, Eq. 7; App. B.3.
 * ============================================================================== */

/* Scratch bytes for pace_vit_attn_importance (host cu_seqlens [B+1]). */
PACE_API size_t pace_vit_attn_importance_workspace_size(int B, const int32_t* cu_seqlens, int n_heads);

/*
 * S_vis: attention each patch receives in a full-attention ViT layer (Sec. 3.3; App. B.3,
 * final ViT block).  For image b (rows cu_seqlens[b] .. cu_seqlens[b+1]) and head h:
 * a_j = sum_h sum_i softmax_j(scale q_ih . k_jh), softmax over all patches of the image,
 * then s_vis_raw[m] = sum of a_j over the `merge` consecutive patches of merged token m.
 * Computed flash-style in two passes (row log-sum-exp, then column sums of
 * exp(s - lse)) on tcgen05 tensor cores; the N x N matrix is never stored.
 *
 *  Q, K        device  bf16 [total, n_heads, head_dim], row-major (head_dim contiguous)
 *  cu_seqlens  host    int32 [B+1], cu_seqlens[0] = 0, nondecreasing; every image
 *                      non-empty with a length and start divisible by `merge`
 *  head_dim    64, 80 or 128;  merge 1, 2 or 4
 *  s_vis_raw   device  float [total / merge]
 *  ws          device  >= pace_vit_attn_importance_workspace_size(...) bytes, 16-B aligned
 */
PACE_API pace_status_t pace_vit_attn_importance(const void* Q, const void* K, const int32_t* cu_seqlens, int B,
                                       int n_heads, int head_dim, float scale, int merge, float* s_vis_raw,
                                       void* ws, size_t ws_bytes, pace_stream_t stream);

/*
 * pace_vit_attn_importance with the row log-sum-exp pass split by query rows, so that it can
 * start while Q is still being copied in: the pass-1 work whose query rows all lie below
 * chunk_end_rows[c] (and whose last row is not below chunk_end_rows[c - 1]) is launched after
 * the stream waits for the CUDA event chunk_ready[c].  Results are bit-identical to
 * pace_vit_attn_importance.  K must be complete when chunk_ready[0] fires.
 *
 *  n_chunks        1 .. 64
 *  chunk_end_rows  host  int64 [n_chunks], nondecreasing global Q rows, the last = cu_seqlens[B]
 *  chunk_ready     host  cudaEvent_t [n_chunks] (passed as void*), recorded by the caller; the
 *                  call only enqueues waits on them, so the caller may release them afterwards
 *  other arguments as for pace_vit_attn_importance
 *  Invalid chunks (n_chunks out of range, a null event, decreasing ends, a last end other than
 *  cu_seqlens[B]): PACE_ERR_INVALID_ARG; anything pace_vit_attn_importance rejects: its status.
 *  Either way before any launch or wait is enqueued.
 */
PACE_API pace_status_t pace_vit_attn_importance_chunked(const void* Q, const void* K, const int32_t* cu_seqlens,
                                               int B, int n_heads, int head_dim, float scale, int merge,
                                               float* s_vis_raw, void* ws, size_t ws_bytes, int n_chunks,
                                               const int64_t* chunk_end_rows, void* const* chunk_ready,
                                               pace_stream_t stream);

/* Scratch bytes for pace_llm_text_visual_importance (host cu_q, cu_k [B+1]). */
PACE_API size_t pace_llm_text_visual_importance_workspace_size(int B, const int32_t* cu_q, const int32_t* cu_k,
                                                      int n_q_heads, int n_kv_heads);

/*
 * S_llm: attention from text query tokens to visual tokens in an LLM prefill layer with
 * grouped-query attention (Sec. 3.3; App. B.3, layer L_ext = 2).  For image b, query head
 * h and its KV head g = h / (n_q_heads / n_kv_heads):
 * u_j = sum_h sum_t softmax_j(scale q_th . k_jg), softmax over the image's visual keys.
 *
 *  Q           device  bf16 [sum Tq, n_q_heads, head_dim]
 *  K           device  bf16 [sum Nv, n_kv_heads, head_dim]
 *  cu_q, cu_k  host    int32 [B+1] prefix sums of Tq_b >= 1 and Nv_b >= 1
 *  n_q_heads % n_kv_heads == 0;  head_dim 64, 80 or 128
 *  s_llm_raw   device  float [sum Nv]
 */
PACE_API pace_status_t pace_llm_text_visual_importance(const void* Q, const void* K, const int32_t* cu_q,
                                              const int32_t* cu_k, int B, int n_q_heads, int n_kv_heads,
                                              int head_dim, float scale, float* s_llm_raw, void* ws,
                                              size_t ws_bytes, pace_stream_t stream);

/* Query sets of the full-sequence S_llm (App. "Impact of Attention Token Sources"): every
 * position from the first visual token on (Vision + Text, the paper's default), the text
 * positions after the visual span, or the last position only. */
typedef enum pace_query_set {
  PACE_QUERY_VISION_TEXT = 0,
  PACE_QUERY_TEXT = 1,
  PACE_QUERY_LAST = 2
} pace_query_set;

/* Scratch bytes for pace_llm_sequence_importance (host arrays as there); 0 if they are invalid. */
PACE_API size_t pace_llm_sequence_importance_workspace_size(int B, const int32_t* cu_seq, const int32_t* vis_start,
                                                  const int32_t* n_vis, int n_q_heads, int n_kv_heads,
                                                  int query_set);

/*
 * Full-sequence S_llm (Sec. 3.3; App. B.3, layer L_ext = 2; App. "Impact of Attention Token
 * Sources").  Sequence b is positions 0 .. S_b - 1 of a causal LLM prefill (system, visual
 * and text tokens), its visual tokens at positions v_b .. v_b + N_b - 1.  For query head h
 * (KV head g = h / (n_q_heads / n_kv_heads)) and query position q in the query set P_b:
 * u_j = sum_h sum_{q in P_b} softmax_{k <= q}(scale q_qh . k_kg)[v_b + j],
 * the softmax over every position up to q.  P_b = {v_b .. S_b - 1} (VISION_TEXT),
 * {v_b + N_b .. S_b - 1} (TEXT; empty when the visual span ends the sequence, giving zeros)
 * or {S_b - 1} (LAST).
 *
 *  Q           device  bf16 [sum S, n_q_heads, head_dim]  (queries of every position)
 *  K           device  bf16 [sum S, n_kv_heads, head_dim]
 *  cu_seq      host    int32 [B+1] prefix sums of S_b >= 1
 *  vis_start   host    int32 [B]   v_b >= 0
 *  n_vis       host    int32 [B]   N_b >= 1, v_b + N_b <= S_b
 *  query_set   pace_query_set
 *  s_llm_raw   device  float [sum N_b]
 *  sum S + 128 B <= 2^30.  Invalid arguments: PACE_ERR_INVALID_ARG before any launch.
 */
PACE_API pace_status_t pace_llm_sequence_importance(const void* Q, const void* K, const int32_t* cu_seq,
                                          const int32_t* vis_start, const int32_t* n_vis, int B,
                                          int n_q_heads, int n_kv_heads, int head_dim, float scale,
                                          int query_set, float* s_llm_raw, void* ws, size_t ws_bytes,
                                          pace_stream_t stream);

/* Fusion of the two maps.  ADAPTIVE is Eq. 7; the other three are the fusion ablations of
 * Sec. 4 ("Effect of Attention Fusion in DDAE"): Only LLM-Attn (alpha_w = 1, beta_w = 0), Only
 * ViT-Attn (alpha_w = 0, beta_w = 1) and Fixed Fusion (0.5 / 0.5). */
typedef enum pace_ddae_fusion {
  PACE_DDAE_ADAPTIVE = 0,
  PACE_DDAE_ONLY_LLM = 1,
  PACE_DDAE_ONLY_VIT = 2,
  PACE_DDAE_FIXED = 3
} pace_ddae_fusion;

typedef struct pace_ddae_params {
  float tau;   /* temperature of Eq. 7; 0.5 */
  int32_t fusion; /* pace_ddae_fusion; PACE_DDAE_ADAPTIVE */
} pace_ddae_params;

/* Fills the paper's defaults: tau = 0.5, adaptive fusion.  (The static-resolution baselines
 * of Sec. 4 "Adaptive Resolution vs. Static Resolution" need no mode: pace_apc_params with
 * r_min = r_max = the fixed ratio.) */
PACE_API void pace_ddae_params_default(pace_ddae_params* params);

/* Token budget K = floor(frac * n_vis + 0.5), clamped to [0, n_vis]. */
PACE_API int32_t pace_budget(int32_t n_vis, double frac);

/*
 * DDAE fusion and top-K (Sec. 3.3, Eq. 7).  Per image b: S_llm, S_vis = min-max
 * normalised maps (a constant map becomes 0); sigma = population standard deviation;
 * [alpha_w, beta_w] = softmax([sigma_llm, sigma_vis] / tau) (or the fixed weights of the
 * params' fusion mode);
 * S_final = alpha_w S_llm + beta_w S_vis; keep the K_b = cu_keep[b+1] - cu_keep[b]
 * highest S_final (ties: lower index first), written in ascending index order.
 * One CTA per map; maps of up to 12288 tokens keep their scores in registers, larger ones
 * (any size) read them again for each pass, with identical results.
 * Raw scores must be finite: a NaN or infinite raw score records PACE_ERR_INVALID_ARG (kernel
 * id 9) in the device status word.  The map's S_final and weights are then not meaningful
 * (the value reaches the normalisation and the Eq. 7 weights), but kept still receives K_b
 * distinct indices of the map in ascending order: a NaN fused score ranks below every other
 * score, ties going to the lower index.
 *
 *  s_llm_raw, s_vis_raw  device  float [sum Nv]
 *  cu_v      host    int32 [B+1]; Nv_b >= 1
 *  cu_keep   host    int32 [B+1]; 0 <= K_b <= Nv_b
 *  params    host    NULL for tau = 0.5
 *  s_final   device  float [sum Nv] (may be NULL)
 *  weights   device  float [B, 2] = (alpha_w, beta_w) (may be NULL)
 *  kept      device  int32 [sum K]: global rows cu_v[b] + i of the kept tokens
 */
PACE_API pace_status_t pace_ddae_select(const float* s_llm_raw, const float* s_vis_raw, const int32_t* cu_v,
                               const int32_t* cu_keep, int B, const pace_ddae_params* params, float* s_final,
                               float* weights, int32_t* kept, pace_stream_t stream);

/*
 * Gather of the kept rows, the pruned LLM context (Sec. 3.3; App. C): dst[r] = src[idx[r]],
 * row_bytes bytes per row, byte-exact.  An index outside [0, n_src_rows) writes a zero row
 * and records PACE_ERR_INVALID_ARG in the device status word.
 *
 *  src  device  [n_src_rows, row_bytes];  idx device int32 [n_idx];  dst device [n_idx, row_bytes]
 */
PACE_API pace_status_t pace_gather(const void* src, int64_t n_src_rows, int64_t row_bytes, const int32_t* idx,
                          int64_t n_idx, void* dst, pace_stream_t stream);

/*
 * Token budget relative to Vanilla (App. C, "B = p1 p2"): K = floor(frac * n_vis_vanilla + 0.5)
 * (the count the uncondensed image would have), capped at the n_vis_condensed tokens that
 * remain after APC.  frac is the final ratio B; pace_budget is the same rule on one count.
 */
PACE_API int32_t pace_budget_vanilla(int32_t n_vis_vanilla, int32_t n_vis_condensed, double frac);

/*
 * Row list of the pruned LLM sequences (Sec. 3.3: the kept tokens "formulate the final LLM
 * context sequence"; App. C: S_post = T + N_keep).  Sequence b occupies rows
 * cu_seq[b] .. cu_seq[b+1]-1 of a packed pre-prune batch and holds its image's visual tokens
 * at rows vis_start[b] .. vis_start[b] + n_vis_b - 1 of the sequence.  Its output keeps every
 * position outside the visual span and the visual positions of its kept tokens, in sequence
 * order, as global pre-prune row numbers:
 *   out rows of sequence b start at sum_{c<b} (n_pre_c - n_vis_c + K_c).
 * The list feeds pace_gather_multi (hidden states, KV-cache rows, position ids).  A kept
 * entry outside image b's tokens writes -1 and records PACE_ERR_INVALID_ARG on the device.
 *
 *  cu_seq     host    int32 [B+1] pre-prune sequence prefix
 *  vis_start  host    int32 [B] start of the visual span within each sequence
 *  cu_vis     host    int32 [B+1] visual tokens per image (as passed to pace_ddae_select)
 *  cu_keep    host    int32 [B+1] kept tokens per image (as passed to pace_ddae_select)
 *  kept       device  int32 [cu_keep[B]] pace_ddae_select's kept list (global visual index,
 *                     ascending within each image)
 *  out_idx    device  int32 [sum_b n_pre_b - n_vis_b + K_b]
 */
PACE_API pace_status_t pace_prune_index(int B, const int32_t* cu_seq, const int32_t* vis_start,
                                        const int32_t* cu_vis, const int32_t* cu_keep, const int32_t* kept,
                                        int32_t* out_idx, pace_stream_t stream);

/* One tensor of pace_gather_multi: n_slabs independent slabs (e.g. layer x KV head) of rows;
 * output row r of slab s copies row_bytes from src row idx[r] of the same slab.  All strides
 * in bytes.  16-byte copies are used when every pointer, stride and row_bytes allows. */
typedef struct pace_gather_tensor {
  const void* src;
  void* dst;
  int64_t row_bytes;
  int64_t src_row_stride;   /* >= row_bytes */
  int64_t dst_row_stride;   /* >= row_bytes */
  int64_t n_slabs;
  int64_t src_slab_stride;
  int64_t dst_slab_stride;
  int64_t n_src_rows;       /* rows per source slab; an index outside [0, n_src_rows) writes a zero
                               row and records PACE_ERR_INVALID_ARG on the device */
} pace_gather_tensor;

#define PACE_GATHER_MAX_TENSORS 16

/*
 * The prune step's gathers in one launch (App. C): every tensor gathered with the same row
 * list idx (device int32 [n_idx]); tensors host [n_tensors] descriptors, n_tensors <= 16.
 * Byte-exact.
 */
PACE_API pace_status_t pace_gather_multi(const pace_gather_tensor* tensors, int n_tensors, const int32_t* idx,
                                         int64_t n_idx, pace_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* PACE_H_ */
