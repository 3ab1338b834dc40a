/*
 * apack.h -- C ABI of the A-PACK inner-LLM prune step on NVIDIA GB300 (sm_103a).
 *
 * A-PACK (Sec. 3.2, "Inner-LLM Query-Aware Compression"; Algorithm 1, the
 * inner-LLM loop) prunes multimodal tokens inside the decoder: at a pruning
 * layer it scores every cached audio and visual token by the attention it
 * receives from the text query (Eq. inner_score), keeps the top fraction of
 * them (Eq. inner) and drops the rest together with their key-value entries,
 * so that later layers and decoding see a shorter sequence.
 *
 * Conventions shared by every entry point:
 *  - Pointers are DEVICE memory unless the name ends in _h (HOST memory).
 *  - The caller owns every buffer.  The library allocates nothing, keeps no
 *    per-call state, never synchronises inside a step and never traps: every
 *    call returns an apack_status.  All device work is enqueued on `stream`
 *    (a cudaStream_t passed as void*; NULL = legacy default stream).
 *  - bf16 data are passed as untyped pointers to 16-bit storage.
 *  - A packed (ragged) batch of B sequences stores token t of sequence b at
 *    row cu_seqlens[b] + t of every per-token array.
 *  - Arguments are checked on the host before anything is enqueued
 *    (APACK_EINVAL).  Problems only the device can see (modality counts that
 *    disagree with the host counts, a bounded wait that gave up) are written
 *    to an error word in the workspace and read with apack_device_error().
 *  - Calls that share a workspace must be ordered (same stream, or joined).
 */
#ifndef APACK_H
#define APACK_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef int32_t apack_status;
enum {
  APACK_OK = 0,
  APACK_EINVAL = 1,        /* bad argument (null, size, alignment, shape, ratio) */
  APACK_ECUDA = 2,         /* a CUDA runtime or driver call failed */
  APACK_EWORKSPACE = 3,    /* workspace too small (see apack_workspace_size) */
  APACK_ETIMEOUT = 4,      /* device error word: a bounded wait gave up */
  APACK_EDEVICE = 5,       /* device error word: device data disagree with host counts */
  APACK_EUNSUPPORTED = 6   /* shape outside what this build supports (e.g. head_dim != 128) */
};

/* Per-token modality codes.  S, the set of prunable "cached multimodal
   tokens" of Sec. 3.2, is every token coded AUDIO or VISUAL; OTHER tokens
   (system prompt, text, the query itself) are never scored or dropped. */
enum { APACK_MOD_OTHER = 0, APACK_MOD_AUDIO = 1, APACK_MOD_VISUAL = 2 };

/* Selection segments.  PER_MODALITY takes the top-k separately for the audio
   and the visual tokens of each sequence (two keep counts per sequence);
   JOINT takes one top-k over all of S, the literal form of Eq. inner. */
enum { APACK_SELECT_PER_MODALITY = 0, APACK_SELECT_JOINT = 1 };

/* Softmax domain of the relevance scores (apack_seqs.softmax_domain).
   MM: Eq. inner_score as printed, the denominator runs over the cached
   multimodal tokens S of the sequence only.
   CAUSAL_ROW: the denominator is the decoder's own attention row, every token
   the query row attends to causally (system, text, audio, visual and the
   query tokens up to and including its own position); query row r sits at
   position q_start + r of its sequence (apack_seqs.q_start_h; by default the
   query rows are the last n_q tokens, q_start = len - n_q), and a token of S
   that a row cannot see contributes 0 for that row. */
enum { APACK_SOFTMAX_MM = 0, APACK_SOFTMAX_CAUSAL_ROW = 1 };

/* Maximum sizes of this build. */
#define APACK_HEAD_DIM 128
#define APACK_MAX_SEQS 4096

/* The packed batch entering a pruning layer. */
typedef struct apack_seqs {
  int32_t num_seqs;             /* B, 1 .. APACK_MAX_SEQS */
  const int32_t *cu_seqlens_h;  /* [B+1] token offsets, cu_seqlens_h[0] == 0, non-decreasing */
  const int32_t *cu_qlens_h;    /* [B+1] offsets of each sequence's query rows in the packed Q */
  const int32_t *n_audio_h;     /* [B] audio tokens per sequence (verified on the device) */
  const int32_t *n_visual_h;    /* [B] visual tokens per sequence (verified on the device);
                                   with APACK_SELECT_JOINT only n_audio_h + n_visual_h = |S| is
                                   used, so a caller that knows only |S| may pass (|S|, 0) */
  const uint8_t *modality;      /* [T] APACK_MOD_* per token, T = cu_seqlens_h[B] */
  int32_t num_q_heads;          /* Hq */
  int32_t num_kv_heads;         /* Hkv; Hq % Hkv == 0, query head h reads key head h / (Hq/Hkv) */
  int32_t head_dim;             /* D; must be APACK_HEAD_DIM */
  int32_t softmax_domain;       /* APACK_SOFTMAX_MM (0, zero-initialised default) or
                                   APACK_SOFTMAX_CAUSAL_ROW (needs n_q <= len per sequence) */
  const int32_t *q_start_h;     /* [B] or NULL: position of each sequence's first query row
                                   within the sequence (the query span of Sec. 3.2's problem
                                   statement), 0 <= q_start, q_start + n_q <= len; NULL means
                                   the span ends the sequence.  Read in the CAUSAL_ROW domain
                                   only (in the MM domain no query token is in S). */
} apack_seqs;

/* One group of per-token planes to compact (e.g. the K cache of layers l..L-1).
   Plane p, token row t lives at  base + p*plane_stride + t*row_stride.
   Rows of >= 16 bytes whose addresses and strides are 16-byte aligned take
   the vectorised path; any other row size is copied with narrower accesses.
   src and dst must not overlap unless src == dst with equal strides (in place). */
typedef struct apack_plane {
  const void *src;
  void *dst;
  int64_t src_plane_stride;     /* bytes between planes of src */
  int64_t dst_plane_stride;     /* bytes between planes of dst */
  int64_t src_row_stride;       /* bytes between token rows of src */
  int64_t dst_row_stride;       /* bytes between token rows of dst */
  int64_t row_bytes;            /* bytes copied per token row */
  int32_t num_planes;
  int32_t reserved;
} apack_plane;

/* Bytes of device workspace the calls below need for this batch (256-byte
   aligned start required).  Depends on B, the query rows and head counts. */
apack_status apack_workspace_size(const apack_seqs *seqs, size_t *bytes);

/* Keep counts of Eq. inner, ceil((1-P)|S|), from keep ratios r = 1-P.
   keep_ratio_h: [B][2] (audio, visual) in [0, 1]; with APACK_SELECT_JOINT
   only [b][0] is used and applies to |S| = n_audio + n_visual.
   The ratio is read on a 1e-6 grid: k = min(n, ceil(round(r*1e6) * n / 1e6))
   in integer arithmetic, so that 0.55 * 100 keeps 55, not 56.
   Outputs (host): keep_count_h [B][2] (JOINT: [b][1] = 0) and
   new_cu_seqlens_h [B+1], the packed offsets after the step. */
apack_status apack_keep_counts(const apack_seqs *seqs, const float *keep_ratio_h, int32_t select_mode,
                               int32_t *keep_count_h, int32_t *new_cu_seqlens_h);

/* Relevance scores of Eq. inner_score (Sec. 3.2), averaged over all Hq query
   heads and all query rows of each sequence:
     I_i = 1/(Hq * n_q) * sum_h sum_r  exp(q_{r,h}.k_{i,g(h)} / sqrt(D))
                                      / sum_{j in S} exp(q_{r,h}.k_{j,g(h)} / sqrt(D))
   for i in S of the sequence, and I_i = 0 for tokens outside S.  With
   seqs->softmax_domain = APACK_SOFTMAX_CAUSAL_ROW the sum in the denominator
   runs over every token j <= p_r (p_r = q_start + r, the row's position within
   its sequence; q_start = len - n_q without seqs->q_start_h) and row r adds to
   I_i only when i <= p_r.
   q: bf16 [sum n_q][Hq][D], contiguous (the query rows at the pruning layer).
   k: bf16 keys of the pruning layer, token t at k + t*k_token_stride, laid
      out [Hkv][D] within the row; k_token_stride a multiple of 16 bytes.
   scores: fp32 [T].  Computed in fp32 from bf16 products on the tensor
   cores; deterministic (fixed reduction order, no atomics).  q and k must be
   device memory (they are read by TMA; host memory gives APACK_EINVAL). */
apack_status apack_score(const apack_seqs *seqs, const void *q, const void *k, int64_t k_token_stride,
                         float *scores, void *ws, size_t ws_bytes, void *stream);

/* Top-k selection of Eq. inner per segment (see APACK_SELECT_*): keeps the
   keep_count_h[b][m] highest scores of each segment, equal scores going to the
   lower token index, plus every token outside S.
   keep_count_h: host [B][2] counts (JOINT: [b][0] over |S|), or NULL: the
   counts come from keep_ratio_h (host [B][2], the keep ratios 1-P of Eq. inner)
   by the rule of apack_keep_counts.
   Outputs: keep_idx [T_out] (kept token indices in ascending order, i.e. the
   original order; T_out = new_cu_seqlens_h[B] of apack_keep_counts),
   modality_out [T_out] (nullable; the compacted modality mask),
   dst_of_src [T] (nullable; output row of each token or -1),
   new_cu_seqlens [B+1] (nullable; device copy of the new offsets).
   scores must be finite and >= 0 (as apack_score produces). */
apack_status apack_select(const apack_seqs *seqs, const float *scores, const float *keep_ratio_h,
                          const int32_t *keep_count_h, int32_t select_mode, int32_t *keep_idx,
                          uint8_t *modality_out, int32_t *dst_of_src, int32_t *new_cu_seqlens, void *ws,
                          size_t ws_bytes, void *stream);

/* KV-cache and hidden-state slicing (Sec. 3.2, last sentence; Algorithm 1,
   "slice their KV-cache entries"): for every plane of every group,
   dst row j = src row keep_idx[j], j < n_out, bit for bit.
   planes_h: host array of num_groups descriptors.
   In place: a group with src == dst (and equal plane and row strides) is
   compacted within its own buffer.  Output row j reads row keep_idx[j] >= j,
   so each store waits (bounded) until every load that reads the rows it
   overwrites is done; the rows must be 16-byte multiples of at most 32 KB,
   16-byte aligned (APACK_EUNSUPPORTED otherwise), planes must not overlap,
   and ws is required: the launch keeps its progress words or wave counter
   in bytes 256..1023 (the workspace of apack_workspace_size has them).
   Host source: a group whose src is pinned host memory (cudaHostAlloc or
   cudaHostRegister) is gathered over the host link by plain loads (zero
   copy): only the kept rows cross the link.  Its dst must be device memory,
   and it cannot be in place (APACK_EINVAL).
   ws: NULL (out of place only), or a 256-byte aligned workspace (e.g. the
   one of apack_score, at least 1024 bytes) whose error word receives
   APACK_ETIMEOUT if a bounded wait gives up. */
apack_status apack_compact(const int32_t *keep_idx, int64_t n_out, const apack_plane *planes_h,
                           int32_t num_groups, void *ws, void *stream);

/* One pruning step at layer `layer` of a num_layers-layer decoder
   (Algorithm 1, one iteration of the inner-LLM loop): apack_score on the
   layer's keys, apack_select, then compaction of the K and V caches of
   layers [layer, num_layers), of the hidden states and of any extra planes.
   k_cache / v_cache: bf16, slab 0 = layer `layer`, slab i at
     + i*kv_layer_stride bytes, token t at + t*Hkv*D*2 bytes within a slab.
   k_out / v_out: the same layout with kv_out_layer_stride; k_out == k_cache
     and v_out == v_cache with equal strides compact in place (the first T_out
     token rows of every slab, see apack_compact).
   hidden / hidden_out: bf16 [T][hidden_dim] / [T_out][hidden_dim] (hidden may be NULL;
     hidden_out == hidden compacts in place).
   keep_count_h: [B][2] counts (e.g. cumulative schedules); when NULL they
   come from keep_ratio_h as in apack_keep_counts.
   new_cu_seqlens_h (host, [B+1]) receives the new offsets before the call
   returns (no device synchronisation needed).
   scores (device [T] fp32) receives the relevance scores.
   stage_events_h: NULL, or 4 cudaEvent_t recorded on `stream` before
   scoring, before selection, before compaction and at the end.
   Every argument, the compaction groups included, is checked before the
   first launch: a status other than APACK_OK and APACK_ECUDA means nothing
   was queued on `stream`. */
apack_status apack_prune_step(const apack_seqs *seqs, int32_t layer, int32_t num_layers,
                              const void *q, const void *k_cache, const void *v_cache,
                              int64_t kv_layer_stride, const void *hidden, int64_t hidden_dim,
                              const float *keep_ratio_h, const int32_t *keep_count_h, int32_t select_mode,
                              void *k_out, void *v_out, int64_t kv_out_layer_stride, void *hidden_out,
                              const apack_plane *extra_planes_h, int32_t num_extra,
                              uint8_t *modality_out, int32_t *keep_idx, int32_t *new_cu_seqlens_h,
                              int32_t *new_cu_seqlens, float *scores, void *ws, size_t ws_bytes,
                              void *const *stage_events_h, void *stream);

/* apack_score for callers that cannot allocate device memory: plugins inside
   an engine that owns every device allocation, and serving processes that fix
   their device memory at start-up.  The paper has no counterpart; it is a
   deployment variant of apack_score.
   Same arguments, checks and results as apack_score (q and k must be device
   memory: host memory is refused with APACK_EINVAL before any device work),
   without the workspace: the
   scratch is one 8 MiB array that the library keeps on every device it is
   loaded on, until the process exits.  Batches whose apack_workspace_size
   exceeds 8 MiB return APACK_EWORKSPACE (a single 7B-shaped sequence with
   135k tokens and 256 query rows needs about 5.6 MiB).  Nothing is allocated.
   The first call on a device looks the array's address up (a CUDA runtime
   call); make that first call before any stream capture on that device.
   All calls share the one array and it keeps the last call's contents: calls
   that can overlap on the GPU (other streams, other threads) race on it and
   must be serialised by the caller.
   device_error_out: NULL, or a device int32 that receives the call's device
   error code (APACK_OK, APACK_ETIMEOUT, APACK_EDEVICE) on `stream`. */
apack_status apack_score_static(const apack_seqs *seqs, const void *q, const void *k, int64_t k_token_stride,
                                float *scores, int32_t *device_error_out, void *stream);

/* Pre-LLM frame alignment (Sec. 3.1, "Coarse pass" and "Gated fine pass";
   Eq. cka and Eq. gate; Algorithm 1, its first pre-LLM steps).  Per video frame f:
     v_f = mean of the frame's visual tokens; a_f = mean of the audio tokens
           resampled onto the frame axis (audio token j belongs to frame
           floor(j * n_frames / n_audio));
     c_f = ||V_f^T A_f||_F^2 / (||A_f^T A_f||_F ||V_f^T V_f||_F), linear CKA of the
           mean-centred window rows f - window/2 .. f + window/2 (cut to the clip;
           0 for a window whose centred rows vanish);
     s_f = c_f if mean(c) >= tau, else (1 - beta) c_f + beta (1 - dn_f), with
           dn_f = the min-max normalised ||v_f - a_f|| over the clip.
   visual: bf16 [n_frames * tokens_per_frame][dim], frame f's tokens at rows
   f*tokens_per_frame ..; audio: bf16 [n_audio][dim]; dim a multiple of 8,
   n_audio >= n_frames >= 1, window odd in 1..7 (the paper uses 3, tau = 0.78,
   beta = 0.90).  Outputs (device, fp32): c_out [F], s_out [F], dnorm_out [F]
   (nullable), cbar_out [1] (nullable).  fp32 accumulation, fixed reduction
   order (deterministic).  ws: 256-byte aligned, apack_frame_alignment_workspace_size. */
apack_status apack_frame_alignment_workspace_size(int32_t n_frames, int64_t dim, size_t *bytes);
apack_status apack_frame_alignment(const void *visual, const void *audio, int32_t n_frames,
                                   int32_t tokens_per_frame, int32_t n_audio, int64_t dim, int32_t window,
                                   float tau, float beta, float *c_out, float *s_out, float *dnorm_out,
                                   float *cbar_out, void *ws, size_t ws_bytes, void *stream);

/* ---- A whole progressive schedule in one call.
   Sec. 3.2: pruning is repeated at later layers, each step keeping a fraction of
   the current tokens (Algorithm 1, the inner-LLM loop).  Step i does what
   apack_prune_step does at layer steps_h[i].layer; its inputs are step i-1's
   outputs (K/V from k_out/v_out at layer offset l_i - l_(i-1), hidden_out,
   modality_out, new_cu_seqlens_h, and the counts kept as the new audio/visual
   counts; (|S|, 0) in joint mode).  Layers are strictly ascending.  Each step
   needs its own keep_idx; outputs of step i+1 may reuse step i-1's buffers
   (ping-pong).  All steps (queries and compaction groups included) are
   checked on the host before the first launch;
   then everything runs in order on `stream` (bit-identical to one
   apack_prune_step per step).  stage_events_h: NULL or 4*num_steps events
   (entries may be NULL), recorded for step i before scoring [4i], after
   scoring [4i+1], after selection [4i+2] and after compaction [4i+3].  ws must
   hold apack_workspace_size of every step's sequences. */
typedef struct apack_step {
  int32_t layer;                   /* pruning layer l_i */
  const void *q;                   /* bf16 [sum n_q][Hq][128]: query rows of layer l_i */
  const int32_t *keep_count_h;     /* host [B][2] kept tokens after the step, or NULL */
  const float *keep_ratio_h;       /* host [B][2] keep ratios, used when keep_count_h is NULL */
  void *k_out, *v_out;             /* bf16 [L - l_i][T_i][Hkv][128] */
  int64_t kv_out_layer_stride;     /* bytes between layers of k_out / v_out */
  void *hidden_out;                /* bf16 [T_i][hidden_dim]; required when hidden is given */
  const apack_plane *extra_planes_h; /* further per-token planes of this step, or NULL */
  int32_t num_extra;
  uint8_t *modality_out;           /* [T_i] */
  int32_t *keep_idx;               /* [T_i] */
  int32_t *new_cu_seqlens_h;       /* host [B+1], written by the call */
  int32_t *new_cu_seqlens;         /* device [B+1] or NULL */
} apack_step;

apack_status apack_prune_schedule(const apack_seqs *seqs, int32_t num_layers, const void *k_cache,
                                  const void *v_cache, int64_t kv_layer_stride, const void *hidden,
                                  int64_t hidden_dim, int32_t select_mode, const apack_step *steps_h,
                                  int32_t num_steps, float *scores, void *ws, size_t ws_bytes,
                                  void *const *stage_events_h, void *stream);

/* ---- The schedule as a CUDA graph.
   apack_prune_schedule_graph makes the same checks and host planning as
   apack_prune_schedule (same arguments, no stage events) once, and captures its
   launches into an executable CUDA graph; it launches nothing itself.  It
   writes steps_h[i].new_cu_seqlens_h as the direct call does.
   apack_graph_launch replays those launches on `stream`, with the same
   pointers, sizes and keep counts: one graph launch instead of one launch per
   kernel, for a schedule that repeats with fixed shapes (a serving bucket).
   Every device buffer named at capture must stay allocated while the graph is
   used; the host-side arguments are not read again after the capture returns.
   apack_graph_destroy frees the graph.  Errors: the capture's own checks
   (as apack_prune_schedule), APACK_ECUDA if the driver refuses the capture. */
typedef struct apack_graph_s *apack_graph;
apack_status apack_prune_schedule_graph(const apack_seqs *seqs, int32_t num_layers, const void *k_cache,
                                        const void *v_cache, int64_t kv_layer_stride, const void *hidden,
                                        int64_t hidden_dim, int32_t select_mode, const apack_step *steps_h,
                                        int32_t num_steps, float *scores, void *ws, size_t ws_bytes,
                                        apack_graph *graph_out);
apack_status apack_graph_launch(apack_graph graph, void *stream);
apack_status apack_graph_destroy(apack_graph graph);

/* ---- Decode-step attention over a (compacted) KV cache.
   Sec. 3.2 (last sentence) and App. G: pruning shortens the cache that every
   autoregressive decode step attends to.  One decode token per sequence:
     out[b][h][:] = sum_j softmax_j(q[b][h] . k[j][g] / sqrt(128)) v[j][g][:],
   g = h / (Hq / Hkv), j over all cu_seqlens_h[b] .. cu_seqlens_h[b+1]-1
   (every cached token, not only the multimodal ones).
   q: bf16 [num_seqs][Hq][128] (8-byte aligned); k, v: bf16 token rows
   [T][Hkv][128] with kv_token_stride bytes between tokens (16-byte aligned,
   a multiple of 16, >= Hkv*256); out: fp32 [num_seqs][Hq][128] (16-byte
   aligned, device).  cu_seqlens_h: host [num_seqs+1], starting at 0; an
   empty sequence gives zeros.  Supported: Hq / Hkv <= 8 and Hkv in
   {1, 2, 4, 8} (APACK_EUNSUPPORTED otherwise).  fp32 accumulation.  With
   Hkv 2 or 4 and at most 8 query heads per KV head (the tensor-core path) the
   CTAs of a sequence claim its 128-key tiles from a counter as they go, so
   the grouping of keys into partial sums, and with it the last bits of out,
   can differ from call to call; the other head layouts merge in a fixed
   order.  ws: 256-byte aligned, apack_decode_workspace_size bytes (the size
   depends on the device's SM count: query it on the device that runs the
   call), zeroed by the caller once before its first use: its first 16 bytes
   are a device error word read by apack_device_error, and it holds the
   claim counters, which every call leaves at zero.  A device-side wait that
   runs out records APACK_ETIMEOUT there.  Two kernel launches per 64
   sequences; no allocation, no synchronisation. */
apack_status apack_decode_workspace_size(int32_t num_seqs, const int32_t *cu_seqlens_h, int32_t num_q_heads,
                                         int32_t num_kv_heads, size_t *bytes);
apack_status apack_decode_attention(int32_t num_seqs, const int32_t *cu_seqlens_h, const void *q, const void *k,
                                    const void *v, int64_t kv_token_stride, int32_t num_q_heads,
                                    int32_t num_kv_heads, float *out, void *ws, size_t ws_bytes, void *stream);

/* Synchronises `stream`, then reads the device error word of `ws` into
   *code_out (APACK_OK, APACK_ETIMEOUT or APACK_EDEVICE) and clears it when
   `clear` is non-zero. */
apack_status apack_device_error(const void *ws, void *stream, int32_t *code_out, int32_t clear);

/* Number of kernels this library has launched in the calling process. */
uint64_t apack_launch_count(void);

/* Human-readable name of a status code (static string). */
const char *apack_status_string(apack_status status);

#ifdef __cplusplus
}
#endif

#endif /* APACK_H */
