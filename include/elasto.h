/*
 * elasto.h -- C-ABI of libelasto: the runtime forward pass of one Descendant
 * Network (DN) of an elastic ViT or ResNet-50, chosen at run time from one
 * shared set of weights (Elastoformer, Section 4.3 "Elastic Neural Network").
 *
 * A DN ("mode") keeps, per layer, a subset of attention heads and of MLP
 * hidden channels (ViT; Eq. 4 and Eq. 6 with structured 0/1 masks), or per
 * bottleneck block subsets of the two inner conv widths (ResNet-50; Eq. 7).
 * Masking whole rows/columns to zero is computed as deleting them: the library
 * gathers each mode's kept rows/columns into contiguous packed weights once,
 * at create time, so switching modes at run time is a pointer swap with no
 * weight copy (the paper measures its switch cost in Section 6.2).
 *
 * Conventions common to every call:
 *  - Every call returns an elasto_status; on failure a thread-local message is
 *    available from elasto_last_error().
 *  - Pointers named *_host are host memory; all others named device are CUDA
 *    device memory of the current device. The library never keeps a caller
 *    pointer past the call that received it.
 *  - Streams are cudaStream_t passed as void* (NULL = legacy default stream).
 *  - Asynchronous CUDA faults surface at the caller's next synchronisation,
 *    and at the next library call as ELASTO_ERR_CUDA.
 *  - A handle is not thread-safe: the caller serialises calls on one handle.
 */
#ifndef ELASTO_H
#define ELASTO_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct elasto_s* elasto_t; /* opaque, owned by the library */

typedef enum {
  ELASTO_OK = 0,
  ELASTO_ERR_INVALID_ARG = -1, /* null pointer, bad size, bad descriptor */
  ELASTO_ERR_BAD_TABLE = -2,   /* kept-index table not sorted/unique/in range */
  ELASTO_ERR_BAD_MODE = -3,    /* mode index out of range */
  ELASTO_ERR_OOM = -4,         /* device allocation failed */
  ELASTO_ERR_CUDA = -5,        /* CUDA runtime/driver error */
  ELASTO_ERR_UNSUPPORTED = -6, /* shape or device the kernels do not support */
  ELASTO_ERR_TIMEOUT = -7,     /* a device-side wait gave up (status word) */
  ELASTO_ERR_GUARD = -8        /* a guard zone after a device buffer was overwritten */
} elasto_status;

enum { ELASTO_ARCH_VIT = 1, ELASTO_ARCH_RESNET50 = 2 };
enum { ELASTO_F32 = 0, ELASTO_BF16 = 1 };

/* Model description.
 * ViT (Section 4.1, 5.2): img_h = img_w, patch P divides img_h, n = (img_h/P)^2 + 1
 *   tokens, dim d, heads h with d/h = 64, mlp d_ff, layers L, classes C.
 * ResNet-50 v1.5: img_c = 3, classes C; patch/dim/heads/mlp/layers ignored
 *   (bottlenecks [3,4,6,3], widths 64..512 are fixed).
 * weight_dtype: storage type of the weights AND of the images given to
 *   forward (ELASTO_F32 or ELASTO_BF16). ViT weights are stored on the device
 *   as bf16 (fp32 inputs as a bf16 hi + lo pair); ResNet-50 convolution
 *   weights (BN folded) and activations as IEEE f16; biases, LayerNorm
 *   parameters, position embeddings and the classifiers stay fp32.
 * max_batch: largest batch forward accepts; sizes the activation workspace. */
typedef struct {
  int arch;
  int img_h, img_w, img_c;
  int patch, dim, heads, mlp, layers, classes;
  int weight_dtype;
  int max_batch;
} elasto_model_desc;

/* Weights: host pointers to the canonical tensors, PyTorch layouts, each of
 * weight_dtype, in this fixed order.
 * ViT (4 + 12 L + 4 tensors):
 *   patch_w [d,C,P,P], patch_b [d], cls [d], pos [n,d],
 *   per layer: ln1_w [d], ln1_b [d], qkv_w [3d,d], qkv_b [3d], proj_w [d,d],
 *              proj_b [d], ln2_w [d], ln2_b [d], fc1_w [f,d], fc1_b [f],
 *              fc2_w [d,f], fc2_b [d],
 *   norm_w [d], norm_b [d], head_w [C,d], head_b [C].
 *   qkv_w rows: blocks q | k | v of d rows each, head-major inside a block.
 * ResNet-50 (5 + 15 per block + 5 per projection + 2 = 267 tensors):
 *   stem_w [64,3,7,7], stem BN gamma, beta, mean, var [64];
 *   per block: conv1_w [w,cin,1,1], bn1 x4, conv2_w [w,w,3,3], bn2 x4,
 *              conv3_w [4w,w,1,1], bn3 x4, and on the first block of each
 *              stage down_w [4w,cin,1,1], down BN x4;
 *   fc_w [C,2048], fc_b [C]. BN eps = 1e-5, LayerNorm eps = 1e-6. */
typedef struct {
  const void* const* tensors;
  int n_tensors;
} elasto_weights;

/* One mode's kept-index tables: int32, strictly increasing, in range.
 * ViT: heads_kept is the concatenation over layers of each layer's kept head
 *   indices (n_heads_kept[l] entries for layer l, 0 <= n <= h); mlp_kept
 *   likewise for MLP hidden channels (0 <= n_mlp_kept[l] <= d_ff).
 * ViT embedding width (Section 4.1: the compress stage also shrinks the
 *   hidden size of the LayerNorm and patch-embedding layers): embed_kept
 *   lists the n_embed_kept kept residual-stream channels, 1 <= n <= dim, the
 *   same set in every layer; the DN is then the ViT of that width (patch
 *   embedding, class token and position embedding, LayerNorm parameters, b^O
 *   and b2 keep those entries; W^O and W2 those output rows; W_qkv, W1 and the
 *   classifier those input columns; each LayerNorm normalises over the kept
 *   channels). n_embed_kept == 0 (embed_kept may be NULL) keeps all dim
 *   channels. A model with any embedding-pruned mode packs every mode
 *   separately (no prefix sharing).
 * ResNet-50: conv_kept_a / conv_kept_b concatenate, per block, the kept
 *   channels after conv1 (S_a) and after conv2 (S_b), 1 <= n <= width.
 * Unused members may be NULL (and counts 0). */
typedef struct {
  const int32_t* heads_kept;
  const int32_t* n_heads_kept;
  const int32_t* mlp_kept;
  const int32_t* n_mlp_kept;
  const int32_t* conv_kept_a;
  const int32_t* n_conv_a;
  const int32_t* conv_kept_b;
  const int32_t* n_conv_b;
  const int32_t* embed_kept;
  int32_t n_embed_kept;
} elasto_mode_tables;

/* Build an elastic model on the current device: validates descriptor and
 * tables, copies the weights to one library-owned device arena, packs every
 * mode's kept rows/columns (Eq. 4, 6, 7 as deletion; "pruning metadata" of
 * Section 4.1-4.2) and allocates the activation workspace for max_batch.
 * ViT: when every layer's kept head sets and MLP channel sets are nested
 * across the modes (Eq. 8) and every MLP count is a multiple of 8, one packed
 * copy per layer serves all modes: heads and channels are ordered "kept by the
 * smallest mode first", each mode computes on a prefix of that copy (packed
 * memory = the largest mode's, not the sum over modes; ELASTO_Q_PREFIX_SHARED
 * reports it). Results then match the per-mode packing up to the fp32
 * summation order of the out-projection and FC2 reductions. Otherwise each
 * mode gets its own packed copy.
 * Synchronous. Mode 0 is current afterwards. The caller may free all inputs
 * when this returns. Errors: INVALID_ARG, BAD_TABLE, OOM, CUDA, UNSUPPORTED. */
elasto_status elasto_create(const elasto_model_desc* desc, const elasto_weights* weights,
                            const elasto_mode_tables* modes, int n_modes, elasto_t* out);

/* Select the DN used by forwards enqueued after this call (Section 4.4: the
 * runtime picks one DN). Host-only, O(1), no device work, no allocation;
 * forwards already enqueued keep the mode they were enqueued with.
 * Errors: INVALID_ARG (null handle), BAD_MODE. */
elasto_status elasto_set_mode(elasto_t h, int mode);
elasto_status elasto_get_mode(elasto_t h, int* mode);

/* Enqueue the current mode's forward pass on `stream`:
 *   images_device: [batch, img_h, img_w, img_c] NHWC of weight_dtype, device;
 *   logits_device: [batch, classes] fp32, device, written.
 * 1 <= batch <= max_batch. Asynchronous; never synchronises. Buffers are
 * caller-owned. Concurrent forwards on one handle share its workspace and
 * must be ordered on one stream. Errors: INVALID_ARG, CUDA. */
elasto_status elasto_forward(elasto_t h, void* stream, const void* images_device, int batch,
                             float* logits_device);

/* The same forward from host memory: copies images_host to a library-owned
 * device buffer, runs the forward, copies the logits back to logits_host and
 * synchronises `stream` before returning (pinned host memory makes the copies
 * asynchronous with respect to the host until that point). */
elasto_status elasto_forward_host(elasto_t h, void* stream, const void* images_host, int batch,
                                  float* logits_host);

/* A sequence of forwards from host memory with the copies overlapped (the
 * serving loop of Section 4.4's runtime: one DN, batches arriving in host
 * memory). Batch i (batch images, all batches of one size) is read from
 * images_host[i] ([batch, img_h, img_w, img_c] NHWC of weight_dtype) and its
 * logits are written to logits_host[i] ([batch, classes] fp32); the two
 * pointer arrays have n_batches entries. Batch i+1's images are copied to
 * the device on one library stream while batch i's forward runs on `stream`,
 * and batch i's logits come back on another while batch i+1 runs, through
 * two library-owned device staging pairs (the second is allocated by the
 * first call on a handle, as are the two copy streams and their events).
 * Returns when every logit is in host memory. Host buffers must be pinned
 * (cudaHostAlloc / cudaHostRegister) for the copies to overlap; pageable
 * memory works but serialises them. Every batch runs in the mode current at
 * the call (as for elasto_forward, set_mode must not run concurrently).
 * Errors: INVALID_ARG (null pointer, n_batches < 1, batch outside
 * [1, max_batch]), OOM, CUDA. */
elasto_status elasto_forward_host_batches(elasto_t h, void* stream, int n_batches, int batch,
                                          const void* const* images_host, float* const* logits_host);

/* The same forward as elasto_forward (ViT handles), for callers that must not
 * allocate device memory when they run inference: e.g. a process whose
 * memory manager takes the whole GPU into its own pool at start-up and
 * forbids later driver allocations, or a latency-critical loop that cannot
 * absorb the device synchronisation a cudaMalloc/cudaFree may trigger.
 * The paper has no counterpart; this is a deployment convenience.
 * It allocates nothing: no cudaMalloc, no cudaFree, no allocating library
 * routine. All activation scratch lives in one fixed 64 MiB device array
 * inside the library (present on every GPU that loads it, until exit), so
 * the handle's own workspace is not used and batch is limited by that array,
 * not by max_batch: a batch whose scratch does not fit is rejected with
 * ELASTO_ERR_INVALID_ARG and a message giving the limit for the model and
 * current mode (e.g. 18 images for the full ViT-B/16 mode, 238 for the tiny ViT).
 * The current device must be the handle's (else INVALID_ARG). The first call
 * in a CUDA context of a device looks up the array's device address
 * (cudaGetSymbolAddress), and the first call for each (mode, batch) builds
 * its launch plans and keeps them with the handle (host memory); make those
 * first calls before any stream capture. Every call uses the same array and it keeps the last call's
 * contents; each call writes all the scratch it reads, so nothing has to be
 * cleared, but calls that overlap on the GPU (e.g. on two streams) race on
 * it: order them on one stream. Asynchronous like elasto_forward; images and
 * logits are caller-owned device buffers with the same layouts.
 * Errors: INVALID_ARG, UNSUPPORTED (ResNet-50 handles), CUDA. */
elasto_status elasto_forward_noalloc(elasto_t h, void* stream, const void* images_device, int batch,
                                     float* logits_device);

/* Synchronise `stream`, then read and clear the handle's device status word
 * (kernels record ELASTO_ERR_TIMEOUT there instead of hanging). Returns the
 * recorded status or ELASTO_OK. */
elasto_status elasto_sync_status(elasto_t h, void* stream);

/* Out-of-bounds write detection (the paper has no counterpart; a check the
 * tests run in place of a device memory checker). Every buffer of a handle's
 * device arena (packed weights, parameters, activations, staging, status
 * word) is followed by a guard zone of at least 1 KiB, filled with the byte
 * 0xA5 when the arena is allocated, before any create-time kernel runs.
 * elasto_check_guards enqueues a check of every zone on `stream`, waits for
 * it, and returns ELASTO_OK if every guard byte is intact, else
 * ELASTO_ERR_GUARD with the first damaged zone's buffer named in
 * elasto_last_error. n_bad (may be null) receives the number of damaged
 * zones. Errors: INVALID_ARG, CUDA. */
elasto_status elasto_check_guards(elasto_t h, void* stream, int* n_bad);

/* Test-only: overwrite the first byte of guard zone `zone` (0 <= zone <
 * elasto_query(ELASTO_Q_GUARD_ZONES)) with a cudaMemset inside the handle's
 * own allocation, so that a test can see elasto_check_guards report it.
 * Synchronous. Errors: INVALID_ARG, CUDA. */
elasto_status elasto_debug_damage_guard(elasto_t h, int zone);

/* Release everything the handle owns (synchronises the device first). */
elasto_status elasto_destroy(elasto_t h);

/* Message of the last failing call on this thread ("" if none). */
const char* elasto_last_error(void);

/* Introspection: ELASTO_Q_* values. `mode` is used where it applies. */
enum {
  ELASTO_Q_N_MODES = 0,
  ELASTO_Q_PACKED_BYTES = 1,     /* device bytes of packed weights one mode's forward reads */
  ELASTO_Q_SHARED_BYTES = 2,     /* device bytes of mode-independent weights */
  ELASTO_Q_WORKSPACE_BYTES = 3,  /* activation workspace for max_batch */
  ELASTO_Q_ARENA_BYTES = 4,      /* total device bytes owned by the handle */
  ELASTO_Q_MODE_MACS = 5,        /* multiply-accumulates per image of the mode */
  ELASTO_Q_LAUNCHES = 6,         /* kernels one forward of the mode launches kernel by kernel
                                    (a one-image ViT forward launches at most one more: its
                                    out-projection and FC2 run split-K, their partial-sum
                                    launches compute the LayerNorms that follow, and the last
                                    FC2's sum stands alone); a one-image forward with a
                                    one-launch plan (ELASTO_Q_ONE_LAUNCH) launches 1 */
  ELASTO_Q_PACKED_TOTAL = 7,     /* device bytes of all modes' packed weights together */
  ELASTO_Q_PREFIX_SHARED = 8,    /* 1 if the modes share one prefix-ordered packed copy */
  ELASTO_Q_GUARD_ZONES = 9,      /* guard zones in the handle's arena (elasto_check_guards) */
  ELASTO_Q_ONE_LAUNCH = 10       /* 1 if the mode's one-image forwards run as one launch
                                    (elasto_set_one_launch), else 0 */
};
elasto_status elasto_query(elasto_t h, int what, int mode, int64_t* value);

/* One-image forwards as one launch (ViT handles; the paper has no
 * counterpart: Section 6.2 measures DN latency at batch 1, where a forward of
 * ~88 dependent kernels is bound by their launch and ramp-up latencies).
 * With it on (off by default), elasto_forward with batch == 1 runs the whole DN
 * forward (patch rows, patch projection, every layer, final norm and
 * classifier) as the phases of one persistent cooperative kernel with one
 * block per SM, preceded by an 8-byte cudaMemsetAsync of its barrier words:
 * the same operations, the same packed weights and the same handle workspace
 * as the kernel-by-kernel forward; results agree within floating-point
 * reassociation (the LayerNorm sums and the split-K partitions differ), not
 * bit for bit. Plans are made at create time for every mode that fits
 * (bf16-stored weights, at most 256 tokens, embedding width <= 1024);
 * elasto_query(ELASTO_Q_ONE_LAUNCH, mode) says which (0 while it is off).
 * Measured on GB300 it is slower than the kernel-by-kernel forward (ViT-B/16
 * 0.61 against 0.51 ms): each of its ~88 phases pays a grid barrier and the
 * latency of its first loads, as each launch of the chain does, and the chain
 * overlaps a launch's set-up with the previous kernel (programmatic dependent
 * launch); it is kept as an alternative, tested like the default path.
 * Phases are separated by grid-wide barriers whose waits are bounded; a wait
 * that gives up records ELASTO_ERR_TIMEOUT in the status word and the launch
 * ends. Forwards of one handle must not overlap on the GPU (as for every
 * forward: they share its workspace). No effect on ResNet-50 handles.
 * Errors: INVALID_ARG (null handle). */
elasto_status elasto_set_one_launch(elasto_t h, int enable);

/* Per-launch timing (diagnostics). While enabled, forward records a CUDA
 * event pair around every kernel it launches; elasto_profile_read
 * synchronises on the last event and returns, for the most recent forward,
 * one record per launch: what ran, its duration, and its algorithmic work
 * (multiply-accumulates for contractions, bytes that must cross HBM for the
 * memory-bound kernels). Events add a few microseconds per forward. */
enum {
  ELASTO_K_PATCHIFY = 0, ELASTO_K_GEMM = 1, ELASTO_K_LAYERNORM = 2, ELASTO_K_ATTENTION = 3,
  ELASTO_K_HEAD = 4,
  ELASTO_K_IM2COL = 5, /* the CNN stem's input rearrangement (space-to-depth) */
  ELASTO_K_POOL = 6,
  ELASTO_K_ONE_LAUNCH = 7 /* a whole one-image ViT forward in one launch (elasto_set_one_launch) */
};
typedef struct {
  int kind;     /* ELASTO_K_* */
  int layer;    /* transformer layer / conv block, -1 outside */
  int m, n, k;  /* GEMM problem (M x N x K); other kernels: rows, cols, 0 */
  float ms;     /* device duration */
  double macs;  /* algorithmic multiply-accumulates */
  double bytes; /* algorithmic HBM bytes (inputs read once + outputs written) */
} elasto_launch_record;
elasto_status elasto_profile_enable(elasto_t h, int enable);
elasto_status elasto_profile_read(elasto_t h, elasto_launch_record* out, int capacity, int* count);

/* Runtime DN selection (Section 4.4, Eq. 10). One look-up-table entry per
 * mode: latency, memory footprint, computational cost, accuracy. */
typedef struct {
  float latency_ms;    /* forward latency at the profiled batch */
  double memory_bytes; /* device bytes of the weights the mode uses (packed view + shared) */
  double gflops;       /* 2 x multiply-accumulates per forward at the profiled batch, 1e9 */
  float accuracy;      /* the caller's measured accuracy in %, NaN when unknown */
} elasto_dn_profile;

/* Profile every mode of h on this GPU: `trials` timed forwards (after 3
 * warm-up forwards) of `batch` images from the handle's own buffers on
 * `stream`, latency = median of CUDA-event durations; memory and FLOPs from
 * the packed layout. accuracy is set to NaN (the paper measures it offline on
 * a validation set; the caller fills it in). Restores the current mode.
 * Synchronous. out: n_modes entries. 1 <= batch <= max_batch, trials >= 1.
 * Errors: INVALID_ARG, CUDA. */
elasto_status elasto_profile_dns(elasto_t h, void* stream, int batch, int trials, elasto_dn_profile* out);

/* Eq. 10 over a look-up table: among entries with latency_ms <= max_latency_ms,
 * memory_bytes <= max_memory_bytes and accuracy >= min_accuracy, the one with
 * the lowest gflops (ties: lower latency, then lower index). A NaN budget
 * disables that constraint; an entry with NaN accuracy fails any non-NaN
 * min_accuracy. Host-only, no CUDA. Writes the index to *mode.
 * Errors: INVALID_ARG (null, n <= 0), BAD_MODE (no entry satisfies them). */
elasto_status elasto_select_dn(const elasto_dn_profile* lut, int n, float max_latency_ms, double max_memory_bytes,
                               float min_accuracy, int* mode);

/* L1-norm saliency of the Compress stage (Section 4.1: a row's saliency is its
 * average absolute weight; the least salient rows are masked, Eq. 4, 6, 7),
 * at the granularity of the kept tables. Computed on the current device from
 * host weights (same descriptor and tensor order as elasto_create; no mode
 * tables). A unit's score is the mean of the row averages it owns:
 * ViT:       scores_a [layers * heads]: head j = its 64 output rows of each of
 *            W^Q, W^K, W^V and its 64 input columns of W^O;
 *            scores_b [layers * mlp]: channel c = row c of W1, column c of W2.
 * ResNet-50: scores_a [sum of block widths]: S_a channel = conv1 output row,
 *            conv2 input slice; scores_b likewise: S_b channel = conv2 output
 *            row, conv3 input column. Blocks in order.
 * Synchronous. Errors: INVALID_ARG, CUDA, OOM. */
elasto_status elasto_saliency(const elasto_model_desc* desc, const elasto_weights* weights, float* scores_a,
                              float* scores_b);

/* Kept table from saliency scores: the k highest-scoring of n units (ties:
 * lower index), written ascending to out[k]. Taking every mode's table from
 * one ranking makes the modes nested (Eq. 8). Host-only. Errors: INVALID_ARG. */
elasto_status elasto_topk(const float* scores, int n, int k, int32_t* out);

/* L1-norm saliency of the d embedding channels of a ViT (Section 4.1: the
 * compress stage also shrinks the hidden size of the LayerNorm and
 * patch-embedding layers). Channel c owns the rows that write it (row c of the
 * patch projection, and of W^O and W2 in every layer) and the columns that
 * read it (column c of W_qkv and W1 in every layer, and of the classifier);
 * scores_e[c] [dim] is the mean of those 2 + 4 * layers row/column averages of
 * |w|. Same descriptor and tensor order as elasto_create; synchronous.
 * elasto_topk on the scores gives nested embed_kept tables (Eq. 8).
 * Errors: INVALID_ARG (not a ViT, null argument), CUDA, OOM. */
elasto_status elasto_saliency_embed(const elasto_model_desc* desc, const elasto_weights* weights, float* scores_e);

/* Test hook: copy one packed buffer of (mode, layer) to host_dst (bytes must
 * equal its size). ViT `which`: 0 qkv_w bf16 [3w,d], 1 qkv_b fp32 [3w],
 * 2 proj_w bf16 [d,w], 3 fc1_w bf16 [f,d], 4 fc1_b fp32 [f], 5 fc2_w bf16 [d,f]
 * (w = 64 x kept heads, f = kept channels). ResNet-50 (layer = block):
 * 0 conv1 f16 [|S_a|, cin], 1 bias1 fp32, 2 conv2 f16 [|S_b|, 3, 3, |S_a|],
 * 3 bias2 fp32, 4 conv3 f16 [4w, |S_b|], 5 bias3 fp32 (BN folded; the
 * ResNet path computes with IEEE f16 operands and fp32 accumulation).
 * Synchronous. Errors: INVALID_ARG, BAD_MODE. */
elasto_status elasto_debug_export_packed(elasto_t h, int mode, int layer, int which, void* host_dst,
                                         size_t bytes);

#ifdef __cplusplus
}
#endif
#endif /* ELASTO_H */
