/*
 * bag.h - C ABI of the GB300 (sm_103a) implementation of BAG's cached DiT sampling path.
 *
 * BAG ("Budget-Aware Gating for Diffusion Caching") runs a T-step sampler in which
 * exactly B steps evaluate the full network and the other T - B reuse the cached
 * stack residual; a small gate decides each step from the remaining budget and the
 * trajectory (Sec. 3.1 problem setup, Eq. 1 gate, Eq. 3 state, Algorithm 2).
 *
 * Conventions (every entry point):
 *   - Returns bag_status; nothing throws across the boundary.  On failure the message
 *     is available from bag_last_error(ctx).  A device-side error (a bounded wait that
 *     timed out inside a kernel) is sticky: every later call on the context returns
 *     BAG_EDEVICE_TIMEOUT until bag_reset.
 *   - "device" pointers are CUDA global-memory pointers on the context's device; "host"
 *     pointers are ordinary CPU memory.  The library never frees caller memory and never
 *     keeps a caller pointer past the call that received it.
 *   - Work is enqueued on the context's stream (bag_set_stream); calls that return
 *     results in host memory synchronise that stream.  A context is not thread-safe.
 *   - Tensors are dense row-major.  Image tokens are ordered row-major over the
 *     (frames, rows, cols) grid; text tokens come first in the joint sequence.
 */
#ifndef BAG_H_
#define BAG_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  BAG_OK = 0,
  BAG_EINVAL = 1,          /* bad argument (null pointer, size out of range, B > T ...) */
  BAG_ENOMEM = 2,          /* device allocation failed */
  BAG_ECUDA = 3,           /* a CUDA runtime call failed (message in bag_last_error) */
  BAG_EORDER = 4,          /* bag_step called with t != the context's next step */
  BAG_EDEVICE_TIMEOUT = 5, /* a kernel's bounded wait expired; results are invalid */
  BAG_ESTATE = 6,          /* call not valid in the context's current state */
  BAG_EUNSUPPORTED = 7     /* shape/type combination the kernels do not implement */
} bag_status;

enum { BAG_KIND_SINGLE = 0, BAG_KIND_MMDIT = 1, BAG_KIND_WAN = 2 };
enum { BAG_F32 = 0, BAG_BF16 = 1 };
/* Gate architectures (Eq. 1; the six-input ones are App. A.2's).  MLP3: inputs
 * [(B-c)/B, (T-t)/T, drift], 3 -> 16 -> 1 (81 params).  FLUX6: the six scalars of Eq. 3
 * [B/T, (B-c)/B, (B-c)/(T-t), t - t_last, drift, step change], 6 -> 8 -> 8 -> 32 -> 1
 * (449 params).  WAN6: the same six inputs, budget (first three) and trajectory (last
 * three) branches 3 -> 8 -> 8 each, concatenated budget-first, 16 -> 32 -> 1 (785
 * params).  Hidden layers use ReLU; the decision is sigmoid(z) > tau. */
enum { BAG_GATE_MLP3 = 0, BAG_GATE_FLUX6 = 1, BAG_GATE_WAN6 = 2 };
/* Samplers on the flow-matching noise levels sigma_i (i = 0..T), u_i = 1 - i/T time-shifted
 * by s: sigma_i = s u_i / (1 + (s - 1) u_i); the model is fed timestep 1000 sigma_i.
 * EULER: x_{i+1} = x_i + (sigma_{i+1} - sigma_i) v_i.  UNIPC: UniPC (Zhao et al. 2023) of
 * order 2 with its corrector, in data-prediction form (m = x - sigma v) with
 * B(h) = e^{-h} - 1, first order at the first and last step; the sampler the paper's Wan
 * experiments cache (Sec. 4.1).  Its multistep history lives in the context. */
enum { BAG_SAMPLER_EULER = 0, BAG_SAMPLER_UNIPC = 1 };
/* Observable of the trajectory signal (Eq. 3's drift and step change, relative L1).
 * MODULATED: the first block's modulated input on the image stream (LayerNorm of the
 * patch-embedded tokens under block 0's first adaLN shift and scale).  EMBEDDED: the
 * post-patch-embedding token tensor x_t itself, the paper's observable (Eq. 3 and the
 * paragraph after it; under guidance both branches share it). */
enum { BAG_OBS_MODULATED = 0, BAG_OBS_EMBEDDED = 1 };
enum {
  BAG_POLICY_BAG = 0,   /* Algorithm 2: gate decision + the two forced pacing rules */
  BAG_POLICY_FULL = 1,  /* uncached sampling: every step evaluates the network */
  BAG_POLICY_MASK = 2,  /* follow a caller-given mask (static schedule) */
  BAG_POLICY_STATIC_UNIFORM = 3, /* Sec. 3.1 static paradigm: B steps evenly spaced */
  BAG_POLICY_THRESHOLD = 4       /* Sec. 3.1 online threshold paradigm: compute when the
                                    drift since the last full step exceeds delta; the
                                    realised NFE is whatever the rule gives */
};

/* Backbone shape.  kind SINGLE: n_single single-stream blocks on the joint [text; image]
 * sequence.  MMDIT: n_double double-stream blocks, then n_single single-stream blocks
 * (FLUX/Qwen-Image layout).  WAN: n_wan blocks of self-attention (3D RoPE),
 * cross-attention to n_txt context tokens and FFN.  hidden = heads * head_dim;
 * rope_axes split head_dim over the (frame, row, col) axes (entries even, sum =
 * head_dim).  dtype: GEMM/attention operand type (the residual stream, latents, the
 * cached residual and all modulation vectors are fp32 in both cases).
 * cfg = 1 adds classifier-free guidance: every full step evaluates the stack for a
 * conditional and an unconditional branch (each its own text, pooled vector and cached
 * residual), both branches share one mask (a step is computed for both or reused for
 * both, App. A.1), the trajectory signal is read on the conditional branch (Eq. 3), and
 * the velocity is v_u + guidance * (v_c - v_u).  cfg = 0 ignores guidance. */
typedef struct {
  int kind;
  int hidden, heads, mlp;
  int n_double, n_single, n_wan;
  int grid[3];        /* frames, rows, cols of image tokens; n_img = product */
  int n_txt;          /* text tokens (joint attention) or context tokens (Wan) */
  int patch_ch;       /* latent channels per image token (64) */
  int rope_axes[3];
  int dtype;          /* BAG_F32 or BAG_BF16 */
  uint64_t weight_seed, gate_seed;
  float tau;          /* gate cutoff: a step computes when sigmoid(z) > tau (0 < tau < 1) */
  int gate_kind;      /* BAG_GATE_* */
  int cfg;            /* 0 or 1: classifier-free guidance with a shared mask */
  float guidance;     /* guidance scale g (finite; used when cfg = 1) */
  int qk_norm;        /* 0 or 1: RMSNorm of every q and k head (eps 1e-6, learned scale per
                         head channel) before RoPE, as in FLUX / Qwen-Image blocks; SINGLE
                         and MMDIT kinds with BAG_BF16 only (else BAG_EUNSUPPORTED) */
  int sampler;        /* BAG_SAMPLER_* */
  float shift;        /* time shift s of the sigma grid (> 0; 0 is read as 1, no shift) */
  int observable;     /* BAG_OBS_*: what the trajectory signal reads */
} bag_arch;

/* Conditioning of one sample (device pointers, read during bag_step / bag_run).
 * txt: [n_txt, hidden] text tokens (fp32 for BAG_F32 contexts, bf16 for BAG_BF16).
 * pooled: [hidden] fp32 pooled text vector added to the time embedding (ignored for
 * WAN; may be null there).  txt_uncond / pooled_uncond: the unconditional branch's,
 * same layouts; required by cfg contexts (pooled_uncond may be null for WAN), ignored
 * otherwise. */
typedef struct {
  const void* txt;
  const float* pooled;
  const void* txt_uncond;
  const float* pooled_uncond;
} bag_cond;

/* Per-sample schedule statistics.  mask / log are optional host arrays supplied by the
 * caller: mask[T] receives m_t, log[T * BAG_LOG_FLOATS] the per-step record
 *   [0..2] (B-c)/B, (T-t)/T, drift;  [3] gate logit z;  [4] raw gate bit;  [5] m_t;
 *   [6] c before the step;  [7] t - t_last;  [8..10] B/T, (B-c)/B, (B-c)/(T-t);
 *   [11] sum|m_t - m_last|;  [12] sum|m_last|;  [13] step change;  [14] sum|m_t - m_{t-1}|;
 *   [15] sum|m_{t-1}|   (m = the signal's observable, see BAG_OBS_*).
 * nfe receives the realised number of full evaluations. */
#define BAG_LOG_FLOATS 16
typedef struct {
  uint8_t* mask;
  float* log;
  int nfe;
  int T, B;
} bag_stats;

typedef struct bag_ctx bag_ctx;

/* Create a context for `arch` with a T-step sampler under budget B (1 <= B <= T,
 * Sec. 3.1: ||m||_1 = B with m_0 = 1).  Allocates and seeds all weights on the current
 * CUDA device from arch->weight_seed (SplitMix64 counter generator), seeds the gate
 * from arch->gate_seed, and allocates every activation buffer the step needs, so that
 * no later call allocates.  *out receives the context (NULL on failure).  Consecutive
 * kernels of a step are launched with programmatic stream serialization (each kernel
 * waits on the device for its predecessor); the environment variable BAG_PDL=0, read
 * here, launches them with plain stream order instead.
 * Errors: EINVAL (bad arch/T/B), ENOMEM, ECUDA, EUNSUPPORTED. */
bag_status bag_create(const bag_arch* arch, int T, int B, bag_ctx** out);

/* Release every device resource of the context (null is a no-op). */
void bag_destroy(bag_ctx* ctx);

/* Text of the last error on this context, or, when ctx is null, of the last failed
 * context-free call (bag_create, bag_rel_l1_noalloc) made by the calling host thread
 * (that text is kept per thread).  Valid until the next call on the context (ctx
 * non-null) or the thread's next context-free call (ctx null). */
const char* bag_last_error(bag_ctx* ctx);

/* Order the context's work after, and before, the caller's `cuda_stream` (a
 * cudaStream_t; null = the legacy stream).  The context keeps its own stream for the
 * captured step graph and bridges the two with events on every call.  The paper runs
 * the T decisions of a sample strictly in sequence (Sec. 3.1 problem setup,
 * Algorithm 2); this call only chooses which caller stream that sequence is ordered
 * against, it never reorders steps. */
bag_status bag_set_stream(bag_ctx* ctx, void* cuda_stream);

/* Replace the gate parameters (Eq. 1; App. A.2 z-scored inputs).  theta: host array of
 * n floats, every layer's W [out][in] (row-major) then its b, in the order listed with
 * BAG_GATE_* (WAN6: budget branch, trajectory branch, fuse layers); n must equal the
 * kind's parameter count (81, 449 or 785) else EINVAL.  mu, sd: host arrays with one
 * float per gate input (3 or 6; z-score statistics; null = 0 and 1; sd nonzero). */
bag_status bag_load_gate(bag_ctx* ctx, const float* theta, int n, const float* mu,
                         const float* sd);

/* Choose the schedule policy (BAG_POLICY_*).  For BAG_POLICY_MASK, host_mask[T] gives
 * the per-step bits (host_mask[0] is ignored: step 0 always computes).
 * BAG_POLICY_STATIC_UNIFORM computes steps floor(i T / B), i < B.  BAG_POLICY_THRESHOLD
 * computes step t >= 1 when the fp32 drift > delta (delta ignored by other policies).
 * The budget pacing of Algorithm 2 applies only to BAG_POLICY_BAG. */
bag_status bag_set_policy(bag_ctx* ctx, int policy, const uint8_t* host_mask, float delta);

/* Change the budget of later samples to B (1 <= B <= T, else EINVAL; Sec. 3.2: the target
 * budget is set at runtime and one gate serves every budget).  The step graph is
 * re-captured on the next run; a static evenly spaced mask is recomputed for B.  Call
 * between samples. */
bag_status bag_set_budget(bag_ctx* ctx, int B);

/* Start a new sample (a new prompt): Algorithm 2's initial state, t = 0 and the spent
 * budget c = 0, with the residual cache invalid so that step 0 computes (m_0 = 1,
 * Sec. 3.1); the sticky device error is cleared. */
bag_status bag_reset(bag_ctx* ctx);

/* One sampler step (Algorithm 2, one iteration).  t must equal the context's next step
 * (0, 1, ..., T-1 after bag_reset) else EORDER.  x: device fp32 [n_img, patch_ch]
 * latent x_t; x_out: device fp32 [n_img, patch_ch] receives x_{t+1} (may equal x).
 * full_or_cached: device int32* written asynchronously with 1 (full evaluation) or 0
 * (cached residual reused); may be null.  The decision is taken on the device: no host
 * synchronisation happens inside the step. */
bag_status bag_step(bag_ctx* ctx, const float* x, int t, const bag_cond* cond, float* x_out,
                    int32_t* full_or_cached);

/* All T steps of one sample from the context's current state (normally right after
 * bag_reset), in place on x_inout (device fp32 [n_img, patch_ch]): Algorithm 2's loop
 * over t = 0 .. T-1, each iteration one bag_step (gate, pacing, full stack or cached
 * residual, sampler update), with exactly B full evaluations (Sec. 3.2 budget-exact
 * inference).  stats (optional, host) receives the schedule after one synchronisation
 * at the end. */
bag_status bag_run(bag_ctx* ctx, float* x_inout, const bag_cond* cond, bag_stats* stats);

/* Same as bag_run with HOST buffers: copies x (fp32 [n_img, patch_ch]) and the
 * conditioning cond_host (every pointer host memory; text fp32 [n_txt, hidden] whatever
 * the context's dtype, converted on device for bf16 contexts; pooled fp32 [hidden], may
 * be null for WAN) to the device, runs the sample and copies the result back into
 * x_host.  For pageable memory the copies are synchronous. */
bag_status bag_run_host(bag_ctx* ctx, float* x_host, const bag_cond* cond_host, bag_stats* stats);

/* ---- inspection and single-operation entry points (tests, benchmarks) ---- */

/* Copy weight tensor `name` of block `block` (-1 = global tensors) to host fp32
 * `out` (n elements, must equal the tensor size).  Names follow the seeded generator's
 * inventory (e.g. "lin1_w", "img_qkv_b", "pe_w", "fmod_w"). */
bag_status bag_get_weight(bag_ctx* ctx, int block, const char* name, float* out, size_t n);

/* Run block `block` of the stack once on a caller-provided stream state, with the
 * modulation of step t_mod of the current sample (modulation is precomputed by
 * bag_prepare).  h: device fp32 joint sequence [n_txt + n_img, hidden] (text rows first)
 * for SINGLE/MMDIT; for WAN h is the image stream [n_img, hidden] and the context comes
 * from the last bag_prepare.  Updated in place. */
bag_status bag_forward_block(bag_ctx* ctx, int block, int t_mod, float* h);

/* Precompute the conditioning of a sample (time embedding and every block's
 * modulation for all T steps) and stage its text tokens; bag_run does this itself. */
bag_status bag_prepare(bag_ctx* ctx, const bag_cond* cond);

/* Profiled sample.  Same as bag_run on a fresh sample, but every kernel is launched
 * directly (no graph) between two CUDA events, and the step's decision is read back
 * after the gate so that only the taken branch is launched.  out[BAG_PROF_KINDS]
 * receives per kernel class: launches, summed event time (ms), summed algorithmic
 * flops and bytes (the work the method needs, not counter values).  Slower than
 * bag_run (one host synchronisation per step); for measurement only. */
enum {
  BAG_PROF_GEMM = 0,   /* projections (tensor cores), incl. patch embed and final layer */
  BAG_PROF_ATTN = 1,   /* attention */
  BAG_PROF_NORM = 2,   /* LayerNorm + modulation inside the stack and the final layer */
  BAG_PROF_SIGNAL = 3, /* trajectory signal (block-0 LN-mod fused with the rel-L1 partials) */
  BAG_PROF_GATE = 4,   /* gate + pacing */
  BAG_PROF_CACHE = 5,  /* cache refresh (full step) and residual reuse (cached step) */
  BAG_PROF_KINDS = 6
};
typedef struct {
  long launches;
  double ms;
  double flops;
  double bytes;
} bag_prof_entry;
bag_status bag_profile_run(bag_ctx* ctx, float* x_inout, const bag_cond* cond, bag_stats* stats,
                           bag_prof_entry* out);

/* Per-launch records of the last bag_profile_run: kind (BAG_PROF_*), shape (GEMM: M, N,
 * K; attention: n_q, n_k, heads; 0 otherwise), event time, algorithmic flops and bytes,
 * and the kernel variant (GEMM: 1 = CTA-pair kernel, 0 = single-CTA kernel; else 0).
 * *n receives the number of records; up to max are copied to out (host; may be null). */
typedef struct {
  int kind, m, n, k;
  float ms;
  double flops, bytes;
  int variant;
} bag_prof_launch;
bag_status bag_profile_launches(bag_ctx* ctx, bag_prof_launch* out, long max, long* n);

/* Number of kernel launches the last bag_run enqueued (graph nodes included). */
bag_status bag_launch_count(bag_ctx* ctx, long* out);

/* C[M,N] = A[M,K] W[N,K]^T (+ bias[N]) on the tensor cores: A, W bf16 device, lda/ldw
 * in elements (multiples of 8), K a multiple of 64, N a multiple of 64; C fp32 device
 * with row stride ldc; bias device fp32 or null.  epilogue: 0 = store, 1 = GELU(tanh).
 * force_simt != 0 runs the CUDA-core kernel instead (cross-check). */
bag_status bag_gemm_bf16(bag_ctx* ctx, const void* A, long lda, const void* W, long ldw,
                         const float* bias, float* C, long ldc, int M, int N, int K,
                         int epilogue, int force_simt);

/* Multi-head attention softmax(q k^T / sqrt(dh)) v (the joint attention of the DiT
 * blocks): q [nq, ld], k [nk, ld] bf16 device, head h at columns [h*dh, (h+1)*dh);
 * o [nq, ld] bf16 device.  v: if vpad > 0, transposed per head, [heads][dh][vpad] bf16
 * (vpad >= nk, multiple of 8; the layout the tensor-core kernel reads); if vpad == 0,
 * [nk, ld] like k (CUDA-core kernel only).  The tensor-core kernel needs dh = 128;
 * force_simt != 0 selects the CUDA-core kernel (dh 64 or 128). */
bag_status bag_attention_bf16(bag_ctx* ctx, const void* q, const void* k, const void* v,
                              void* o, long ld, int nq, int nk, int heads, int dh, long vpad,
                              int force_simt);

/* bag_attention_bf16 with fp16 q, k and v (same layouts; v transposed per head, vpad > 0)
 * and a bf16 output o: the operand type the sampling path of bf16 backbones uses for
 * attention (an 11-bit significand for q and k, whose rounding the softmax exponent
 * amplifies; the softmax probabilities P enter the PV product as fp16 too).  Tensor-core
 * kernel only (dh 128), else BAG_EUNSUPPORTED. */
bag_status bag_attention_f16(bag_ctx* ctx, const void* q, const void* k, const void* v, void* o,
                             long ld, int nq, int nk, int heads, int dh, long vpad);

/* y = (1 + scale) * LayerNorm(x) + shift row-wise (eps 1e-6, no affine): x fp32 device
 * [rows, cols], shift/scale fp32 device [cols] (null = plain LayerNorm), y bf16 device. */
bag_status bag_ln_mod(bag_ctx* ctx, const float* x, const float* shift, const float* scale,
                      void* y, int rows, int cols);

/* Trajectory signal of Eq. 3 with the L1 norm: relative change sum|a - b| / sum|b| of
 * two device tensors a, b [rows, cols] (dtype BAG_F32 or BAG_BF16; b is the reference).
 * scratch: caller-owned device fp32 [2 * rows] for per-row partial sums (overwritten);
 * out: device fp32 [3] receives {sum|a-b| / sum|b|, sum|a-b|, sum|b|}.  The row
 * partials are summed in a fixed order, so repeated calls give identical results. */
bag_status bag_rel_l1(bag_ctx* ctx, const void* a, const void* b, int dtype, long rows,
                      long cols, float* scratch, float* out);

/* Allocation-free bag_rel_l1 (the paper has no counterpart: this is a deployment
 * variant).  For callers that cannot call cudaMalloc - code inside a framework whose
 * caching allocator owns the device memory, or loops that cannot take cudaMalloc's
 * implicit synchronisation - and so cannot create a context either: no context, no
 * allocation.  a, b: device [rows, cols] (dtype BAG_F32 or BAG_BF16); out: device fp32
 * [3] as for bag_rel_l1; work runs on cuda_stream (a cudaStream_t, null = legacy).
 * The row partials live in a fixed file-scope device array of 2 * 65536 floats held by
 * every GPU that loads the library until exit: rows > 65536 returns BAG_EINVAL.  The
 * first call on a device looks the array's address up (cudaGetSymbolAddress) and
 * should come before any stream capture; the address is kept per CUDA context and
 * looked up again when the device's current context changes (e.g. after
 * cudaDeviceReset).  All calls share the array and it keeps the last call's contents
 * (each call writes what it reads); calls that overlap on the GPU race.  Errors are
 * reported through bag_last_error(NULL). */
bag_status bag_rel_l1_noalloc(const void* a, const void* b, int dtype, long rows, long cols,
                              float* out, void* cuda_stream);

/* Failure-path check: launches one kernel whose mbarrier wait can never complete (no
 * thread arrives on it), so its bounded wait gives up after the library's wait limit
 * (about 2 s), records the sticky device error and returns; nothing faults or hangs.
 * Returns BAG_EDEVICE_TIMEOUT once the stream reaches it; bag_run and bag_step report
 * the sticky error until bag_reset.  For tests of the error path only. */
bag_status bag_check_wait_timeout(bag_ctx* ctx);

/* Skip path (plain residual reuse): out = h_in + R, fp32 device, n elements (n % 4 == 0). */
bag_status bag_residual_add(bag_ctx* ctx, float* out, const float* h_in, const float* R, long n);

#ifdef __cplusplus
}
#endif

#endif /* BAG_H_ */
