// Internal interface between the C-ABI layer (bag_api.cu) and the kernels.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <utility>

namespace bag {

// Set between consecutive kernels of one enqueued segment of a step: launch_kernel then
// gives the launch programmatic stream serialization, so the kernel's CTAs are resident
// and waiting (grid_dep_sync) when its predecessor completes.
extern thread_local bool g_pdl;

template <typename... P, typename... A>
inline cudaError_t launch_kernel(void (*k)(P...), dim3 grid, dim3 block, size_t smem,
                                 cudaStream_t s, A&&... args) {
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t c = {};
  c.gridDim = grid;
  c.blockDim = block;
  c.dynamicSmemBytes = smem;
  c.stream = s;
  c.attrs = at;
  c.numAttrs = g_pdl ? 1 : 0;
  return cudaLaunchKernelEx(&c, k, std::forward<A>(args)...);
}

// Per-sample state the step kernels read and write on the device, so that a whole
// denoising step can be replayed from a CUDA graph with no host round trip.
struct DevState {
  int t;          // current step index (advanced on device at the end of each step)
  int c;          // full evaluations spent so far (Algorithm 2's counter)
  int t_last;     // last fully computed step
  int flag;       // decision of the current step: 1 = full, 0 = reuse
  int err;        // sticky error word (device wait timeout etc.)
  int pad[3];
};

// Per-step log record (written by the gate kernel).
constexpr int kLogFloats = 16;
// [0..2]  gate inputs  (B-c)/B, (T-t)/T, drift
// [3]     gate logit z
// [4]     raw gate bit, [5] final decision m_t, [6] c before the step, [7] t - t_last
// [8..10] budget state of Eq. 3: B/T, (B-c)/B, (B-c)/(T-t)
// [11]    drift numerator sum|m_t - m_last|, [12] denominator sum|m_last|
// [13]    step-to-step change, [14] its numerator sum|m_t - m_{t-1}|, [15] sum|m_{t-1}|

// gate parameter buffer: layers from 0, z-score mean / sd at fixed offsets
constexpr int kGateMaxParams = 800;
constexpr int kGateMu = 800;
constexpr int kGateSd = 806;
constexpr int kGateFloats = 812;

enum EpiKind : int {
  EPI_STORE = 0,      // out = acc + bias                       (out_bf16 selects type)
  EPI_GELU = 1,       // out = gelu(acc + bias)
  EPI_SILU = 2,       // out = silu(acc + bias)
  EPI_QKV = 3,        // attention operands (+RoPE) and, past 3d, GELU(mlp) part
  EPI_GATED_RES = 4,  // resid += gate * (acc + bias)
  EPI_RES_ADD = 5,    // resid += acc + bias
  EPI_EULER = 6,      // x += dsig[t] * (acc + bias); xb = bf16(x)
  EPI_VEC = 7,        // out = acc + bias + addend; out2 = silu(out) (bf16 or f32)
  EPI_DUAL_F32 = 8,   // out = out2 = acc + bias (f32)
};

// UniPC coefficients per step: sigma_i; corrector weights of x_i, the previous corrected
// sample, m_{i-1}, m_{i-2}, m_i; predictor weights of the corrected sample, m_i, m_{i-1}.
enum { UC_SIG = 0, UC_CX, UC_CLAST, UC_CM1, UC_CM2, UC_CMT, UC_DX, UC_DM0, UC_DM1, kUniCoefs };

// Storage types of epilogue outputs (the *_bf16 flags hold 0 or 1; type fields any)
enum { kStoreF32 = 0, kStoreBF16 = 1, kStoreF16 = 2 };

struct Epi {
  int kind = EPI_STORE;
  int M = 0, N = 0;
  const float* bias = nullptr;
  // plain stores
  void* out = nullptr;
  long ldo = 0;
  int out_bf16 = 0;                // storage type of out (kStore*: 0 fp32, 1 bf16, 2 fp16)
  void* out2 = nullptr;
  long ldo2 = 0;
  int out2_bf16 = 0;
  const float* addend = nullptr;  // EPI_VEC: [N] vector added to every row
  // residual updates
  float* resid = nullptr;
  long ldr = 0;
  const float* gate = nullptr;    // gate for step t = gate + t * gate_step
  const float* gate_u = nullptr;  // unconditional branch's gate (rows >= br_rows)
  long gate_step = 0;
  // attention operands
  void* q = nullptr;
  void* k = nullptr;
  void* v = nullptr;       // v_mode 0: [rows, ldqk]; v_mode 1: transposed [H][dh][vpad]
  int v_mode = 0;
  long ldqk = 0;
  int d = 0, dh = 0;
  long vpad = 0;
  int row_off = 0;         // joint-sequence row of this GEMM's row 0
  // Two guidance branches in one problem: rows [0, br_rows) are the conditional branch,
  // rows [br_rows, 2 br_rows) the unconditional one (br_rows = 0: a single branch).
  // EPI_QKV writes branch 1's q / k rows br_qk rows further and its transposed V br_vt
  // elements further; EPI_GATED_RES takes branch 1's gate from gate_u.
  int br_rows = 0;
  long br_qk = 0, br_vt = 0;
  int col_base = 0;        // logical column of this GEMM's column 0 (q=0, k=d, v=2d, mlp=3d)
  const float2* rope = nullptr;  // [joint rows][dh/2] (cos, sin); null = no rotation
  int act_bf16 = 1;        // mlp storage type (1 bf16, 0 fp32)
  int qkv_type = 1;        // q/k/v storage type (kStoreF32, kStoreBF16 or kStoreF16)
  void* mlp = nullptr;     // GELU(mlp) columns go to mlp[row * ldm + (col - 3d)]
  long ldm = 0;
  // sampler update
  float* x = nullptr;
  __nv_bfloat16* xb = nullptr;  // [rows, 2 * ldx]: bf16 hi | lo halves of the updated x
  long ldx = 0;
  const float* dsig = nullptr;  // [T]: sigma_{t+1} - sigma_t
  const float* qn_q = nullptr;  // EPI_QKV: per-head RMSNorm scales [dh] of q and k (both
  const float* qn_k = nullptr;  //   set or both null), applied before RoPE
  const float* vcond = nullptr; // guidance: conditional velocity [rows, ldx]; null = none
  float guidance = 0.f;         // v = v_u + guidance * (vcond - v_u), v_u this GEMM's output
  // EPI_EULER as a UniPC step when uni_coef is set: per step kUniCoefs coefficients,
  // the previous corrected sample uni_xl and the data predictions of the last two
  // steps in uni_m[step & 1] (all fp32 [rows, ldx])
  const float* uni_coef = nullptr;
  float* uni_xl = nullptr;
  float* uni_m0 = nullptr;
  float* uni_m1 = nullptr;
  // step-dependent addressing and early exit
  const DevState* st = nullptr;  // null: step 0, no flag check
  int flag_want = -1;            // -1: always run; 0/1: run only when st->flag equals it
};

// ---------------------------------------------------------------------------
// launchers (all asynchronous on the given stream); return cudaError_t
// ---------------------------------------------------------------------------
// C[M,N] = A[M,K] W[N,K]^T with the fused epilogue.  Tensor-core path for bf16
// operands; fp32 operands (and shapes the tensor-core path does not tile) go to the
// CUDA-core path.
// a_split (bf16 only): A is [M, 2K] = [hi | lo] bf16 halves of an fp32 activation
// (see split_bf16); the product then carries fp32-level accuracy in A.
cudaError_t gemm(const void* A, long lda, const void* W, long ldw, int M, int N, int K,
                 int in_bf16, const Epi& epi, int* err, cudaStream_t s, int force_simt = 0,
                 int a_split = 0);
// dst [rows, 2*cols] bf16 = [bf16(x) | bf16(x - bf16(x))] of src fp32 [rows, cols]
cudaError_t split_bf16(__nv_bfloat16* dst, const float* src, long rows, long cols, cudaStream_t s);
int gemm_tc_supported(int M, int N, int K, long lda, long ldw);
// 1 when a bf16 launch of these shapes runs on the CTA-pair kernel (gemm_pair_kernel)
int gemm_uses_pair(int M0, int M1, int N);
// Two bf16 problems with the same N and K in one tensor-core launch (e.g. the image and
// text streams of a double-stream block); M1 may be 0.
cudaError_t gemm2(const void* A0, long lda0, const void* W0, long ldw0, int M0, const Epi& epi0,
                  const void* A1, long lda1, const void* W1, long ldw1, int M1, const Epi& epi1,
                  int N, int K, int* err, cudaStream_t s);

struct AttnArgs {
  const void* q;  long ldq;      // [Nq rows][ldq], head h at column h*dh
  const void* k;  long ldk;      // [Nk rows][ldk]
  const void* v;  int v_mode; long ldv; long vpad;  // mode 0 like k; mode 1 [H][dh][vpad]
  void* o;        long ldo;      // output [Nq][ldo], head h at column h*dh
  void* o2 = nullptr; int o_split = 0;  // rows >= o_split go to o2 (+ row * ldo) instead
  // nbr = 2 (tensor-core kernel): two guidance branches in one launch; branch 1's q and k
  // rows start br_q_rows / br_k_rows rows further, its transposed V heads * dh rows
  // further (each branch has its own [heads][dh][vpad] block), and its output goes to
  // o_b1 / o2_b1 with the same row split
  int nbr = 1;
  long br_q_rows = 0, br_k_rows = 0;
  void* o_b1 = nullptr;
  void* o2_b1 = nullptr;
  int nq, nk, heads, dh;
  int bf16;                      // 16-bit operands and output (else fp32)
  int f16 = 0;                   // with bf16: q, k, v are fp16 (output stays bf16)
  const DevState* st; int flag_want;
};
cudaError_t attention(const AttnArgs& a, int* err, cudaStream_t s, int force_simt = 0);
int attention_tc_supported(const AttnArgs& a);

// Row-wise LayerNorm (no affine, eps 1e-6) + adaLN modulation over rows [0, rows).
// Rows < split use (shift_a, scale_a), the rest (shift_b, scale_b); modulation vectors
// are read at base + t * mod_step.  shift/scale null = plain LayerNorm.
struct LnArgs {
  const float* x; long ldx;
  void* y; long ldy; int y_bf16;
  int rows, cols, split;
  const float* shift_a; const float* scale_a;
  const float* shift_b; const float* scale_b;
  // up to four row segments: [0, split) a, [split, split2) b, [split2, split3) c,
  // [split3, rows) d (split2 = split3 = 0: two segments)
  int split2 = 0, split3 = 0;
  const float* shift_c = nullptr; const float* scale_c = nullptr;
  const float* shift_d = nullptr; const float* scale_d = nullptr;
  long mod_step;
  // fused trajectory signal: per-row partial sums of |y - ref|, |ref|, |y - ref2|,
  // |ref2| (4 floats per row); ref2 may alias y (it is read before y is stored).
  // sig_ref_w (optional, = sig_ref): when the previous step was fully computed
  // (st->t_last == st->t - 1) its observable ref2 is the new reference, so the kernel
  // reads ref2 once, takes it as ref and writes it into sig_ref_w as it goes (the
  // reference refresh of Algorithm 2 without a separate copy).
  const void* sig_ref; const void* sig_ref2; float* sig_partial; int sig_on;
  void* sig_ref_w = nullptr;
  // identity: y = x (no normalisation or modulation; the observable is x itself)
  int identity = 0;
  // rows ahead whose x (and signal references) a CTA pulls into L2 for a CTA of a later
  // wave (set by the launcher: resident CTAs of the whole GPU; 0 = none)
  int prefetch_rows = 0;
  const DevState* st; int flag_want;
};
cudaError_t ln_mod(const LnArgs& a, cudaStream_t s);

cudaError_t gate_step(DevState* st, const float* sig_partial, int sig_rows, const float* gate_params,
                      int gate_kind, float thr, int T, int B, int policy,
                      const uint8_t* policy_mask, float delta, float* log,
                      unsigned long long cond_handle, int use_cond, cudaStream_t s);
cudaError_t cache_refresh(const DevState* st, const float* h_img, const float* h_in, float* R, long n,
                          int flag_want, cudaStream_t s);
cudaError_t cache_reuse(const DevState* st, float* h_img, const float* h_in, const float* R,
                        long n, int flag_want, cudaStream_t s);
cudaError_t copy_rows_f32(const DevState* st, int flag_want, float* dst, long ldd, const void* src,
                          long lds, int src_bf16, int rows, int cols, cudaStream_t s);
cudaError_t advance_step(DevState* st, cudaStream_t s);
// one thread waits (bounded) on an mbarrier nothing arrives on, then sets st->err
cudaError_t wait_timeout_probe(DevState* st, cudaStream_t s);
cudaError_t sinusoid_all(void* out, int out_bf16, const double* sigma, int T, int dim, cudaStream_t s);
cudaError_t expand_wan_mod(float* mod_all, const float* shared6d, const float* tables,
                           int T, int nblocks, int d, cudaStream_t s);
cudaError_t to_bf16(__nv_bfloat16* dst, const float* src, long n, cudaStream_t s);
cudaError_t fill_synth(void* dst, long n, uint64_t start, float offset, float c32, int bf16,
                       cudaStream_t s);
cudaError_t residual_add(float* out, const float* a, const float* b, long n, cudaStream_t s);
cudaError_t rel_l1_partials(const void* a, const void* b, int a_bf16, long rows, long cols,
                            float* partial, cudaStream_t s);
cudaError_t rel_l1_finalize(const float* partial, long rows, float* out, cudaStream_t s);

// message returned by bag_last_error(NULL) (entry points without a context)
}  // namespace bag
#include <string>
namespace bag {
void set_global_error(const std::string& msg);

// one-time kernel attribute setup (dynamic shared memory limits); call before capture
cudaError_t kernels_init();

// host-side TMA descriptor encoding (driver entry point resolved at run time)
int encode_tmap_2d_bf16(CUtensorMap* map, const void* base, uint64_t inner, uint64_t outer,
                        uint64_t row_stride_bytes, uint32_t box_inner, uint32_t box_outer);

}  // namespace bag
