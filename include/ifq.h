/*
 * ifq.h -- C ABI of the GB300 library for the quantized substructure of
 * IFQ-Net (Gao et al., "IFQ-Net: Integrated Fixed-point Quantization Networks
 * for Embedded Vision", arXiv:1911.08076).
 *
 * The library computes, on one GPU, the quantized convolution of Eq. (1) with
 * +-1 filters W_b and unsigned k-bit input codes X_q (k = 2, 3 or 4), and
 * applies the integrated fixed-point conversion of Sec. 3.2 as its epilogue:
 * the integer accumulator W_b (x) X_q is compared with per-channel integer
 * thresholds (Eq. (7) after the floor; Eq. (8) for k bits), which emits the
 * next layer's k-bit codes.
 *
 * Conventions shared by every call:
 *   - Return value: an ifq_status.  Argument, shape, alignment and range
 *     errors are returned synchronously, before anything is launched.
 *   - Pointers marked (device) are CUDA device pointers; (host) are host
 *     pointers.  The caller owns every buffer; nothing is retained after the
 *     call returns, and the library allocates no device memory in any call
 *     named here except ifq_graph_create (which owns the captured graph).
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *     stream).  Device work is enqueued on it and the call returns without
 *     waiting, except where stated.
 *   - Device-side failures (a bounded wait that ran out, a failed bounds
 *     check) never trap: they set a device status word that
 *     ifq_device_status reads.
 *   - A batch of n = 0 images is valid everywhere: arguments are checked as
 *     usual and nothing is launched.
 *
 * Data formats:
 *   - Codes: NHWC, packed along C in fields of f bits: f = 2 for k = 2 (four
 *     codes per byte), f = 4 for k = 3 and k = 4 (two codes per byte, a 3-bit
 *     code in the low bits of its field).  Channel c of a pixel is bits
 *     f*(c%(8/f)) .. f*(c%(8/f))+f-1 of byte c/(8/f) of that pixel.  C must be
 *     a multiple of 4, so a pixel is C*f/8 bytes.  Buffers are at least
 *     16-byte aligned (cudaMalloc / torch allocations are).
 *   - Filter signs: one row per output channel over K = kh*kw*cin in
 *     (dy, dx, c) order (c fastest); bit k%32 of 32-bit word k/32 is 1 for +1
 *     and 0 for -1; a row is ceil(K/32) words.
 *   - Thresholds: int32 [cout][2^k - 1], ascending (not necessarily strictly),
 *     and int8 sign [cout] in {+1, -1}; the code of accumulator A in channel n
 *     is the number of i with sign[n]*A > T[n][i].
 *   - Accumulators: int32 NHWC [n][ho][wo][cout].
 *   - Convolution geometry: cross-correlation, symmetric zero padding `pad`
 *     (a padded cell is code 0), ho = (h + 2*pad - kh)/stride + 1.
 *   - Pooling geometry: k x k windows starting at (oy*stride, ox*stride),
 *     `pad` extra empty cells at the bottom and right that are skipped,
 *     ho = (h + pad - k)/stride + 1.
 */
#ifndef IFQ_H
#define IFQ_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  IFQ_OK = 0,
  IFQ_EINVAL = 1,        /* null pointer or invalid parameter value */
  IFQ_ESHAPE = 2,        /* inconsistent or unsupported shape */
  IFQ_EALIGN = 3,        /* pointer not aligned as required */
  IFQ_ERANGE = 4,        /* a size exceeds what the library supports */
  IFQ_ECUDA = 5,         /* a CUDA runtime call failed */
  IFQ_ETIMEOUT = 6,      /* (device status) a bounded wait in a kernel ran out */
  IFQ_EUNSUPPORTED = 7,  /* valid request that the library does not implement */
  IFQ_EWORKSPACE = 8     /* workspace missing or too small */
} ifq_status;

/* Output selection of a convolution. */
enum { IFQ_OUT_CODES = 1, IFQ_OUT_ACC = 2, IFQ_OUT_BOTH = 3 };

/* Kernel path of a convolution (ifq_conv_desc.path). */
enum {
  IFQ_PATH_AUTO = 0,
  IFQ_PATH_TC = 1,
  IFQ_PATH_BITSERIAL = 2,
  IFQ_PATH_DIRECT = 3,
  IFQ_PATH_WIN = 4,
  IFQ_PATH_WARP = 5
};

/* Layer kinds of ifq_forward. */
enum { IFQ_LAYER_CONV = 1, IFQ_LAYER_POOL = 2, IFQ_LAYER_FIXED = 3 };

/* Text for a status code (static storage; never NULL). */
const char* ifq_status_str(int status);

/* Library ABI version: 100*major + minor. */
int ifq_version(void);

/*
 * Environment switches, read on every call that uses them (for experiments; the defaults are the
 * measured best):
 *   IFQ_FORCE_PATH   = 1 / 2 / 3 / 4 / 5: request IFQ_PATH_TC / IFQ_PATH_BITSERIAL / IFQ_PATH_DIRECT /
 *                      IFQ_PATH_WIN / IFQ_PATH_WARP where a descriptor says IFQ_PATH_AUTO
 *                      (ifq_conv_plan reports the result).
 *   IFQ_WIN          = 0: never take the window path (IFQ_PATH_WIN requests take the tensor-core path).
 *   IFQ_WARP         = 0: never take the warp-MMA path (IFQ_PATH_WARP requests take the tensor-core
 *                      path).
 *   IFQ_TC_BN        = 32 / 64 / 128: the tensor-core kernel's output-channel tile width.
 *   IFQ_TC_KS        = 1 / 2: forbid / force splitting K over clusters of two CTAs (by default only
 *                      layers that would leave more than half of the SMs idle are split).
 *   IFQ_TC_BX        = 1 / 2: the split tensor-core kernel expands its filter tiles in shared memory
 *                      from the sign bits (1 bit per weight read instead of 8) for layers with at most
 *                      two 128-row tiles / wherever it runs (off by default: not faster where measured).
 *   IFQ_PDL          = 0: launch without programmatic dependent launch.
 *   IFQ_GRAPH_BRANCH = 0: capture stacks as one chain, without side branches.
 *   IFQ_STACK        = 1: run qualifying stacks as one persistent launch (ifq_forward).
 * None changes a result; all change only how it is computed.
 */

/*
 * ifq_fold_layer -- integrated fixed-point conversion of one quantized
 * substructure (Sec. 3.2, Eq. (6)-(7), floor of the composed thresholds).
 * Host only, pure, thread-safe; nothing is launched.
 *
 * For output channel n the float substructure is
 *   y = alpha[n]*delta_in*A + bias[n]                        (Eq. (1))
 *   z = gamma[n]*(y - mean[n])/sqrt(var[n] + eps) + beta[n]   (Eq. (2), affine BN)
 *   code = #{ i in 1..L : z > q_base*i + q_offset }           (Eq. (3), L = 2^kbits - 1)
 * and the fold returns T[n][i-1] and sign[n] such that
 *   code = #{ i : sign[n]*A > T[n][i-1] }
 * for every integer A with |A| <= L*K:
 *   tau_i = ((thr_i - beta)*sqrt(var + eps)/gamma + mean - bias)/(alpha*delta_in)
 *   gamma > 0: sign = +1, T = floor(tau_i);  gamma < 0: sign = -1, T = floor(-tau_i)
 *   gamma = 0: sign = +1, T = -L*K-1 if beta > thr_i else L*K
 * T is clamped to [-L*K-1, L*K].  The arithmetic is IEEE double in the order
 * written above.
 *
 * Arguments (host): alpha, gamma, beta, mean, var: [cout] float; bias: [cout]
 * or NULL (zero); thr_out: [cout][L] int32; sign_out: [cout] int8.
 * Requires cout >= 1, K >= 1, 1 <= kbits <= 8, delta_in > 0, q_base > 0,
 * alpha[n] > 0, var[n] + eps > 0, all values finite (else IFQ_EINVAL).
 */
int ifq_fold_layer(int cout, int K, int kbits, const float* alpha, float delta_in, const float* bias,
                   const float* gamma, const float* beta, const float* mean, const float* var, float eps,
                   float q_base, float q_offset, int32_t* thr_out, int8_t* sign_out);

/*
 * ifq_fold_layer_separated -- the same thresholds for the SEPARATED fixed-point
 * conversion of Sec. 2.2 (Fig. 3a), the baseline the paper compares against:
 * with Q = 2^m each float is floored at its own scale, a = floor(alpha*Q),
 * d = floor(delta_in*Q), bq = floor(bias*Q^2), theta = floor(mean*Q),
 * sigma = floor(sqrt(var + eps)/gamma * Q) (the affine BN's divisor),
 * be = floor(beta*Q), t_i = floor(thr_i*Q), and the substructure computes
 *   Y^conv = (a*d*A + bq)/Q^2,  Y^BN = (Y^conv - theta/Q)/(sigma/Q) + be/Q,
 *   code = #{ i : Y^BN > t_i/Q }.
 * That is monotone in A, so it too is code = #{ i : sign*A > T_i }; this
 * returns those exact integer thresholds (64-bit integer arithmetic, no
 * rounding), to run the separated conversion on the same kernels.
 * Same arguments as ifq_fold_layer plus m (1..20); IFQ_EINVAL also when some
 * channel's sigma floors to 0 (no fixed-point divisor).
 */
int ifq_fold_layer_separated(int cout, int K, int kbits, int m, const float* alpha, float delta_in,
                             const float* bias, const float* gamma, const float* beta, const float* mean,
                             const float* var, float eps, float q_base, float q_offset, int32_t* thr_out,
                             int8_t* sign_out);

/*
 * Size in bits/8 (rounded up) of an n x h x w x c map of densely packed
 * kbits-bit codes, 1 <= kbits <= 32 (host, pure): the memory count of the
 * paper's comparison of feature-map sizes.  The library's own buffers use the
 * field format above; ifq_codes_storage_bytes gives their size.
 */
int ifq_codes_bytes(int n, int h, int w, int c, int kbits, size_t* bytes);

/*
 * Bytes of a packed code buffer in the library's format (host, pure):
 * n*h*w*c*f/8 with f = 2 (kbits 0 or 2) or 4 (kbits 3, 4); c % 4 == 0
 * (IFQ_ESHAPE otherwise); other kbits: IFQ_EUNSUPPORTED (negative: IFQ_EINVAL).
 */
int ifq_codes_storage_bytes(int n, int h, int w, int c, int kbits, size_t* bytes);

/*
 * Convolution descriptor.  Input codes NHWC [n][h][w][cin] (cin % 4 == 0),
 * filters [cout][kh][kw][cin], output [n][ho][wo][cout].  out_mode is one of
 * IFQ_OUT_*; codes output needs cout % 4 == 0.  path selects a kernel path
 * (IFQ_PATH_AUTO lets the library choose).  Limits: n >= 0, all other sizes >= 1,
 * K = kh*kw*cin <= 65536, cout <= 65536, n*ho*wo < 2^31.
 * kbits: the code width k of the input codes and of the output codes (0
 * means 2; 2, 3 or 4, else IFQ_EUNSUPPORTED); the thresholds are then
 * [cout][2^k - 1] (Eq. (8)).
 * in_bits: 0 (or kbits) for k-bit input codes; 8 for unsigned 8-bit input
 * values, one byte each (a first layer on image pixels, whose substructure
 * the integrated conversion covers as well: binary filters, integer inputs).
 * An 8-bit input needs cin % 4 == 0 (pad RGB with a zero channel), the
 * tensor-core path and 255*K <= 196608 (IFQ_EUNSUPPORTED otherwise); its
 * layer can only read the stack input in ifq_forward, and its fold takes
 * K_fold = ceil(255*K / (2^k - 1)) so that the clamp covers |A| <= 255*K.
 * pool: 0 or 1 for none; p = 2 or 4 max-pools the convolution output over
 * p x p windows with stride p before the thresholds (Sec. 2.1: the pool acts
 * on Y^conv, before BN and the quantizer), so that the codes are those of the
 * window maximum of A and the output is [n][ho/p][wo/p][cout].  Needs
 * ho % p == 0, wo % p == 0, out_mode IFQ_OUT_CODES and the tensor-core path
 * (IFQ_EUNSUPPORTED otherwise).
 */
typedef struct {
  int n, h, w, cin;
  int cout;
  int kh, kw, stride, pad;
  int out_mode;
  int path;
  int pool;
  int kbits;
  int in_bits;
} ifq_conv_desc;

/* Output spatial size of a conv descriptor (host, pure). */
int ifq_conv_out_shape(const ifq_conv_desc* d, int* ho, int* wo);   /* after the pool, if any */

/*
 * Size of the prepared-filter buffer that ifq_pack_weights fills for `d`
 * (host, pure).  The prepared layout is private to the library.
 */
int ifq_weights_prep_bytes(const ifq_conv_desc* d, size_t* bytes);

/*
 * ifq_pack_weights -- expand the filter sign bits of Eq. (1)'s W_b into the
 * library's prepared form (tensor-core operand rows and a sign-bit copy).
 * w_bits (device): [cout][ceil(K/32)] uint32 sign words as in the header;
 * w_prep (device): ifq_weights_prep_bytes bytes, 16-byte aligned.
 * Run once per layer; the result is reused by every ifq_conv2bit call.
 */
int ifq_pack_weights(const ifq_conv_desc* d, const uint32_t* w_bits, void* w_prep, void* stream);

/*
 * The kernel path ifq_conv2bit takes for `d` (host; reads IFQ_FORCE_PATH as
 * ifq_conv2bit does): IFQ_PATH_TC, IFQ_PATH_BITSERIAL, IFQ_PATH_DIRECT,
 * IFQ_PATH_WIN or IFQ_PATH_WARP.  The warp-MMA path (mma.sync e4m3 tiles of
 * 16 pixels x 8 channels, accumulators and the fused pool in registers)
 * serves 3 x 3 stride-1 layers with padding 1 on 2-bit codes with cin 8 or 16
 * or on 8-bit values with cin 4, with 2-bit codes or accumulators out,
 * cout 8, 16 or 32, and no pool or a 2 x 2 pool on even sizes; it is the
 * default (where it was measured faster) for such layers on codes with cin 8
 * and for such layers on 8-bit values without a pool, and a request for it
 * elsewhere takes the tensor-core path.  The window path serves stride-1 k x k layers with "same"
 * padding (k odd, <= 7) on 2-bit codes with cin 16 or a multiple of 32, cout
 * 32, 64 or a multiple of 128, no pool or a 2 x 2 pool on even sizes, input
 * rows of whole 16-byte units, output rows of at most 256 pixels, and a
 * filter bank that stays resident in one CTA's shared memory; it is the
 * default for such layers with a fused 2 x 2 pool and cin <= 64 (where it was
 * measured faster), and a request for it elsewhere takes the tensor-core
 * path.  The
 * tensor-core path needs (2^k - 1)*K <= 196608 (the accumulator range checked
 * exact on the fp8 tensor cores; 255*K for 8-bit inputs), kh, kw <= 15, and
 * for k = 3, 4 cin % 8 == 0; a request for it outside that range takes the
 * bit-serial path.  The direct CUDA-core path serves layers on 8-bit inputs
 * with cout <= 32 and K <= 257 (the default for them); a request for it
 * elsewhere takes the tensor-core path.  IFQ_EUNSUPPORTED for a fused pool
 * or an 8-bit input that would land on the bit-serial path.
 */
int ifq_conv_plan(const ifq_conv_desc* d, int* path);

/* Device workspace that ifq_conv2bit needs for `d` (host, pure); may be 0. */
int ifq_conv_workspace_bytes(const ifq_conv_desc* d, size_t* bytes);

/*
 * ifq_conv2bit -- one quantized substructure (Eq. (1) integer core followed
 * by the thresholds of Eq. (7), or of Eq. (8) for k bits; the name keeps the
 * paper's k = 2 case).  For every output pixel and channel n:
 *   A = sum over (dy, dx, c) of w[n][dy][dx][c] * x[b][oy*s+dy-pad][ox*s+dx-pad][c]
 *   y_codes = #{ i : sign[n]*A > thr[n][i] }  (k-bit codes, packed)
 *   y_acc   = A                                (int32), per out_mode
 * x (device): packed codes; w_prep (device): from ifq_pack_weights for the
 * same descriptor; thr (device): int32 [cout][2^k - 1], ascending per channel;
 * sign (device): int8 [cout];
 * y_codes (device, out_mode & CODES): packed [n][ho][wo][cout*f/8] bytes;
 * y_acc (device, out_mode & ACC): int32 [n][ho][wo][cout];
 * ws (device): ifq_conv_workspace_bytes bytes (may be NULL if that is 0).
 * The results are exact integers; x must not alias the outputs.
 */
int ifq_conv2bit(const ifq_conv_desc* d, const void* x, const void* w_prep, const int32_t* thr,
                 const int8_t* sign, void* y_codes, int32_t* y_acc, void* ws, size_t ws_bytes, void* stream);

/* Pooling descriptor (geometry in the header comment); c % 4 == 0; kbits is the code width as in
 * ifq_conv_desc (0 means 2). */
typedef struct {
  int n, h, w, c;
  int k, stride, pad;
  int kbits;
} ifq_pool_desc;

int ifq_pool_out_shape(const ifq_pool_desc* d, int* ho, int* wo);

/*
 * ifq_maxpool2bit -- max pooling placed between conv and BN (Sec. 2.1),
 * computed on the codes.  With sign (device, int8 [c]) given, channel c takes
 * the max of its codes where sign = +1 and the min where sign = -1; since the
 * composed conv/BN/quantizer map is monotone in the accumulator (increasing
 * for +1, decreasing for -1), this equals quantizing the max of Y^conv.  With
 * sign NULL it is the plain max of the codes (pooling after the quantizer).
 * x, y (device): packed codes of width d->kbits.  Limit: the output's packed
 * bytes n*ho*wo*c*f/8 < 2^31 (IFQ_ERANGE).
 */
int ifq_maxpool2bit(const ifq_pool_desc* d, const void* x, const int8_t* sign, void* y, void* stream);

/*
 * ifq_fold_output_separated -- the separated fixed-point conversion (Sec. 2.2)
 * of a NON-quantized substructure's output (the linear detection conv of a
 * YOLO head; AlexNet's last substructure): with Q = 2^m,
 *   mul[n] = floor(alpha[n]*Q) * floor(delta_in*Q),  add[n] = floor(bias[n]*Q^2)
 * so that Y^conv = (mul*A + add) / Q^2 is Eq. (1) with every float floored at
 * its own scale.  Host, pure.  alpha: [cout] > 0, finite; bias: [cout] or NULL;
 * delta_in > 0; m in 1..24; mul_out, add_out: [cout] int64 (IFQ_EINVAL otherwise).
 */
int ifq_fold_output_separated(int cout, int m, const float* alpha, float delta_in, const float* bias,
                              int64_t* mul_out, int64_t* add_out);

/*
 * ifq_fixed_output -- the fixed-point value of that output at scale Q = 2^m:
 *   y[r][n] = floor((mul[n]*A[r][n] + add[n]) / 2^m)   (exact 64-bit integer
 * arithmetic), saturated to the int32 range, i.e. y/Q is Y^conv with m
 * fractional bits.  acc (device): int32 [rows][cout]; mul, add (device): int64
 * [cout] from ifq_fold_output_separated; y (device): int32 [rows][cout];
 * m in 1..24, rows >= 0, cout >= 1; pointers 8-byte aligned (mul, add) and
 * 4-byte aligned (acc, y).
 */
int ifq_fixed_output(const int32_t* acc, int rows, int cout, const int64_t* mul, const int64_t* add, int m,
                     int32_t* y, void* stream);

/* Fixed-point output layer of ifq_forward (kind IFQ_LAYER_FIXED). */
typedef struct {
  int m;
} ifq_fixed_desc;

/*
 * One layer of a stack for ifq_forward.  src is the index of the layer whose
 * output codes are this layer's input (-1: the stack input x).  For a conv,
 * `conv`, w_prep, thr and sign describe it and y_codes / y_acc receive its
 * outputs per conv.out_mode; for a pool, `pool` describes it, sign is the
 * pooled layer's channel signs (or NULL for a plain max) and y_codes receives
 * the pooled codes.  For a fixed-point output (IFQ_LAYER_FIXED), src is a
 * conv layer that writes int32 accumulators, `fixed`, fx_mul and fx_add
 * describe the conversion (ifq_fixed_output) and y_acc receives the int32
 * fixed-point values [rows][cout] of the source conv's shape.  All pointers
 * are device pointers owned by the caller.
 */
typedef struct {
  int kind;
  int src;
  ifq_conv_desc conv;
  ifq_pool_desc pool;
  const void* w_prep;
  const int32_t* thr;
  const int8_t* sign;
  void* y_codes;
  int32_t* y_acc;
  ifq_fixed_desc fixed;
  const int64_t* fx_mul;
  const int64_t* fx_add;
} ifq_layer;

/*
 * Workspace that lets ifq_forward run `layers` as one persistent launch (host;
 * reads the environment variable IFQ_STACK): 4 bytes per 128-output-row block
 * of every layer, rounded up to 256; 0 when the persistent launch is not
 * selected (IFQ_STACK is not "1") or the stack does not qualify (it then runs
 * one launch per layer and needs no workspace).
 */
int ifq_forward_workspace_bytes(const ifq_layer* layers, int nlayers, size_t* bytes);

/*
 * ifq_forward -- run a layer stack in order on one stream (Sec. 3.1: a
 * quantized network is a chain of substructures; the codes of one are the
 * input of the next, and the output scale of one is the input step of the
 * next).  Shapes are checked along the chain before any launch.
 * x (device): the stack input codes; ws (device): workspace, or NULL.
 * By default one launch per layer in stream order (consecutive launches
 * overlap their prologues through programmatic dependent launch).  With
 * IFQ_STACK=1 in the environment and a workspace of
 * ifq_forward_workspace_bytes bytes, a stack of conv layers that all take the
 * tensor-core path, whose written buffers overlap no other buffer of the
 * stack, runs instead as one cooperative persistent launch: its completion
 * counters (in ws, zeroed on `stream` by every call) let each output tile
 * start as soon as the rows it reads exist.  Calls in flight at the same time
 * must not share a workspace.  Results are identical either way.
 */
int ifq_forward(const ifq_layer* layers, int nlayers, const void* x, void* ws, size_t ws_bytes, void* stream);

/*
 * ifq_forward_noalloc -- ifq_forward for callers that cannot hand the library
 * device scratch: a plain C host that owns no device allocator, or a serving
 * loop that must not call cudaMalloc (which can synchronize the whole device).
 * The paper has no counterpart; this is a deployment convenience.  It
 * allocates nothing.  A stack that qualifies for the persistent launch (see
 * ifq_forward; IFQ_STACK is not consulted) keeps that launch's completion
 * counters in a file-scope device array of 256 KiB: 65536 counters, one per
 * 128-output-row block of every layer.  A stack that needs more counters is
 * rejected with IFQ_EWORKSPACE before anything is launched.  The counters
 * must be zero when the kernel starts: every call zeroes the part it uses, on
 * `stream`, before the launch.  Other stacks run one launch per layer, which
 * needs no scratch.  The first call on each device looks up the array's device
 * address (cudaGetSymbolAddress with that device current, no allocation) and
 * should come before any stream capture.  All calls on one device share the
 * array, so calls whose executions overlap in time (on other streams or from
 * other host threads) race on it and must be serialised by the caller.
 * The looked-up address is kept for the life of the process: after
 * cudaDeviceReset (or anything else that destroys the device's primary
 * context) it is stale, so a process that resets a device must not call this
 * entry point on that device again.  Results are identical to ifq_forward's.
 */
int ifq_forward_noalloc(const ifq_layer* layers, int nlayers, const void* x, void* stream);

/*
 * ifq_last_forward_mode -- how the calling host thread's last successful
 * ifq_forward or ifq_forward_noalloc call ran its stack: IFQ_FORWARD_LAYERS
 * (one launch per layer) or IFQ_FORWARD_PERSISTENT (the whole stack as one
 * persistent launch).  The paper has no counterpart; this is a diagnostic for
 * callers and tests that need to know which launch served a request (results
 * are identical either way).  Host only, thread-local; IFQ_EINVAL if `mode` is
 * NULL or the thread has made no successful forward call.
 */
enum { IFQ_FORWARD_LAYERS = 1, IFQ_FORWARD_PERSISTENT = 2 };
int ifq_last_forward_mode(int* mode);

/*
 * CUDA-graph form of ifq_forward: ifq_graph_create captures the launches of
 * ifq_forward(layers, nlayers, x, ws, ws_bytes) on `stream` into a graph that
 * ifq_graph_launch replays on any stream with the same buffers.  The graph is
 * owned by the returned handle; ifq_graph_destroy frees it.  In the graph a
 * layer whose output no later layer reads (other than the last layer) hangs
 * off its source layer as a side branch joined at the end, so it overlaps the
 * layers after it (IFQ_GRAPH_BRANCH=0 keeps one chain); results are identical.
 */
typedef struct ifq_graph ifq_graph;
int ifq_graph_create(const ifq_layer* layers, int nlayers, const void* x, void* ws, size_t ws_bytes, void* stream,
                     ifq_graph** out);
int ifq_graph_launch(ifq_graph* g, void* stream);
int ifq_graph_destroy(ifq_graph* g);

/*
 * ifq_graph_create_io -- ifq_graph_create whose graph also moves the stack's
 * input in and its results out, so that one ifq_graph_launch serves a request
 * end to end.  The paper has no counterpart; this is a serving convenience.
 *   x_src, x_bytes: when x_src is not NULL, the graph first copies x_bytes from
 *     x_src to x.  x_bytes must equal the bytes of packed input that the layers
 *     with src = -1 read (n * h * w * c * field bits / 8; IFQ_ESHAPE otherwise).
 *   y_codes_dst, y_acc_dst: NULL, or arrays of nlayers destinations.  When entry
 *     i is not NULL, the graph copies layer i's y_codes (y_acc) buffer, all of
 *     it, to that address right after layer i, on layer i's branch of the graph.
 *     The results of a side branch are then copied while the main chain runs.
 *     A destination for a buffer that layer i does not have is IFQ_EINVAL.
 * The addresses are part of the graph: every launch copies from and to the same
 * buffers.  A copy between buffers the device addresses directly (device
 * memory, or pinned host memory under unified addressing), 16-byte aligned and
 * a multiple of 16 bytes, runs on the SMs as in ifq_copy_bytes; any other is a
 * cudaMemcpyAsync node.  Argument errors are returned before anything is
 * captured.
 */
int ifq_graph_create_io(const ifq_layer* layers, int nlayers, const void* x, void* ws, size_t ws_bytes,
                        const void* x_src, size_t x_bytes, void* const* y_codes_dst, void* const* y_acc_dst,
                        void* stream, ifq_graph** out);

/*
 * Codes <-> packed format helpers (device buffers; n % 4 == 0 codes, one code
 * per byte on the unpacked side).  The _kbits forms take the code width
 * (0, 2, 3, 4; a code keeps its low f bits); the plain forms are kbits = 2.
 */
int ifq_pack_codes(const uint8_t* codes, void* packed, size_t n, void* stream);
int ifq_unpack_codes(const void* packed, uint8_t* codes, size_t n, void* stream);
int ifq_pack_codes_kbits(const uint8_t* codes, void* packed, size_t n, int kbits, void* stream);
int ifq_unpack_codes_kbits(const void* packed, uint8_t* codes, size_t n, int kbits, void* stream);
/* +-1 int8 filters [rows][K] (device) -> sign words [rows][ceil(K/32)] (device). */
int ifq_pack_signs(const int8_t* w, uint32_t* bits, int rows, int K, void* stream);

/*
 * ifq_copy_bytes -- copy n bytes on `stream` (either side may be device memory
 * or pinned host memory that the device addresses directly under unified
 * addressing).  With both pointers 16-byte aligned, n % 16 == 0 and both
 * addressable by the device at the same address (device memory, or host memory
 * from cudaHostAlloc / cudaHostRegister), the SMs do the copy with 16-byte loads
 * and stores (on a GB300 over NVLink-C2C for host memory); otherwise it is
 * cudaMemcpyAsync.  For staging a stack's inputs and results.
 */
int ifq_copy_bytes(void* dst, const void* src, size_t n, void* stream);

/*
 * ifq_wait_selftest -- exercise the failure path of the bounded device waits:
 * one warp waits on an mbarrier phase that nothing completes for limit_us
 * microseconds (1..1000000), then records IFQ_ETIMEOUT in the device status
 * word and returns normally, as every kernel's waits do after 2 s.  Read it
 * with ifq_device_status; the context stays usable.
 */
int ifq_wait_selftest(int limit_us, void* stream);

/*
 * ifq_device_status -- synchronize `stream`, then read and clear the device
 * status word of the current device: IFQ_OK, or the first device-side error
 * recorded (IFQ_ETIMEOUT, IFQ_ERANGE) since the last read.
 */
int ifq_device_status(void* stream, int* status);

#ifdef __cplusplus
}
#endif

#endif /* IFQ_H */
