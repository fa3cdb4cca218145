// Internal launchers of the CUDA path.  Every launcher validates its launch shape on the host and
// returns the CUDA error of the launch; all work is asynchronous on `stream`.
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <string>

namespace lsgd {

// Launch `kernel` with programmatic dependent launch allowed (the kernel begins with pdl_begin()):
// it may be scheduled while the previous kernel on the stream finishes, hiding launch latency and
// its own prologue.
template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                              cudaStream_t stream, Args... args) {
  static_assert(sizeof...(KArgs) == sizeof...(Args), "argument count");
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}


// Record the message lsgd_last_error(NULL) returns on this thread.
void set_last_error(const std::string& msg);

// Parameters of the fused local update (arrays indexed like the GEMM output C).
struct SgdParams {
  float* w;
  float* u;      // may be NULL when mom == 0
  uint16_t* wb;  // bf16 shadow (may be NULL)
  float lr, mom, wd;
  int nesterov;
  int sign;      // signSGD local steps: w -= lr sign(step)
};

// ---- element-wise / reduction kernels (kernels.cu) ----
// sampling: LSGD_SAMPLE_SHARDS (i.i.d. within static shards) or LSGD_SAMPLE_RESHUFFLE (epoch
// permutation, disjoint partitions, in-order pass)
cudaError_t launch_sample_indices(int32_t* idx, uint64_t seed, int64_t step, int K, int B, int64_t N,
                                  int sampling, cudaStream_t stream);
// dst[r][0..D) = X[idx[r]][0..D) (idx == NULL: row r), cast to bf16 when dst_bf16; labels too.
cudaError_t launch_gather_rows(void* dst, bool dst_bf16, int ld_dst, const float* X, int D,
                               const int32_t* idx, int rows, const int32_t* labels_in,
                               int32_t* labels_out, const float* targets_in, float* targets_out,
                               cudaStream_t stream);
// Softmax cross-entropy over logits [G][B][ld]; dz = (softmax - onehot) / B into [G][B][ld_dz]
// (skipped when dz == NULL); loss_mean[g] = mean row loss, loss_sum[g] = sum, row_loss[g B + j]
// = row loss (each may be NULL).
cudaError_t launch_softmax_xent(const float* logits, int ld, int C, const int32_t* labels, int G,
                                int B, void* dz, bool dz_bf16, int ld_dz, float* loss_mean,
                                float* loss_sum, float* row_loss, cudaStream_t stream);
// Least squares: z [G][B][ld] (column 0), r = z - t; loss = r^2 / 2; dz = r / B.
cudaError_t launch_lsq_loss(const float* z, int ld, const float* targets, int G, int B, void* dz,
                            bool dz_bf16, int ld_dz, float* loss_mean, float* loss_sum,
                            float* row_loss, cudaStream_t stream);
// gb[g * gb_gs + o] = sum_j dz[g][j][o] for o < out.
// out[g][j][n] = sum over s < S, in order, of part[s * sstride + (g B + j) ld + n], plus
// bias[g bias_gs + n] (bias may be null): the split-K partial products of a narrow layer.
cudaError_t launch_split_bias_sum(const float* part, int S, int64_t sstride, const float* bias,
                                  int64_t bias_gs, int G, int B, int N, int ld, float* out,
                                  cudaStream_t stream);
cudaError_t launch_colsum(const void* dz, bool dz_bf16, int ld, int G, int B, int out, float* gb,
                          int64_t gb_gs, cudaStream_t stream);
// Bias gradient fused with the local update: b (at sgd.w + g * gs) receives the update step
// computed from sum_j dz[g][j][o] instead of the gradient being stored.
cudaError_t launch_colsum_update(const void* dz, bool dz_bf16, int ld, int G, int B, int out,
                                 int64_t gs, const SgdParams& sgd, cudaStream_t stream);
cudaError_t launch_sgd_update(float* w, float* u, const float* g, uint16_t* wb, int64_t n, float lr,
                              float momentum, int nesterov, float weight_decay, int64_t period,
                              int64_t decay_end, cudaStream_t stream, int sign_steps = 0);
// ---- synchronisation variants (Sec. C.3.1 global momentum; Algorithms 4 and 5) ----
// p[k] = ||wref - W[k] (+ E[k])||_1 / d_canon, through per-chunk partials `part` [K][nq]
// (nq = l1_chunks(d)), combined in chunk order.
int l1_chunks(int64_t d);
cudaError_t launch_l1_norms(const float* W, const float* wref, const float* E, int K, int64_t d,
                            int64_t d_canon, float* part, float* p, cudaStream_t stream);
// wref -= (1/K) sum_k sign(Delta_k) p[k], Delta_k = wref - W[k] (+ E[k]); E[k] = Delta_k - s p
// when E != NULL; every replica (and its bf16 shadow) becomes wref.
cudaError_t launch_sign_sync(float* W, uint16_t* Wb, float* wref, float* E, const float* p, int K,
                             int64_t d, cudaStream_t stream);
// ug = mg ug + (wref - mean_k W[k]) / lr; wref -= lr ug; every replica becomes wref.
cudaError_t launch_gm_sync(float* W, uint16_t* Wb, float* wref, float* ug, int K, int64_t d,
                           float lr, float mg, cudaStream_t stream);
cudaError_t launch_kway_average(float* W, uint16_t* Wb, int K, int64_t d, cudaStream_t stream);
// Segments of a replica (float4 offset and length, within d_pad) for the segment average.
constexpr int kMaxAvgSegments = 2 * 8 + 2;
struct AvgSegments {
  int n;
  int64_t off4[kMaxAvgSegments], len4[kMaxAvgSegments];
};
// The K-way average of kway_average restricted to the listed segments of each replica.
cudaError_t launch_average_segments(float* W, uint16_t* Wb, int K, int64_t d_pad,
                                   const AvgSegments& sg, cudaStream_t stream);
// Replica 0's copy of the listed segments (and of their bf16 shadow, if Wb) to every other replica.
cudaError_t launch_broadcast_segments(float* W, uint16_t* Wb, int K, int64_t d_pad,
                                      const AvgSegments& sg, cudaStream_t stream);

// Average within each of `groups` groups of Kp consecutive replicas (replica stride d).
cudaError_t launch_group_average(float* W, uint16_t* Wb, int Kp, int groups, int64_t d,
                                 cudaStream_t stream);
cudaError_t launch_init_normal(float* w, int64_t n, double stddev, uint64_t seed, uint32_t tensor_id,
                               cudaStream_t stream);
cudaError_t launch_fill(float* w, int64_t n, float v, cudaStream_t stream);
cudaError_t launch_broadcast(float* W, int K, int64_t d, cudaStream_t stream);
cudaError_t launch_to_bf16(const float* w, uint16_t* wb, int64_t n, cudaStream_t stream);
cudaError_t launch_check_finite(const float* w, int64_t n, int* flag, cudaStream_t stream);

// ---- grouped GEMM: C[g](m, n) = sum_k A[g](m, k) B[g](k, n), with a fused epilogue ----
enum GemmEpilogue {
  EPI_STORE = 0,      // C = acc
  EPI_BIAS = 1,       // C = acc + bias[n]
  EPI_BIAS_RELU = 2,  // C = max(acc + bias[n], 0)
  EPI_MASK = 3        // C = mask(m, n) > 0 ? acc : 0   (ReLU derivative from the stored activation)
};

struct GemmArgs {
  int M, N, Kd, G;
  const void* A;
  int64_t a_rs, a_cs, a_gs;  // element strides of A(m, k) and per group
  bool a_bf16;
  const void* B;
  int64_t b_rs, b_cs, b_gs;  // element strides of B(k, n)
  bool b_bf16;
  void* C;
  int64_t c_rs, c_gs;  // C(m, n) at C + g c_gs + m c_rs + n
  bool c_bf16;
  int epi;
  const float* bias;
  int64_t bias_gs;
  const void* mask;
  int64_t mask_rs, mask_gs;
  bool mask_bf16;
  // EPI_MASK with M <= 128 (one tile holds the whole mini-batch): also form the column sums of the
  // stored result -- the bias gradient of the layer it feeds -- and apply the local update to that
  // bias through bsgd (bsgd.w at the bias, replica stride bias_gs), or, with bsgd.w == NULL, write
  // it to bias_grad (same indexing)
  bool bias_colsum;
  SgdParams bsgd;
  float* bias_grad;
  // implicit 3x3 convolution (zero padding 1): C[p][n] = sum over taps t and k < cv_ck of
  // in[shift_t(p)][k] B[n][t][k].  A is a rank-5 map over the NHWC input {cv_ck, W, H, B, G} whose
  // box is {cv_ck, Wout * s, rows * s, images, 1} with element strides {1, s, s, 1, 1}; B a rank-3
  // map over the [N][9][cv_ck] weights {9 cv_ck, N, G} with box {cv_ck, 64}; both swizzled by
  // cv_ck * 2 bytes.  M = pixels of the output (whole rows per 128-pixel tile), Kd unused.
  int conv;
  int cv_ck, cv_stride, cv_hout, cv_wout;
  // split-K (SIMT): with ws (ws_floats floats) a long reduction over few output tiles may be cut
  // into up to ws_floats / (G M N) contiguous k ranges, each CTA's raw sums going to
  // ws[g][split][m][n] and a second kernel adding them in split order before the epilogue
  float* ws;
  int64_t ws_floats;
};
// Persistent implicit-GEMM 3x3 convolution (zero padding 1): out[g][p][n] (fp32, replica stride
// out_gs) = sum over taps t and k < ck of in[g][shift_t(p)][k] w[g][n][t][k].  in_map: the rank-5
// map of make_tma_map_conv; w_map: a rank-3 map over the [N][9][ck] weights {9 ck, N, G} with box
// {ck, np} and a ck * 2-byte swizzle.  ck, N in {16, 32, 64}, np = N; P = output pixels per
// replica, a multiple of 128 and of hout * wout.
// A data gradient whose result feeds the BatchNorm backward of the layer below (ResNet-20's
// backward pass, Sec. A.2): the convolution's epilogue adds the option-A shortcut's share of the
// block's output gradient (sc_dout non-null: stride 1 at every pixel, stride 2 at the pixels on
// the stride grid, the first N of sc_C channels, masked by the block output sc_out > 0), applies
// the ReLU mask of that layer (mask > 0), writes g = (dx + shortcut) * (mask > 0) instead of dx,
// and each epilogue warp sums g and g * xhat per channel (xhat = (y - mean) rstd) over its rows of
// every tile: part[g][part_off + 4 q + warp][n] = (sum g, sum g xhat) for CTA q.  mask and y have
// dx's layout; sc_dout / sc_out are [G][pixels of the block output][sc_C] (per replica sc_gs
// elements).
struct ConvBwdFuse {
  const uint16_t* mask;
  const float* y;
  const float* mean;
  const float* rstd;
  const float* sc_dout;
  const uint16_t* sc_out;
  int64_t sc_gs;
  int sc_C, sc_stride;
  float2* part;
  int64_t part_gs;  // partials per replica (all launches that share the buffer)
  int part_off;     // this launch's first partial
};
struct ConvArgs {
  CUtensorMap in_map, w_map;
  int ck, stride, hout, wout, N, np, G, P;
  float* out;
  int64_t out_gs;
  int ring_bytes;  // input ring size (set by the launcher)
  // dst_h > 0: output pixel (image, y, x) of the Hout x Wout grid goes to pixel
  // (image, 2 y + ph_y, 2 x + ph_x) of a dst_h x dst_w grid (one parity phase of a stride-2
  // convolution's data gradient); else to pixel (image, y, x)
  int ph_y, ph_x, dst_h, dst_w;
  // non-null (only with dst_h = 0): partial BatchNorm statistics of the output, stats[g][q][n] =
  // (count, mean, sum of squared deviations, 0) over the pixels of epilogue warp q % 4 of CTA q / 4
  float4* stats;
  int strip;  // stage form: 1 = strip (in_map made with strip = true), 0 = per kernel row
  int st32;   // out 32-byte aligned: 256-bit stores (set by the launcher)
  int nacc, nsplit;  // accumulator buffers and column partials per tile (set by the launcher)
  ConvBwdFuse bwd;   // bwd.y non-null: the data gradient's BatchNorm-backward epilogue
};
// TMEM columns of the convolution kernel for n accumulators (buffers x partials) of np columns: a
// power of two >= 32.
__host__ __device__ inline uint32_t conv_tmem_cols(int n, int np) {
  uint32_t c = 32;
  while (c < (uint32_t)(n * np)) c <<= 1;
  return c;
}
// Stride 1 and tiles of whole image rows with a width that is a multiple of 8: the convolution's
// input boxes carry one halo row above and below (make_tma_map_conv) and one stage feeds all nine
// taps of a tile.
bool conv_strip_ok(int hout, int wout, int stride);
// ctas_per_replica (if non-null) receives the statistics partials per replica (4 per CTA).
cudaError_t launch_conv_tc(const ConvArgs& a, cudaStream_t stream, int* ctas_per_replica = nullptr);
// The CTAs per replica launch_conv_tc will use for these arguments (0 if it would reject them).
int conv_tc_ctas(const ConvArgs& a);
// Weight gradient of a 3x3 convolution (zero padding 1, stride 1 or 2) on the tensor cores, the
// column matrix built in shared memory: part[g][q][co][t Cin + ci] = the sum over CTA q's 64-pixel
// output blocks of dy[g][p][co] x[g][src_t(p)][ci], src_t(p) the input pixel under tap t of output
// pixel p (zero outside the image).  x_map: make_tma_map_halo over the NHWC input; dy_map: rank-3
// bf16 map over [G][P][Cout] with box {64, 64} and a 128-byte swizzle.  Cin 16 / 32 / 64, Cout a
// multiple of 16 up to 64, Wout dividing 64, Hout Wout a multiple of 64.  dy_map's box is
// {nb, 64} with a 2 nb-byte swizzle.
struct ConvWgradArgs {
  CUtensorMap x_map, dy_map;
  int cin, cout, stride, hin, win, hout, wout, G, P;
  int cpr;      // CTAs (partials) per replica, from conv_wgrad_ctas
  float* part;  // [G][cpr][cout][9 cin]
  int ni, na;   // input stages and A buffers (set by the launcher)
  int nb;       // the MMAs' N and the output-gradient tile's channels (16, 32 or 64; dy_map's box)
};
bool conv_wgrad_tc_ok(int cin, int cout, int stride, int hin, int win, int hout, int wout);
int conv_wgrad_ctas(int cin, int stride, int wout, int G, int64_t P);
// The input strip of one 64-pixel output block: rank-5 map {Cin, Win, Hin, B, G} with box
// {Cin, Win, rows, 1, 1}, rows = (64 / Wout - 1) stride + 3, swizzled at the 2 Cin-byte row.
bool make_tma_map_halo(CUtensorMap* map, const void* base, int cin, int win, int hin, int B, int G,
                       int stride, int wout);
cudaError_t launch_conv_wgrad_tc(const ConvWgradArgs& a, cudaStream_t stream);
// The tile geometry of an implicit convolution with an Hout x Wout output: whole output rows,
// 128 pixels per tile.  False when the shape does not tile that way.
bool conv_tile_shape(int hout, int wout, int* rows, int* images);
// strip: the box of the strip form (rows + 2 rows; conv_strip_ok must hold), else the tile's
// rows at the convolution stride.
bool make_tma_map_conv(CUtensorMap* map, const void* base, int ck, int win, int hin, int B, int G,
                       int wout, int hout, int stride, bool strip = false);

cudaError_t launch_gemm_simt(const GemmArgs& a, cudaStream_t stream);

// ---- tcgen05 / TMEM / TMA grouped GEMM (gemm_tc.cu), bf16 operands, fp32 accumulation ----
// A is M x Kd, B is N x Kd (as stored: "K-major" = Kd contiguous, "MN-major" = M/N contiguous),
// both described by rank-3 TMA maps whose outermost dimension is the replica (group).
struct TcOperand {
  CUtensorMap map;  // box: K-major {64 (Kd), box_rows}; MN-major {64 (M or N), 64 (Kd)}
  bool mn_major;
  int box_rows;     // rows of the box the map was encoded with (checked before launch)
};

struct TcGemmArgs {
  int M, N, Kd, G;
  TcOperand A, B;
  // split-K: the reduction is cut into `splits` contiguous ranges of k-blocks, split s writing its
  // partial product at C + g c_gs + s c_split_stride (EPI_STORE only); 0 or 1 = no split
  int splits;
  int64_t c_split_stride;
  // epilogue (same semantics as GemmArgs), C(m, n) at C + g c_gs + m c_rs + n
  void* C;
  int64_t c_rs, c_gs;
  bool c_bf16;
  int epi;
  const float* bias;
  int64_t bias_gs;
  const void* mask;
  int64_t mask_rs, mask_gs;
  bool mask_bf16;
  // EPI_MASK with M <= 128 (one tile holds the whole mini-batch): also form the column sums of the
  // stored result -- the bias gradient of the layer it feeds -- and apply the local update to that
  // bias through bsgd (bsgd.w at the bias, replica stride bias_gs), or, with bsgd.w == NULL, write
  // it to bias_grad (same indexing)
  bool bias_colsum;
  SgdParams bsgd;
  float* bias_grad;
  // implicit 3x3 convolution (zero padding 1): C[p][n] = sum over taps t and k < cv_ck of
  // in[shift_t(p)][k] B[n][t][k].  A is a rank-5 map over the NHWC input {cv_ck, W, H, B, G} whose
  // box is {cv_ck, Wout * s, rows * s, images, 1} with element strides {1, s, s, 1, 1}; B a rank-3
  // map over the [N][9][cv_ck] weights {9 cv_ck, N, G} with box {cv_ck, 64}; both swizzled by
  // cv_ck * 2 bytes.  M = pixels of the output (whole rows per 128-pixel tile), Kd unused.
  int conv;
  int cv_ck, cv_stride, cv_hout, cv_wout;
  // b_shared = 1 (not with conv): every group reads B from group 0 -- the replicas' weights are
  // identical (the step follows an average), so one copy serves all, mostly from L2
  int b_shared;
};

// The weight gradient of one dense layer fused with the local update, for G replicas: W[g] (M x
// N, row stride N) -= update(dZ[g]^T act[g]) with the momentum and bf16 shadow of SgdParams.
// wmap / umap: fp32 maps over sgd.w / sgd.u, dims {N, M, G}, strides {N, replica stride}, box
// {32, 128}, 128-byte swizzle; wbmap: the same over sgd.wb in bf16 with a 64-byte swizzle.
// One layer of a weight-gradient + update launch: dZ (m = output unit) and act (n = input) as for
// the weight-gradient GEMM, and 128 x 32 chunk maps of the layer's w, u (fp32) and bf16 shadow.
struct WgradUpdateLayer {
  int M, N;
  TcOperand A, B;
  CUtensorMap wmap, umap, wbmap;
};
// Up to kWgradMaxLayers layers share one persistent launch (their tiles form one list in layer
// order).  All layers have the same contraction length Kd (= B_loc), replica count G and update
// rule; sgd's pointers matter only for being null or not (u: momentum, wb: bf16 shadow).
constexpr int kWgradMaxLayers = 3;
struct WgradUpdateArgs {
  int Kd, G, nl;
  WgradUpdateLayer L[kWgradMaxLayers];
  SgdParams sgd;
  // avg = 1: the step ends with the K-way average (Eq. 2 right): every replica's tile is updated
  // as above, and the mean of the updated tiles (the average kernel's arithmetic) is written to
  // replica 0's parameters and shadow (the other replicas' copies are left to the caller).
  // w_rep0 = 1: the replicas are identical at the step's start, so each tile's parameters are
  // read from replica 0.
  int avg, w_rep0;
};
cudaError_t launch_wgrad_update(const WgradUpdateArgs& a, cudaStream_t stream);
// The classifier head (last dense layer with at most kHeadMaxClasses outputs, bf16 mode): the
// forward product + softmax cross-entropy, then data / weight / bias gradients with the fused
// update (or the gradient into `grad`).  Replica g's parameters start at g * rep_stride.
constexpr int kHeadMaxClasses = 16;
struct HeadArgs {
  int C, B, in, reps;
  int64_t rep_stride, w_off, b_off;
  const uint16_t* act;  // [reps][B][ld_in] bf16 input of the last layer
  int ld_in;
  const uint16_t* Wb;   // bf16 shadow of the parameters (the products' operand)
  const float* W;       // fp32 parameters (the bias of the forward)
  const int32_t* labels;  // [reps][B]
  uint16_t* dz;         // [reps][B][ld_dz] bf16 logits gradient
  int ld_dz;
  uint16_t* dz_prev;    // [reps][B][ld_dz_prev] data gradient for the layer below (NULL: none)
  int ld_dz_prev;
  float* row_loss;      // [reps][B]
  float* loss_mean;     // [reps]
  int fused;            // 1: apply the update through sgd (arena base pointers); 0: write grad
  SgdParams sgd;
  float* grad;
  // backward only: the bias gradient of the layer below (sum over rows of dz_prev, which the
  // forward kernel wrote) and its update, column block by column block; b_prev_off < 0: none
  int64_t b_prev_off;
};
bool head_supported(int C, int B, int in);
cudaError_t launch_head_forward(const HeadArgs& h, cudaStream_t stream);
cudaError_t launch_head_backward(const HeadArgs& h, cudaStream_t stream);

// Rank-3 TMA map over [dim2][dim1][dim0] (fp32 or bf16) with strides (elements) s1, s2, box
// {box0, box1, 1} and a swizzle of 0, 32, 64 or 128 bytes.
bool make_tma_map(CUtensorMap* map, const void* base, bool bf16, uint64_t dim0, uint64_t dim1,
                  uint64_t dim2, uint64_t s1, uint64_t s2, uint32_t box0, uint32_t box1,
                  int swizzle_bytes);

// Encode a rank-3 bf16 TMA map over [dim2][dim1][dim0] with strides (elements) s1, s2.
bool make_tma_map_bf16(CUtensorMap* map, const void* base, uint64_t dim0, uint64_t dim1,
                       uint64_t dim2, uint64_t s1, uint64_t s2, uint32_t box0, uint32_t box1);
// The same for fp32 data, without swizzling (used for L2 prefetches of parameter tiles).
bool make_tma_map_f32(CUtensorMap* map, const void* base, uint64_t dim0, uint64_t dim1,
                      uint64_t dim2, uint64_t s1, uint64_t s2, uint32_t box0, uint32_t box1);
cudaError_t launch_gemm_tc(const TcGemmArgs& a, cudaStream_t stream);
// N-tile width the tcgen05 kernel uses for a reduction of length Kd (the row count a K-major B
// operand's TMA box must have).
int tc_tile_n(int Kd);
// The largest split count <= want for which every split of a Kd-long reduction is nonempty.
int tc_valid_splits(int Kd, int want);
constexpr int kTcTileM = 128;
bool tc_available();
// 1 if a bounded wait inside a tcgen05 kernel ran out since the last call (then cleared).
int tc_take_timeout_flag();
// One bounded mbarrier wait (the GEMM's mbar_wait) with the given cycle limit (<= the GEMM's):
// *out (device) = 1 if the phase completed (arrive != 0), 0 if the wait ran out.
cudaError_t launch_bounded_wait_selftest(long long limit_cycles, int arrive, int* out,
                                         cudaStream_t stream);

}  // namespace lsgd
