// ResNet-20 plan of the CUDA path (per-replica implicit-GEMM convolutions, batch-stat BatchNorm,
// option-A shortcuts), driven by the runtime in runtime.cu.
#pragma once
#include <cuda_runtime.h>
#include <stdint.h>

#include <functional>
#include <string>

#include "../../include/lsgd.h"

namespace lsgd {

struct ResNetPlan;

bool resnet_supported(const lsgd_config& cfg, std::string* why);
ResNetPlan* resnet_plan_create(const lsgd_config& cfg);
void resnet_destroy(ResNetPlan* p);
int64_t resnet_num_params(const ResNetPlan* p);
int64_t resnet_d_pad(const ResNetPlan* p);
// Calls f(canonical offset, padded offset, length) for every parameter tensor.
void resnet_segments(const ResNetPlan* p, const std::function<void(int64_t, int64_t, int64_t)>& f);
// Weight decay applies to padded offsets (i mod period) < decay_end.
void resnet_decay_region(const ResNetPlan* p, int64_t* period, int64_t* decay_end);
lsgd_status resnet_alloc(ResNetPlan* p, const std::function<void*(size_t)>& alloc);
lsgd_status resnet_init_params(ResNetPlan* p, float* W, uint64_t seed, cudaStream_t s,
                               int64_t* launches);
// One forward + backward over the K replicas' gathered inputs; gradients into G, per-replica mean
// loss into loss_mean[K].
lsgd_status resnet_forward_backward(ResNetPlan* p, const float* W, const uint16_t* Wb, float* G,
                                    int64_t d_pad, const int32_t* labels, float* loss_mean,
                                    cudaStream_t s, int64_t* launches);
// Forward only with replica k's weights for `groups` groups of B_loc rows; per-row losses.
lsgd_status resnet_eval(ResNetPlan* p, const float* W, const uint16_t* Wb, int64_t d_pad, int k,
                        int groups, const int32_t* labels, float* row_loss, cudaStream_t s,
                        int64_t* launches);
void* resnet_input(ResNetPlan* p);

// Per-replica BatchNorm batch statistics of y [G][P][C] fp32 into mean, rstd [G][C], through the
// chunk partials `part` (batchnorm_stats_scratch_floats(P, C, G) floats, fully overwritten).
size_t batchnorm_stats_scratch_floats(int64_t P, int C, int G);
// Weight gradient of a 3x3 convolution (zero padding 1, stride 1 or 2) for G groups on the tensor
// cores: dW[g dW_gs + (co 9 + kh 3 + kw) Cin + ci] = sum over b, oy, ox of dy[g][b][oy][ox][co]
// x[g][b][oy s + kh - 1][ox s + kw - 1][ci] (zero outside the image), NHWC bf16 operands; the
// per-CTA partials go to `part` (conv_wgrad_scratch_floats floats) and are summed in order.
// cin_out < cin (> 0): x has cin channels of which only the first cin_out are real (zero
// padding), and dW is [Cout][3][3][cin_out].  Shapes as conv_wgrad_tc_ok accepts them, else
// cudaErrorInvalidValue.
size_t conv_wgrad_scratch_floats(int G, int B, int hout, int wout, int cin, int cout, int stride);
cudaError_t launch_conv_wgrad_bf16(const uint16_t* x, const uint16_t* dy, float* dW, int64_t dW_gs,
                                   int G, int B, int hout, int wout, int cin, int cout, int stride,
                                   float* part, cudaStream_t s, int cin_out = 0);
// A 3x3 convolution (zero padding 1, stride 1 or 2) of G groups on the persistent implicit-GEMM
// kernel, exactly as the ResNet-20 step runs it.  mode 0: out = y [G][B][Hout][Wout][cout] from
// in = x [G][B][hin][win][cin] (cin < 16: the stem form, padded to 16 channels); mode 1: out = dx
// [G][B][hin][win][cin] from in = dy [G][B][Hout][Wout][cout].  w [G][cout][3][3][cin] bf16,
// contiguous.  scratch: conv3x3_scratch_bytes bytes of device memory (may be NULL when 0).
// LSGD_EUNSUPPORTED when conv3x3_tc_route rejects the shape.
size_t conv3x3_scratch_bytes(int mode, int G, int B, int hin, int win, int cin, int cout, int stride);
bool conv3x3_tc_route(int mode, int B, int hin, int win, int cin, int cout, int stride);
lsgd_status conv3x3_bf16(int mode, const uint16_t* in, const uint16_t* w, float* out, int G, int B,
                         int hin, int win, int cin, int cout, int stride, void* scratch,
                         cudaStream_t s, std::string* err);
// Mode 0 of conv3x3_bf16 with the output's per-replica BatchNorm statistics formed in the
// convolution's epilogue (as the ResNet-20 step forms them): mean, rstd [G][cout], rstd = 1 /
// sqrt(biased variance + 1e-5).  cout <= 64.  scratch: conv3x3_bn_scratch_bytes bytes.
size_t conv3x3_bn_scratch_bytes(int G, int B, int hin, int win, int cin, int cout, int stride);
lsgd_status conv3x3_bn_bf16(const uint16_t* in, const uint16_t* w, float* y, float* mean,
                            float* rstd, int G, int B, int hin, int win, int cin, int cout,
                            int stride, void* scratch, cudaStream_t s, std::string* err);
cudaError_t launch_batchnorm_stats(const float* y, int64_t P, int C, int G, float* mean,
                                   float* rstd, float* part, cudaStream_t s);
const char* resnet_last_error(const ResNetPlan* p);

}  // namespace lsgd
