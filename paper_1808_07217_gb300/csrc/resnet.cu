// ResNet-20 on the CUDA path.
#include "resnet.h"

namespace lsgd {

struct ResNetPlan {
  std::string err;
};

bool resnet_supported(const lsgd_config&, std::string* why) {
  if (why) *why = "ResNet-20 is not available in this build";
  return false;
}
ResNetPlan* resnet_plan_create(const lsgd_config&) { return nullptr; }
void resnet_destroy(ResNetPlan* p) { delete p; }
int64_t resnet_num_params(const ResNetPlan*) { return 0; }
int64_t resnet_d_pad(const ResNetPlan*) { return 0; }
void resnet_segments(const ResNetPlan*, const std::function<void(int64_t, int64_t, int64_t)>&) {}
void resnet_decay_region(const ResNetPlan*, int64_t* period, int64_t* decay_end) {
  *period = 0;
  *decay_end = 0;
}
lsgd_status resnet_alloc(ResNetPlan*, const std::function<void*(size_t)>&) { return LSGD_EUNSUPPORTED; }
lsgd_status resnet_init_params(ResNetPlan*, float*, uint64_t, cudaStream_t, int64_t*) {
  return LSGD_EUNSUPPORTED;
}
lsgd_status resnet_forward_backward(ResNetPlan*, const float*, const uint16_t*, float*, int64_t,
                                    const int32_t*, float*, cudaStream_t, int64_t*) {
  return LSGD_EUNSUPPORTED;
}
lsgd_status resnet_eval(ResNetPlan*, const float*, const uint16_t*, int64_t, int, int, const int32_t*,
                        float*, cudaStream_t, int64_t*) {
  return LSGD_EUNSUPPORTED;
}
void* resnet_input(ResNetPlan*) { return nullptr; }
const char* resnet_last_error(const ResNetPlan* p) { return p ? p->err.c_str() : ""; }

}  // namespace lsgd
