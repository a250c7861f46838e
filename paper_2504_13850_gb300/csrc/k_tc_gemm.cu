// Tensor-core path (placeholder: no op is routed to tensor cores yet).
#include "fo_server_impl.h"
#include "fo_tc.h"

namespace fo {

struct TcContext {};
struct TcGemm {};

int tc_create(TcContext** out, fo_server*) {
  *out = new TcContext();
  return 0;
}
void tc_destroy(TcContext* c) { delete c; }
void tc_set_input(TcContext*, int) {}
TcGemm* tc_plan_forward(TcContext*, fo_server*, int) { return nullptr; }
TcGemm* tc_plan_dgrad(TcContext*, fo_server*, int, int) { return nullptr; }
TcGemm* tc_plan_wgrad(TcContext*, fo_server*, int) { return nullptr; }
void tc_run(TcGemm*, const void*, cudaStream_t) {}
const char* tc_name(const TcGemm*) { return "tc"; }

}  // namespace fo
